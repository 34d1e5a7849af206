"""CPU oracle for the meta-game solvers on a payoff table (test infrastructure).

The paper's PSRO loop (Sec. 4.2, Leduc experiment) solves the meta-game given
by the empirical payoff table with fictitious play, mentions an exact LP
solver, and aggregates payoffs under the resulting equilibrium (the
``aggregate(equilibrium)`` and ``aggregate(equilibrium, brs)`` calls of the
training-loop listing in App. C.2). This module restates those steps plainly
in numpy, fp64. Only the tests, the smoke check and the benchmark's CPU
baseline use it; the GPU path never imports it.

Payoff convention: ``A[i, j]`` is the row player's (seat 0's) payoff when row
policy i meets column policy j; the game is zero-sum, so the column player
receives ``-A[i, j]``.

Readings where the paper is silent (each listed in the design notes):

* Fictitious play is the simultaneous discrete-time form: both players play
  their first policy at t = 1; afterwards each plays a best response to the
  opponent's empirical play so far. Ties go to the lowest index. The
  cumulative payoff vectors are updated by adding one column (row) of A per
  play, in play order, so the fp64 sums have a fixed order.
* Bounds: after T plays, ``lower = min_j (x^T A)_j`` and
  ``upper = max_i (A y)_i`` for the empirical mixtures x, y; the game value
  lies between them and ``upper - lower`` is their NashConv.
* The LP solver returns the game value and one equilibrium; equilibria need
  not be unique, so only the value and the equilibrium property are fixed.
"""
from __future__ import annotations

import numpy as np


def fictitious_play(A, iters: int):
    """Simultaneous fictitious play on the zero-sum matrix game ``A`` (m x n).

    Returns ``(x, y, lower, upper, row_counts, col_counts)`` after ``iters``
    plays: x, y the empirical mixtures (counts / T), lower / upper the bounds
    on the game value defined above.
    """
    A = np.asarray(A, dtype=np.float64)
    m, n = A.shape
    T = int(iters)
    if T < 1 or m < 1 or n < 1:
        raise ValueError("need iters >= 1 and a non-empty payoff table")
    row_counts = np.zeros(m, np.int64)
    col_counts = np.zeros(n, np.int64)
    u_row = np.zeros(m, np.float64)      # sum over plays of A[:, j_s]
    u_col = np.zeros(n, np.float64)      # sum over plays of A[i_s, :]
    i, j = 0, 0                          # both start with their first policy
    for t in range(T):
        row_counts[i] += 1
        col_counts[j] += 1
        u_row += A[:, j]
        u_col += A[i, :]
        i = int(np.argmax(u_row))        # first index attaining the maximum
        j = int(np.argmin(u_col))        # first index attaining the minimum
    x = row_counts / float(T)
    y = col_counts / float(T)
    lower = float(u_col.min()) / float(T)
    upper = float(u_row.max()) / float(T)
    return x, y, lower, upper, row_counts, col_counts


def aggregate(A, x, y):
    """Payoffs under a pair of mixtures: ``(A y, x^T A, x^T A y)``.

    ``A y`` is the payoff of every row policy against the column mixture (the
    payoff a new best-response row would be credited with), ``x^T A`` the
    same for columns, and ``x^T A y`` the expected payoff of the equilibrium.
    """
    A = np.asarray(A, dtype=np.float64)
    x = np.asarray(x, dtype=np.float64)
    y = np.asarray(y, dtype=np.float64)
    ay = A @ y
    xa = x @ A
    return ay, xa, float(x @ ay)


def lp_nash(A):
    """Game value and one equilibrium of the zero-sum game ``A`` by linear
    programming: the row player maximises v subject to ``(x^T A)_j >= v`` for
    every column, x a distribution; the column player's problem is the dual.
    Solved with scipy's LP routine (HiGHS). Returns ``(x, y, value)``.
    """
    from scipy.optimize import linprog

    A = np.asarray(A, dtype=np.float64)
    m, n = A.shape
    # row player: variables (x_1..x_m, v); minimise -v
    c = np.zeros(m + 1)
    c[-1] = -1.0
    A_ub = np.hstack([-A.T, np.ones((n, 1))])          # v - (x^T A)_j <= 0
    b_ub = np.zeros(n)
    A_eq = np.hstack([np.ones((1, m)), np.zeros((1, 1))])
    b_eq = np.ones(1)
    bounds = [(0, None)] * m + [(None, None)]
    r = linprog(c, A_ub=A_ub, b_ub=b_ub, A_eq=A_eq, b_eq=b_eq, bounds=bounds, method="highs")
    if r.status != 0:
        raise RuntimeError(f"row LP failed: {r.message}")
    x = np.clip(r.x[:m], 0.0, None)
    x /= x.sum()
    v = float(r.x[-1])
    # column player: variables (y_1..y_n, w); minimise w s.t. (A y)_i <= w
    c = np.zeros(n + 1)
    c[-1] = 1.0
    A_ub = np.hstack([A, -np.ones((m, 1))])
    b_ub = np.zeros(m)
    A_eq = np.hstack([np.ones((1, n)), np.zeros((1, 1))])
    bounds = [(0, None)] * n + [(None, None)]
    r = linprog(c, A_ub=A_ub, b_ub=b_ub, A_eq=A_eq, b_eq=b_eq, bounds=bounds, method="highs")
    if r.status != 0:
        raise RuntimeError(f"column LP failed: {r.message}")
    y = np.clip(r.x[:n], 0.0, None)
    y /= y.sum()
    return x, y, v


def nash_conv(A, x, y):
    """``max_i (A y)_i - min_j (x^T A)_j`` >= 0, zero exactly at equilibria."""
    A = np.asarray(A, dtype=np.float64)
    return float((A @ np.asarray(y)).max() - (np.asarray(x) @ A).min())
