"""Pins for the oracle's meta-game solvers (Sec. 4.2: fictitious play as the
PSRO meta-solver, an exact LP solver; App. C.2: payoff aggregation under the
equilibrium).

Fixed by mathematics, independently of the oracle's code:
* the closed-form value and equilibrium of 2x2 games without a saddle point;
* Robinson's bracketing: for any mixtures, min_j (x^T A)_j <= v <= max_i (A y)_i;
* dominance and saddle points, where fictitious play's plays are forced;
* a hand-worked trace of the first plays on rock-paper-scissors;
* zero-sum symmetry: the game -A^T has value -v;
* the LP's value against the 2x2 formula and against fictitious play's bounds.
"""
import itertools

import numpy as np
import pytest

from oracle import meta_solver as ms


def value_2x2(a, b, c, d):
    # no saddle point: v = (ad - bc) / (a + d - b - c), x_0 = (d - c) / (a + d - b - c)
    den = a + d - b - c
    return (a * d - b * c) / den, (d - c) / den, (d - b) / den


GAMES_2X2 = [(3.0, -1.0, -2.0, 1.0), (1.0, -1.0, -1.0, 1.0), (5.0, 1.0, 2.0, 4.0)]


@pytest.mark.parametrize("g", GAMES_2X2)
def test_fp_brackets_2x2_value(g):
    a, b, c, d = g
    v, x0, y0 = value_2x2(a, b, c, d)
    A = np.array([[a, b], [c, d]])
    for T in (1, 2, 3, 7, 100, 5000):
        _, _, lo, hi, _, _ = ms.fictitious_play(A, T)
        assert lo <= v + 1e-12 and v <= hi + 1e-12
    x, y, lo, hi, _, _ = ms.fictitious_play(A, 20000)
    assert hi - lo < 0.02
    assert abs(x[0] - x0) < 0.02 and abs(y[0] - y0) < 0.02


def test_fp_rps_hand_trace():
    A = np.array([[0, -1, 1], [1, 0, -1], [-1, 1, 0]], float)
    # plays (0,0), (1,1), (1,1), (1,1), (2,2): worked by hand from the rule
    x, y, lo, hi, rc, cc = ms.fictitious_play(A, 5)
    assert rc.tolist() == [1, 3, 1] and cc.tolist() == [1, 3, 1]
    assert lo == -2 / 5 and hi == 2 / 5
    x, y, lo, hi, rc, cc = ms.fictitious_play(A, 3)
    assert rc.tolist() == [1, 2, 0] and cc.tolist() == [1, 2, 0]


def test_fp_rps_converges_to_uniform():
    A = np.array([[0, -1, 1], [1, 0, -1], [-1, 1, 0]], float)
    x, y, lo, hi, _, _ = ms.fictitious_play(A, 30000)
    assert lo <= 0.0 <= hi and hi - lo < 0.05
    assert np.abs(x - 1 / 3).max() < 0.03 and np.abs(y - 1 / 3).max() < 0.03


def test_fp_dominance_forced():
    # row 0 beats every other row in every column; column 0 gives the row
    # player the least in every row: (0, 0) is played forever.
    A = np.array([[2.0, 3.0, 4.0], [1.0, 2.5, 3.0], [0.5, 2.0, 1.0]])
    x, y, lo, hi, rc, cc = ms.fictitious_play(A, 50)
    assert rc.tolist() == [50, 0, 0] and cc.tolist() == [50, 0, 0]
    assert lo == hi == 2.0


def test_fp_saddle_point_reached():
    # saddle at (1, 2): A[1,2] = 2 is the minimum of row 1 and the maximum of column 2
    A = np.array([[0.0, 5.0, 1.0], [3.0, 4.0, 2.0], [-1.0, 6.0, 0.5]])
    x, y, lo, hi, rc, cc = ms.fictitious_play(A, 1000)
    assert lo <= 2.0 <= hi
    assert rc[1] >= 990 and cc[2] >= 990
    assert hi - lo < 0.05


def test_fp_invariants_random():
    rng = np.random.default_rng(7)
    A = rng.normal(size=(9, 13))
    T = 777
    x, y, lo, hi, rc, cc = ms.fictitious_play(A, T)
    assert rc.sum() == T and cc.sum() == T
    assert np.allclose(x.sum(), 1.0) and np.allclose(y.sum(), 1.0)
    ay, xa, val = ms.aggregate(A, x, y)
    # bounds recomputed from the mixtures by matrix products (not by the
    # incremental sums the solver uses)
    assert abs(hi - ay.max()) < 1e-12 * T and abs(lo - xa.min()) < 1e-12 * T
    assert lo - 1e-12 <= val <= hi + 1e-12


def test_fp_negated_transpose_swaps_roles():
    rng = np.random.default_rng(3)
    A = rng.integers(-5, 6, size=(4, 6)).astype(float)
    _, _, lo, hi, _, _ = ms.fictitious_play(A, 4000)
    _, _, lo2, hi2, _, _ = ms.fictitious_play(-A.T, 4000)
    _, _, v = ms.lp_nash(A)
    assert lo - 1e-12 <= v <= hi + 1e-12
    assert lo2 - 1e-12 <= -v <= hi2 + 1e-12


@pytest.mark.parametrize("g", GAMES_2X2)
def test_lp_2x2_closed_form(g):
    a, b, c, d = g
    v, x0, y0 = value_2x2(a, b, c, d)
    x, y, val = ms.lp_nash(np.array([[a, b], [c, d]]))
    assert abs(val - v) < 1e-9 and abs(x[0] - x0) < 1e-9 and abs(y[0] - y0) < 1e-9


def test_lp_rps_uniform():
    A = np.array([[0, -1, 1], [1, 0, -1], [-1, 1, 0]], float)
    x, y, v = ms.lp_nash(A)
    assert abs(v) < 1e-12 and np.abs(x - 1 / 3).max() < 1e-9 and np.abs(y - 1 / 3).max() < 1e-9


def test_lp_random_equilibrium_and_fp_bracket():
    rng = np.random.default_rng(11)
    for m, n in [(5, 5), (8, 3), (16, 20)]:
        A = rng.normal(size=(m, n))
        x, y, v = ms.lp_nash(A)
        assert ms.nash_conv(A, x, y) < 1e-8
        _, _, lo, hi, _, _ = ms.fictitious_play(A, 3000)
        assert lo - 1e-9 <= v <= hi + 1e-9


def test_aggregate_brute_force():
    rng = np.random.default_rng(5)
    A = rng.normal(size=(4, 3))
    x = rng.dirichlet(np.ones(4))
    y = rng.dirichlet(np.ones(3))
    ay, xa, val = ms.aggregate(A, x, y)
    brute = sum(x[i] * y[j] * A[i, j] for i, j in itertools.product(range(4), range(3)))
    assert abs(val - brute) < 1e-12
    for i in range(4):
        assert abs(ay[i] - sum(A[i, j] * y[j] for j in range(3))) < 1e-12
    for j in range(3):
        assert abs(xa[j] - sum(A[i, j] * x[i] for i in range(4))) < 1e-12
