"""GPU parity for the meta-game solvers (Sec. 4.2 meta-solver, App. C.2
aggregation) against the oracle:

* fictitious play is bit-exact: identical play counts (so identical mixtures)
  and identical fp64 bounds, including tie-heavy integer tables, ragged and
  1 x n shapes, tables held off chip, batches, and the stride-4 read of an
  evaluation output;
* the LP's value is within 1e-9 of the oracle's (scaled by the payoff range)
  and its mixtures form an equilibrium (NashConv <= 1e-8); equilibria need not
  be unique, so the mixtures are checked by that property, not element-wise;
* aggregation is within 1e-12 (relative) of the oracle's matrix products.
"""
import numpy as np
import pytest

from gpu_util import context, need_gpu
from oracle import meta_solver as ms

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    c = context()
    yield c
    c.close()


def run_fp(ctx, tables, iters, stride=1, raw=None):
    torch = need_gpu()
    G, m, n = tables.shape
    src = raw if raw is not None else tables
    P = torch.from_numpy(np.ascontiguousarray(src)).cuda()
    x = torch.empty((G, m), dtype=torch.float64, device="cuda")
    y = torch.empty((G, n), dtype=torch.float64, device="cuda")
    b = torch.empty((G, 2), dtype=torch.float64, device="cuda")
    ctx.meta_fictitious_play(P, iters, x, y, b, stride=stride)
    ctx.sync()
    return x.cpu().numpy(), y.cpu().numpy(), b.cpu().numpy()


def check_fp_exact(tables, iters, gx, gy, gb):
    for g in range(tables.shape[0]):
        x, y, lo, hi, _, _ = ms.fictitious_play(tables[g], iters)
        assert np.array_equal(gx[g], x), g
        assert np.array_equal(gy[g], y), g
        assert gb[g, 0] == lo and gb[g, 1] == hi, (g, gb[g], lo, hi)


@pytest.mark.parametrize("m,n", [(1, 1), (1, 7), (6, 1), (2, 2), (37, 53), (64, 64), (100, 100)])
@pytest.mark.parametrize("iters", [1, 2, 500])
def test_fp_bit_exact_normal(ctx, m, n, iters):
    rng = np.random.default_rng(1000 * m + n)
    tables = rng.normal(size=(3, m, n))
    check_fp_exact(tables, iters, *run_fp(ctx, tables, iters))


def test_fp_bit_exact_ties(ctx):
    rng = np.random.default_rng(9)
    tables = rng.integers(-2, 3, size=(8, 20, 30)).astype(np.float64)
    tables[0] = 0.0                                  # every play ties
    check_fp_exact(tables, 777, *run_fp(ctx, tables, 777))


def test_fp_bit_exact_off_chip_and_max(ctx):
    rng = np.random.default_rng(4)
    t1 = rng.normal(size=(2, 300, 257))             # 300 x 257 fp64 > 200 KB: read from L2
    check_fp_exact(t1, 300, *run_fp(ctx, t1, 300))
    t2 = rng.normal(size=(1, 1024, 1024))           # the largest supported table
    check_fp_exact(t2, 50, *run_fp(ctx, t2, 50))
    t3 = rng.normal(size=(3, 256, 200))             # 256 rows, one per thread, read from L2
    check_fp_exact(t3, 120, *run_fp(ctx, t3, 120))
    t4 = rng.normal(size=(2, 257, 100))             # 257 rows: two per thread for some
    check_fp_exact(t4, 120, *run_fp(ctx, t4, 120))


def test_fp_many_games(ctx):
    rng = np.random.default_rng(21)
    tables = rng.normal(size=(700, 8, 8))           # more games than CTAs in the grid
    gx, gy, gb = run_fp(ctx, tables, 200)
    for g in range(0, 700, 37):
        x, y, lo, hi, _, _ = ms.fictitious_play(tables[g], 200)
        assert np.array_equal(gx[g], x) and np.array_equal(gy[g], y)
        assert gb[g, 0] == lo and gb[g, 1] == hi


def test_fp_reads_mean_column_of_eval_output(ctx):
    rng = np.random.default_rng(8)
    m, n = 5, 6
    raw = rng.normal(size=(1, m, n, 4))            # [pairs][mean, SE, sum, sumsq] layout
    tables = np.ascontiguousarray(raw[..., 0])
    check_fp_exact(tables, 321, *run_fp(ctx, tables, 321, stride=4, raw=raw))


def run_lp(ctx, tables):
    torch = need_gpu()
    G, m, n = tables.shape
    P = torch.from_numpy(np.ascontiguousarray(tables)).cuda()
    x = torch.empty((G, m), dtype=torch.float64, device="cuda")
    y = torch.empty((G, n), dtype=torch.float64, device="cuda")
    v = torch.empty((G,), dtype=torch.float64, device="cuda")
    ctx.meta_lp_nash(P, x, y, v)
    ctx.sync()
    return x.cpu().numpy(), y.cpu().numpy(), v.cpu().numpy()


def check_lp(tables, gx, gy, gv):
    for g in range(tables.shape[0]):
        A = tables[g]
        scale = max(1.0, float(A.max() - A.min()))
        _, _, v = ms.lp_nash(A)
        assert abs(gv[g] - v) <= 1e-9 * scale, (g, gv[g], v)
        assert gx[g].min() >= -1e-12 and gy[g].min() >= -1e-12
        assert abs(gx[g].sum() - 1) < 1e-9 and abs(gy[g].sum() - 1) < 1e-9
        assert ms.nash_conv(A, gx[g], gy[g]) <= 1e-8 * scale


@pytest.mark.parametrize("m,n", [(1, 1), (1, 5), (4, 1), (2, 2), (5, 5), (16, 20), (64, 64),
                                 (100, 100)])
def test_lp_value_and_equilibrium(ctx, m, n):
    rng = np.random.default_rng(50 + m * n)
    tables = rng.normal(size=(3, m, n))
    check_lp(tables, *run_lp(ctx, tables))


def test_lp_closed_forms_and_degenerate(ctx):
    rps = np.array([[0, -1, 1], [1, 0, -1], [-1, 1, 0]], float)
    two = np.array([[3.0, -1.0], [-2.0, 1.0]])
    tables = np.zeros((4, 3, 3))
    tables[0] = rps
    tables[1, :2, :2] = two
    tables[1, 2, :] = -10.0                          # dominated row
    tables[1, :, 2] = 10.0                           # dominated column
    tables[2] = 0.25                                 # constant game
    tables[3] = np.array([[1, 1, 2], [1, 1, 2], [0, 0, 3]], float)   # ties everywhere
    gx, gy, gv = run_lp(ctx, tables)
    check_lp(tables, gx, gy, gv)
    assert abs(gv[0]) < 1e-12 and np.abs(gx[0] - 1 / 3).max() < 1e-9
    assert abs(gv[1] - (3 * 1 - (-1) * (-2)) / (3 + 1 + 1 + 2)) < 1e-12
    assert abs(gv[2] - 0.25) < 1e-15


def test_lp_off_chip(ctx):
    rng = np.random.default_rng(77)
    tables = rng.normal(size=(2, 300, 200))          # tableau 301 x 501 fp64 > 200 KB
    check_lp(tables, *run_lp(ctx, tables))


def test_lp_pivot_limit_reports_not_converged(ctx):
    """A game that needs more simplex pivots than the caller's limit raises
    ENOTCONVERGED at the next sync; the flag is cleared once read and the
    context stays usable. Rock-paper-scissors needs at least 3 pivots (its
    optimal basis holds all 3 columns, one enters per pivot); a 1 x 1 game
    needs exactly 1, so a limit of 1 still converges."""
    torch = need_gpu()
    from paper_2106_07551_gb300 import MALIB_ENOTCONVERGED, MalibError
    rps = np.array([[[0, -1, 1], [1, 0, -1], [-1, 1, 0]]], float)
    P = torch.from_numpy(rps).cuda()
    x = torch.empty((1, 3), dtype=torch.float64, device="cuda")
    y = torch.empty((1, 3), dtype=torch.float64, device="cuda")
    v = torch.empty((1,), dtype=torch.float64, device="cuda")
    ctx.meta_lp_nash(P, x, y, v, max_pivots=2)
    with pytest.raises(MalibError) as e:
        ctx.sync()
    assert e.value.code == MALIB_ENOTCONVERGED and "ENOTCONVERGED" in str(e.value)
    ctx.sync()                                       # cleared once reported
    ctx.meta_lp_nash(P, x, y, v, max_pivots=3 * 6)
    ctx.sync()
    check_lp(rps, x.cpu().numpy(), y.cpu().numpy(), v.cpu().numpy())
    one = torch.full((1, 1, 1), 0.5, dtype=torch.float64, device="cuda")
    x1 = torch.empty((1, 1), dtype=torch.float64, device="cuda")
    ctx.meta_lp_nash(one, x1, x1.clone(), v, max_pivots=1)
    ctx.sync()
    assert abs(float(v[0]) - 0.5) < 1e-15
    with pytest.raises(MalibError):
        ctx.meta_lp_nash(P, x, y, v, max_pivots=-1)


def test_aggregate(ctx):
    torch = need_gpu()
    rng = np.random.default_rng(13)
    G, m, n = 4, 33, 65
    tables = rng.normal(size=(G, m, n))
    x = rng.dirichlet(np.ones(m), size=G)
    y = rng.dirichlet(np.ones(n), size=G)
    d = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    ay = torch.empty((G, m), dtype=torch.float64, device="cuda")
    xa = torch.empty((G, n), dtype=torch.float64, device="cuda")
    val = torch.empty((G,), dtype=torch.float64, device="cuda")
    ctx.meta_aggregate(d(tables), d(x), d(y), ay, xa, val)
    ctx.sync()
    for g in range(G):
        r_ay, r_xa, r_v = ms.aggregate(tables[g], x[g], y[g])
        s = np.abs(tables[g]).max()
        assert np.abs(ay[g].cpu().numpy() - r_ay).max() <= 1e-12 * s * n
        assert np.abs(xa[g].cpu().numpy() - r_xa).max() <= 1e-12 * s * m
        assert abs(float(val[g]) - r_v) <= 1e-12 * s * (m + n)


def test_errors(ctx):
    torch = need_gpu()
    from paper_2106_07551_gb300 import MalibError
    P = torch.zeros((1, 4, 4), dtype=torch.float64, device="cuda")
    x = torch.empty((1, 4), dtype=torch.float64, device="cuda")
    b = torch.empty((1, 2), dtype=torch.float64, device="cuda")
    with pytest.raises(MalibError):
        ctx.meta_fictitious_play(P, 0, x, x, b)                     # iters < 1
    with pytest.raises(MalibError):
        ctx.meta_fictitious_play(P.cpu(), 5, x, x, b)               # host table
    big = torch.zeros((1, 1025, 2), dtype=torch.float64, device="cuda")
    with pytest.raises(MalibError):
        ctx.meta_fictitious_play(big, 5, torch.empty((1, 1025), dtype=torch.float64, device="cuda"),
                                 torch.empty((1, 2), dtype=torch.float64, device="cuda"), b)
