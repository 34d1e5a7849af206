"""GPU parity for Kuhn poker evaluation (4x4 tabular populations):
integer payoff sums equal the oracle's exactly (same Philox streams), per-hand
records equal the oracle's traces, the exact mode is within 1e-6 of the
oracle's enumeration, and the Monte-Carlo table lies within 4 SE of it."""
import numpy as np
import pytest

import workloads
from gpu_util import context, four_se_rule, load_population, need_gpu

pytestmark = pytest.mark.gpu

from paper_2106_07551_gb300 import (MALIB_DUMP_LOGITS, MALIB_EXACT_EXPECTATION, MalibError,
                                    alloc_eval_dump, MALIB_ENV_KUHN)


@pytest.fixture(scope="module")
def kuhn_ctx():
    w = workloads.kuhn()
    ctx = context()
    load_population(ctx, w)
    yield ctx, w
    ctx.close()


def tables(w):
    return np.stack([p.params for p in w.policies])


def test_full_workload_exact_integer_parity(kuhn_ctx, orc):
    ctx, w = kuhn_ctx
    got = ctx.eval_payoff(w.pair_ids, w.n_episodes, w.seed)
    ref, _ = orc.kuhn_eval(tables(w), w.pair_ids, w.n_episodes, w.seed)
    np.testing.assert_array_equal(got[:, 2:], ref[:, 2:])
    np.testing.assert_allclose(got[:, :2], ref[:, :2], rtol=1e-12, atol=1e-15)
    ex = np.array([orc.kuhn_exact(tables(w)[i], tables(w)[j]) for i, j in w.pair_ids])
    n_out, zmax = four_se_rule(got[:, 0], got[:, 1], ex)
    assert n_out <= 1 and zmax < 5, (n_out, zmax)


def test_exact_expectation_mode(kuhn_ctx, orc):
    ctx, w = kuhn_ctx
    got = ctx.eval_payoff_ex(w.pair_ids, 0, 0, MALIB_EXACT_EXPECTATION)
    ex = np.array([orc.kuhn_exact(tables(w)[i], tables(w)[j]) for i, j in w.pair_ids])
    assert np.abs(got[:, 0] - ex).max() < 1e-6
    assert np.all(got[:, 1:] == 0)


def test_nash_profile_value():
    torch = need_gpu()
    a = 0.2
    p0 = np.array([a, 0, 0, a + 1 / 3, 3 * a, 1], np.float32)
    p1 = np.array([1 / 3, 0, 0, 1 / 3, 1, 1], np.float32)
    w = workloads.Workload("kuhn_nash", workloads.ENV_KUHN, 2, 0, 0, 2, 0, 0)
    w.policies = [workloads.Policy(workloads.POL_TABULAR, workloads.F32, 0, (6, 0, 0, 1), p0),
                  workloads.Policy(workloads.POL_TABULAR, workloads.F32, 1, (6, 0, 0, 1), p1)]
    ctx = context()
    load_population(ctx, w)
    pairs = np.array([[0, 1]], np.int32)
    got = ctx.eval_payoff_ex(pairs, 0, 0, MALIB_EXACT_EXPECTATION)
    assert abs(got[0, 0] + 1 / 18) < 1e-6
    mc = ctx.eval_payoff(pairs, 200_000, 3)
    assert abs(mc[0, 0] + 1 / 18) < 4 * mc[0, 1]
    ctx.close()


@pytest.mark.parametrize("n_eps", [1, 2, 255, 257, 1000])
def test_ragged_episode_counts_and_dump(kuhn_ctx, orc, n_eps):
    torch = need_gpu()
    ctx, w = kuhn_ctx
    n_dump = min(n_eps, 300)
    dump = alloc_eval_dump(MALIB_ENV_KUHN, w.n_pairs, n_dump)
    got = ctx.eval_payoff_ex(w.pair_ids, n_eps, 77, MALIB_DUMP_LOGITS, dump=dump, n_dump=n_dump)
    ref, tr = orc.kuhn_eval(tables(w), w.pair_ids, n_eps, 77, n_trace=n_dump)
    np.testing.assert_array_equal(got[:, 2:], ref[:, 2:])
    if n_eps == 1:
        assert np.all(got[:, 1] == 0)
    act = dump["action"].cpu().numpy().astype(np.int32)
    act[act == 255] = -1
    np.testing.assert_array_equal(act, tr[:, :, 3:6])
    rew = dump["reward"].cpu().numpy()
    nd = tr[:, :, 2]
    last = np.take_along_axis(rew, (nd - 1)[..., None], axis=2)[..., 0]
    np.testing.assert_array_equal(last, tr[:, :, 6].astype(np.float32))
    np.testing.assert_array_equal(rew.sum(-1), tr[:, :, 6].astype(np.float32))
    done = dump["done"].cpu().numpy()
    for t in range(3):
        np.testing.assert_array_equal(done[:, :, t], (t >= nd - 1).astype(np.uint8))


def test_device_buffers_and_determinism(kuhn_ctx):
    torch = need_gpu()
    ctx, w = kuhn_ctx
    d_pairs = torch.from_numpy(w.pair_ids).cuda()
    d_out = torch.zeros((w.n_pairs, 4), dtype=torch.float64, device="cuda")
    ctx.eval_payoff(d_pairs, 5000, 11, d_out)
    ctx.sync()
    host = ctx.eval_payoff(w.pair_ids, 5000, 11)
    np.testing.assert_array_equal(d_out.cpu().numpy(), host)
    again = ctx.eval_payoff(w.pair_ids, 5000, 11)
    np.testing.assert_array_equal(again, host)


def test_invalid_arguments(kuhn_ctx):
    torch = need_gpu()
    ctx, w = kuhn_ctx
    bad = w.pair_ids.copy()
    bad[3, 1] = 99
    with pytest.raises(MalibError, match="EINVAL"):
        ctx.eval_payoff(bad, 10, 0)
    swapped = w.pair_ids[:, ::-1].copy()          # seat-1 policy in seat 0
    with pytest.raises(MalibError, match="EINVAL"):
        ctx.eval_payoff(swapped, 10, 0)
    with pytest.raises(MalibError, match="EINVAL"):
        ctx.eval_payoff(w.pair_ids, 0, 0)
    out = ctx.eval_payoff(w.pair_ids[:0], 10, 0)  # empty table: no-op
    assert out.shape == (0, 4)
    # an invalid id in a DEVICE pair table is reported by the next sync
    d_bad = torch.from_numpy(bad).cuda()
    d_out = torch.zeros((w.n_pairs, 4), dtype=torch.float64, device="cuda")
    ctx.eval_payoff(d_bad, 10, 0, d_out)
    with pytest.raises(MalibError, match="EINVAL"):
        ctx.sync()
    ctx.sync()   # cleared


def test_hand_ids_beyond_32_bits_and_64_bit_sums(kuhn_ctx, orc):
    """3 pairs x 2.2e9 hands: the third pair's hand ids start at 4.4e9 > 2^32 and
    every pair's sum of r^2 passes 2^31. The first 256 records of every pair
    equal the oracle's hands at the same global ids; the integer sums are
    consistent with payoffs in {+-1, +-2}; the means lie within 4 SE of the
    exact values."""
    need_gpu()
    ctx, w = kuhn_ctx
    n, n_dump, seed = 2_200_000_000, 256, 5
    pairs = np.ascontiguousarray(w.pair_ids[:3])
    dump = alloc_eval_dump(MALIB_ENV_KUHN, 3, n_dump)
    got = ctx.eval_payoff_ex(pairs, n, seed, MALIB_DUMP_LOGITS, dump=dump, n_dump=n_dump)
    act = dump["action"].cpu().numpy().astype(np.int32)
    act[act == 255] = -1
    rew = dump["reward"].cpu().numpy()
    T = tables(w)
    for k, (i, j) in enumerate(pairs):
        ref = orc.kuhn_hands(T[i], T[j], k * n, n_dump, seed)
        np.testing.assert_array_equal(act[k], ref[:, 3:6])
        np.testing.assert_array_equal(rew[k].sum(axis=1), ref[:, 6])
    s1, s2 = got[:, 2], got[:, 3]
    assert np.all(s2 >= n) and np.all(s2 <= 4 * n) and np.all(np.abs(s1) <= s2)
    ex = np.array([orc.kuhn_exact(T[i], T[j]) for i, j in pairs])
    n_out, zmax = four_se_rule(got[:, 0], got[:, 1], ex)
    assert n_out == 0 and zmax < 4.5, (n_out, zmax)


def test_evaluation_size_limit(kuhn_ctx):
    need_gpu()
    ctx, w = kuhn_ctx
    with pytest.raises(MalibError, match="EINVAL"):            # 2 x (2^39 + 1) > 2^40 hands
        ctx.eval_payoff(np.ascontiguousarray(w.pair_ids[:2]), (1 << 39) + 1, 0)
    ctx.sync()
