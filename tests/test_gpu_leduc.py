"""GPU parity for Leduc hold'em evaluation with fp32 MLP policies.

Every dumped hand is replayed by the oracle with the GPU's logits: observations,
actions, per-hand payoffs and the integer payoff sums must then match exactly,
and the GPU logits must match the oracle's own within 1e-5 relative
(|g - o| <= 1e-5 max(|o|, rms of the row)). At the full 8x8 x 65,536 workload
(the launch configuration the benchmark times) sampled hands are replayed and
the table is checked against the exact tree expectation (4-SE rule)."""
import concurrent.futures as cf

import numpy as np
import pytest

import workloads
from gpu_util import context, four_se_rule, load_population, logits_close, need_gpu

pytestmark = pytest.mark.gpu

from paper_2106_07551_gb300 import MALIB_DUMP_LOGITS, MALIB_ENV_LEDUC, alloc_eval_dump

RTOL = 1e-5


def run_dumped(ctx, w, n_eps, seed, n_dump):
    dump = alloc_eval_dump(MALIB_ENV_LEDUC, w.n_pairs, n_dump)
    res = ctx.eval_payoff_ex(w.pair_ids, n_eps, seed, MALIB_DUMP_LOGITS, dump=dump, n_dump=n_dump)
    ctx.sync()
    return res, {k: v.cpu().numpy() for k, v in dump.items()}


def check_replay(orc, w, res, d, n_eps, seed, n_dump, full):
    params = [p.params for p in w.policies]
    dims = w.policies[0].dims
    ref, rec = orc.leduc_eval(params, dims, w.pair_ids, n_eps, seed, n_rec=n_dump,
                              ext_logits=d["logits"], n_sim=n_eps if full else n_dump)
    act = d["action"].astype(np.int32)
    act[act == 255] = -1
    np.testing.assert_array_equal(act, rec["action"])
    steps = rec["action"] >= 0
    np.testing.assert_array_equal(d["obs"][..., :17][steps], rec["obs"][steps])
    assert np.all(d["obs"][..., 17:] == 0)
    assert np.all(d["obs"][~steps] == 0) and np.all(d["logits"][~steps] == 0)
    n_bad, worst = logits_close(d["logits"][steps], rec["logits"][steps], RTOL)
    assert n_bad == 0, (n_bad, worst)
    np.testing.assert_array_equal(d["reward"].sum(-1), rec["payoff"].astype(np.float32))
    nd = rec["ndec"]
    done = d["done"]
    for t in range(8):
        np.testing.assert_array_equal(done[:, :, t], (t >= nd - 1).astype(np.uint8))
    if full:
        np.testing.assert_array_equal(res[:, 2:], ref[:, 2:])
        np.testing.assert_allclose(res[:, :2], ref[:, :2], rtol=1e-12, atol=1e-15)
    return worst


@pytest.mark.parametrize("hidden,n_eps", [(128, 512), (128, 1000), (64, 777)])
def test_full_replay_parity(orc, hidden, n_eps):
    """Every hand of a 4x4 population (random biases) is dumped and replayed."""
    need_gpu()
    w = workloads.leduc(pop=4, hidden=hidden, with_bias=True, seed=100 + hidden)
    ctx = context()
    load_population(ctx, w)
    res, d = run_dumped(ctx, w, n_eps, 4242, n_eps)
    check_replay(orc, w, res, d, n_eps, 4242, n_eps, full=True)
    # determinism: a second call gives the same bits
    res2, d2 = run_dumped(ctx, w, n_eps, 4242, n_eps)
    np.testing.assert_array_equal(res2, res)
    np.testing.assert_array_equal(d2["logits"], d["logits"])
    ctx.close()


@pytest.mark.parametrize("n_eps", [1, 3, 249])
def test_small_and_ragged(orc, n_eps):
    need_gpu()
    w = workloads.leduc(pop=2, with_bias=True, seed=5)
    ctx = context()
    load_population(ctx, w)
    res, d = run_dumped(ctx, w, n_eps, 9, n_eps)
    check_replay(orc, w, res, d, n_eps, 9, n_eps, full=True)
    if n_eps == 1:
        assert np.all(res[:, 1] == 0)
    ctx.close()


@pytest.mark.parametrize("n_eps", [3, 1000])
def test_claimed_hands_across_pairs(orc, n_eps):
    """64 pairs: with 3 hands per pair one CTA walks every pair; with 1,000 more
    CTAs than pairs share each pair's hands. Every hand is replayed."""
    need_gpu()
    w = workloads.leduc(pop=8, hidden=128, with_bias=True, seed=77)
    ctx = context()
    load_population(ctx, w)
    res, d = run_dumped(ctx, w, n_eps, 31, n_eps)
    check_replay(orc, w, res, d, n_eps, 31, n_eps, full=True)
    res2, _ = run_dumped(ctx, w, n_eps, 31, n_eps)
    np.testing.assert_array_equal(res2, res)
    ctx.close()


def test_full_workload_sampled_replay_and_exact_expectation(orc):
    """8x8 pairs x 65,536 hands in the benchmark's launch configuration."""
    need_gpu()
    w = workloads.config(2)
    ctx = context()
    load_population(ctx, w)
    n_dump = 24
    res, d = run_dumped(ctx, w, w.n_episodes, w.seed, n_dump)
    check_replay(orc, w, res, d, w.n_episodes, w.seed, n_dump, full=False)
    # same table without the dump (the benchmark's call)
    plain = ctx.eval_payoff(w.pair_ids, w.n_episodes, w.seed)
    np.testing.assert_array_equal(plain, res)
    params = [p.params for p in w.policies]
    dims = w.policies[0].dims
    with cf.ThreadPoolExecutor(8) as ex:
        exact = np.array(list(ex.map(lambda ij: orc.leduc_exact(params[ij[0]], params[ij[1]], dims),
                                     [tuple(x) for x in w.pair_ids])))
    n_out, zmax = four_se_rule(res[:, 0], res[:, 1], exact)
    assert n_out <= 3 and zmax < 5, (n_out, zmax)
    assert np.all(res[:, 2] == np.round(res[:, 2]))
    ctx.close()
