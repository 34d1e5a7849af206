"""GPU parity for Leduc hold'em evaluation with bf16 MLP policies
17-256-256-3 on the tensor cores.

Every dumped hand is replayed by the oracle (bf16 emulation: weights and layer
inputs rounded to bf16, fp64 sums) with the GPU's logits: observations,
actions, payoffs and the integer payoff sums must match exactly, and the GPU
logits must match the oracle's within 2e-2 relative (|g - o| <= 2e-2 max(|o|,
rms of the row)). At the full 64x64 x 16,384 workload, the first 16 hands of
every pair are replayed and every one of the 4,096 entries is checked against
the exact tree expectation (at most 3 beyond 4 SE, none beyond 5)."""
import concurrent.futures as cf
import os

import numpy as np
import pytest

import workloads
from gpu_util import context, four_se_rule, load_population, logits_close, need_gpu

pytestmark = pytest.mark.gpu

from paper_2106_07551_gb300 import MALIB_DUMP_LOGITS, MALIB_ENV_LEDUC, alloc_eval_dump

RTOL = 2e-2


def run(ctx, w, n_eps, seed, n_dump):
    dump = alloc_eval_dump(MALIB_ENV_LEDUC, w.n_pairs, n_dump)
    res = ctx.eval_payoff_ex(w.pair_ids, n_eps, seed, MALIB_DUMP_LOGITS, dump=dump, n_dump=n_dump)
    ctx.sync()
    return res, {k: v.cpu().numpy() for k, v in dump.items()}


def replay(orc, w, res, d, n_eps, seed, n_dump, full, pairs=None):
    params = [p.params for p in w.policies]
    dims = w.policies[0].dims
    pair_ids = w.pair_ids if pairs is None else w.pair_ids[pairs]
    sel = slice(None) if pairs is None else pairs
    ref, rec = orc.leduc_eval(params, dims, w.pair_ids, n_eps, seed, bf16=True, n_rec=n_dump,
                              ext_logits=d["logits"], n_sim=n_eps if full else n_dump)
    act = d["action"].astype(np.int32)
    act[act == 255] = -1
    np.testing.assert_array_equal(act, rec["action"])
    steps = rec["action"] >= 0
    np.testing.assert_array_equal(d["obs"][..., :17][steps], rec["obs"][steps])
    n_bad, worst = logits_close(d["logits"][steps], rec["logits"][steps], RTOL)
    assert n_bad == 0, (n_bad, worst)
    np.testing.assert_array_equal(d["reward"].sum(-1), rec["payoff"].astype(np.float32))
    if full:
        np.testing.assert_array_equal(res[:, 2:], ref[:, 2:])
    return worst


@pytest.mark.parametrize("n_eps", [1, 3, 300, 1000])
def test_full_replay_parity(orc, n_eps):
    need_gpu()
    w = workloads.leduc(pop=3, hidden=256, dtype=workloads.BF16, with_bias=True, seed=500 + n_eps)
    ctx = context()
    load_population(ctx, w)
    res, d = run(ctx, w, n_eps, 77, n_eps)
    replay(orc, w, res, d, n_eps, 77, n_eps, full=True)
    res2, d2 = run(ctx, w, n_eps, 77, n_eps)          # deterministic
    np.testing.assert_array_equal(res2, res)
    np.testing.assert_array_equal(d2["logits"], d["logits"])
    # the kernel instance without the recording code plays the same hands
    np.testing.assert_array_equal(ctx.eval_payoff(w.pair_ids, n_eps, 77), res)
    ctx.close()


def test_split_tail_units_replay(orc):
    """More pairs than SMs: the last pairs claimed are played in two halves of
    their hands. 13 x 13 pairs x 600 hands, every hand of every pair replayed
    and the integer sums compared exactly."""
    torch = need_gpu()
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    w = workloads.leduc(pop=13, hidden=256, dtype=workloads.BF16, with_bias=True, seed=613)
    assert w.n_pairs > n_sm                      # the split applies
    ctx = context()
    load_population(ctx, w)
    res, d = run(ctx, w, 600, 29, 600)
    replay(orc, w, res, d, 600, 29, 600, full=True)
    np.testing.assert_array_equal(ctx.eval_payoff(w.pair_ids, 600, 29), res)   # no recording
    ctx.close()


def test_full_workload_every_cell(orc):
    """64x64 pairs x 16,384 hands: 16 hands of every pair replayed; all 4,096
    entries against the exact tree expectation."""
    need_gpu()
    w = workloads.config(5)
    ctx = context()
    load_population(ctx, w)
    res, d = run(ctx, w, w.n_episodes, w.seed, 16)
    replay(orc, w, res, d, w.n_episodes, w.seed, 16, full=False)
    plain = ctx.eval_payoff(w.pair_ids, w.n_episodes, w.seed)
    np.testing.assert_array_equal(plain, res)
    ctx.close()
    params = [p.params for p in w.policies]
    dims = w.policies[0].dims
    with cf.ThreadPoolExecutor(os.cpu_count() or 4) as ex:
        exact = np.array(list(ex.map(
            lambda k: orc.leduc_exact(params[w.pair_ids[k][0]], params[w.pair_ids[k][1]], dims,
                                      bf16=True), range(w.n_pairs))))
    assert np.all(res[:, 2] == np.round(res[:, 0] * w.n_episodes))
    n_out, zmax = four_se_rule(res[:, 0], res[:, 1], exact)
    assert n_out <= 3 and zmax < 5, (n_out, zmax)
