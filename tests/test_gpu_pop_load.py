"""Population loading converts on the device: the same population loaded from
pageable host memory, pinned host memory or device tensors, at once or over
several calls (the arena then grows by a device copy), and after a reset,
gives bit-identical payoff sums and logits, for every image kind a kernel
reads: the fp32 layout, the bf16 tensor-core image and the Kuhn table (bf16
weights in the fp32 layout load, but no evaluation, rollout or exploitability
kernel takes them)."""
import numpy as np
import pytest

import workloads
from gpu_util import context, need_gpu, spec_of

pytestmark = pytest.mark.gpu

from paper_2106_07551_gb300 import (MALIB_DUMP_LOGITS, MALIB_ENV_KUHN, MALIB_ENV_LEDUC,
                                    alloc_eval_dump, policy_desc)


def load(ctx, w, arrays, chunks):
    spec = spec_of(w)
    ids = []
    bounds = np.linspace(0, len(w.policies), chunks + 1).astype(int)
    for lo, hi in zip(bounds[:-1], bounds[1:]):
        descs = [policy_desc(p.kind, p.dtype, p.seat, p.dims, a)
                 for p, a in zip(w.policies[lo:hi], arrays[lo:hi])]
        ids += list(ctx.pop_load(spec, descs))
    assert ids == list(range(len(w.policies)))


def evaluate(ctx, w, kuhn):
    if kuhn:
        return ctx.eval_payoff(w.pair_ids, w.n_episodes, w.seed), None
    dump = alloc_eval_dump(MALIB_ENV_LEDUC, w.n_pairs, 40)
    res = ctx.eval_payoff_ex(w.pair_ids, w.n_episodes, w.seed, MALIB_DUMP_LOGITS, dump=dump, n_dump=40)
    ctx.sync()
    return res, dump["logits"].cpu().numpy()


@pytest.mark.parametrize("case", ["f32_h128", "f32_h64", "bf16_h256", "kuhn"])
def test_load_sources_and_growth_agree(case):
    torch = need_gpu()
    if case == "kuhn":
        w = workloads.kuhn(n_episodes=3000)
    else:
        hidden = int(case.split("_h")[1])
        dtype = workloads.BF16 if case.startswith("bf16") else workloads.F32
        w = workloads.leduc(pop=3, hidden=hidden, dtype=dtype, with_bias=True, n_episodes=300,
                            seed=900 + hidden)
    kuhn = case == "kuhn"
    host = [np.ascontiguousarray(p.params) for p in w.policies]
    pinned = [torch.from_numpy(a).pin_memory() for a in host]
    device = [torch.from_numpy(a).cuda() for a in host]
    results = []
    for arrays, chunks in ((host, 1), (pinned, 3), (device, len(w.policies))):
        ctx = context()
        load(ctx, w, arrays, chunks)
        results.append(evaluate(ctx, w, kuhn))
        ctx.pop_reset()
        load(ctx, w, host, 2)
        results.append(evaluate(ctx, w, kuhn))
        ctx.close()
    res0, lg0 = results[0]
    for res, lg in results[1:]:
        np.testing.assert_array_equal(res, res0)
        if lg0 is not None:
            np.testing.assert_array_equal(lg, lg0)
    assert np.all(res0[:, 1] > 0)
