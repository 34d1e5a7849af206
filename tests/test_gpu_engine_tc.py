"""GPU parity of the pipelined tensor-core policy forward (two tiles in flight,
layer 3 on the CUDA cores) through malib_selftest_mlp_tc: logits of bf16 MLP
policies 34-256-256-5 and 17-256-256-3 (Leduc image, feature 15 folded into
b1) against the oracle's fp64 forward with bf16 weights and layer inputs,
within 2e-2 relative (|g - o| <= 2e-2 max(|o|, rms of the row)). Row counts
cover one partial tile, many tiles with a ragged tail (more tiles than SMs, so
every CTA runs the pipeline for several tiles), and repeated passes."""
import numpy as np
import pytest

import workloads
from gpu_util import context, load_population, logits_close, need_gpu

pytestmark = pytest.mark.gpu

RTOL = 2e-2


def _rows(rng, n, in_dim, leduc):
    x = rng.standard_normal((n, in_dim)).astype(np.float32)
    if leduc:
        x[:, 15] = 1.0                       # constant in every Leduc state
    return x


@pytest.mark.parametrize("kind", ["spread8", "leduc"])
@pytest.mark.parametrize("n,reps", [(37, 1), (128 * 173 + 45, 1), (1000, 3)])
def test_engine_logits_match_oracle(orc, kind, n, reps):
    torch = need_gpu()
    if kind == "leduc":
        w = workloads.leduc(pop=2, hidden=256, dtype=workloads.BF16, with_bias=True, seed=31)
    else:
        w = workloads.spread(n_agents=8, n_envs=128, pop=3, hidden=256, dtype=workloads.BF16,
                             envs_per_pair=128, with_bias=True, seed=32)
    dims = w.policies[0].dims
    rng = np.random.default_rng(n + reps)
    x = _rows(rng, n, dims[0], kind == "leduc")
    ctx = context()
    load_population(ctx, w)
    pid = len(w.policies) - 1
    dx = torch.from_numpy(x).cuda()
    out = torch.full((n, dims[3]), float("nan"), dtype=torch.float32, device="cuda")
    ctx.selftest_mlp_tc(pid, dx, out, reps=reps)
    ctx.sync()
    g = out.cpu().numpy()
    ctx.close()
    ref = orc.mlp_forward(w.policies[pid].params, dims, x, bf16=True)
    assert np.all(np.isfinite(g))
    n_bad, worst = logits_close(g, ref, RTOL)
    assert n_bad == 0, (n_bad, worst)
