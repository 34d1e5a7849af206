"""GPU parity for the particle-spread rollout with N = 8 agents and bf16 MLP
policies 34-256-256-5 on the tensor cores.

The oracle replays the same environments with the GPU's logits (bf16
emulation for its own logits): observations (with zero padding), actions,
rewards and done flags must match bit for bit, and the GPU logits must match
the oracle's within 2e-2 relative. The full 65,536-env workload is checked in
the benchmark's launch (two episodes per environment) on slices of 16
environments from 8 combinations spread across the combination table (first,
middle and last environments of a combination among them)."""
import numpy as np
import pytest

import workloads
from gpu_util import context, load_population, logits_close, need_gpu, spec_of

pytestmark = pytest.mark.gpu

from paper_2106_07551_gb300 import MALIB_DUMP_LOGITS, alloc_traj

RTOL = 2e-2


def rollout(ctx, w, n_eps, seed, local_ratio=None):
    spec = spec_of(w, MALIB_DUMP_LOGITS, None, local_ratio)
    traj = alloc_traj(spec, n_eps, logits=True)
    ctx.rollout(spec, w.pair_ids, n_eps, seed, traj)
    ctx.sync()
    return {k: v.cpu().numpy() for k, v in traj.items()}


def check(orc, w, g, n_eps, seed, lo, hi, local_ratio=None):
    params = [p.params for p in w.policies]
    dims = w.policies[0].dims
    sl = slice(lo, hi)
    ref = orc.spread_rollout(params, dims, w.n_agents, w.n_landmarks, w.episode_len, w.n_envs,
                             w.pair_ids, n_eps, seed, bf16=True, env_lo=lo, env_hi=hi,
                             ext_logits=g["logits"][:, :, sl], local_ratio=local_ratio)
    np.testing.assert_array_equal(g["obs"][:, :, sl, :, :w.obs_dim], ref["obs"])
    assert np.all(g["obs"][..., w.obs_dim:] == 0)
    np.testing.assert_array_equal(g["action"][:, :, sl].astype(np.int8), ref["action"])
    np.testing.assert_array_equal(g["reward"][:, :, sl], ref["reward"])
    done = g["done"][:, :, sl]
    assert np.all(done[:, -1] == 1) and np.all(done[:, :-1] == 0)
    n_bad, worst = logits_close(g["logits"][:, :, sl], ref["logits"], RTOL)
    assert n_bad == 0, (n_bad, worst)


@pytest.mark.parametrize("n_envs,epp,n_eps", [(512, 128, 2), (192, 64, 1), (40, 40, 3)])
def test_full_replay_parity(orc, n_envs, epp, n_eps):
    need_gpu()
    w = workloads.spread(n_agents=8, n_envs=n_envs, pop=5, hidden=256, dtype=workloads.BF16,
                         envs_per_pair=epp, with_bias=True, seed=700 + epp)
    ctx = context()
    load_population(ctx, w)
    g = rollout(ctx, w, n_eps, 4321)
    check(orc, w, g, n_eps, 4321, 0, n_envs)
    g2 = rollout(ctx, w, n_eps, 4321)
    for k in g:
        np.testing.assert_array_equal(g2[k], g[k])
    ctx.close()


def test_local_ratio_replay_parity(orc):
    """App. B.1's local_ratio weighting of the reward: bit-exact under replay."""
    need_gpu()
    w = workloads.spread(n_agents=8, n_envs=256, pop=4, hidden=256, dtype=workloads.BF16,
                         envs_per_pair=128, with_bias=True, seed=91)
    ctx = context()
    load_population(ctx, w)
    g = rollout(ctx, w, 1, 777, local_ratio=0.3)
    check(orc, w, g, 1, 777, 0, 256, local_ratio=0.3)
    ctx.close()


def test_full_workload_sampled_envs(orc):
    """65,536 envs, 512 combinations of 128 envs, population 32, two episodes."""
    need_gpu()
    w = workloads.config(4)
    n_eps = 2
    ctx = context()
    load_population(ctx, w)
    spec = spec_of(w, MALIB_DUMP_LOGITS)
    traj = alloc_traj(spec, n_eps, logits=True)
    ctx.rollout(spec, w.pair_ids, n_eps, w.seed, traj)
    ctx.sync()
    assert bool((traj["reward"] <= 0).all())
    epp = w.n_envs // w.n_pairs
    combos = [0, 37, 101, 178, 255, 300, 433, w.n_pairs - 1]
    offs = [(0, 16), (56, 72), (112, 128)]
    for j, c in enumerate(combos):
        a, b = offs[j % len(offs)]
        lo, hi = c * epp + a, c * epp + b
        g = {k: v[:, :, lo:hi].cpu().numpy() for k, v in traj.items()}
        params = [p.params for p in w.policies]
        ref = orc.spread_rollout(params, w.policies[0].dims, w.n_agents, w.n_landmarks,
                                 w.episode_len, w.n_envs, w.pair_ids, n_eps, w.seed, bf16=True,
                                 env_lo=lo, env_hi=hi, ext_logits=g["logits"])
        np.testing.assert_array_equal(g["obs"][..., :w.obs_dim], ref["obs"])
        assert np.all(g["obs"][..., w.obs_dim:] == 0)
        np.testing.assert_array_equal(g["action"].astype(np.int8), ref["action"])
        np.testing.assert_array_equal(g["reward"], ref["reward"])
        assert np.all(g["done"][:, -1] == 1) and np.all(g["done"][:, :-1] == 0)
        n_bad, worst = logits_close(g["logits"], ref["logits"], RTOL)
        assert n_bad == 0, (c, n_bad, worst)
    ctx.close()


def test_forced_episode_closed_form(orc):
    """bf16 policies with zero weights and b3 = (0, 100, 0, 0, 0) push all 8
    agents +x in every step (the tensor-core forward then yields exactly b3).
    From rest, after k moves v_k = 0.4 (1 - 0.75^k) and
    p_k = p_0 + 0.04 (k - 3 (1 - 0.75^k)) along x; the GPU's observations and
    rewards must follow that closed form (rewards recomputed in fp64; the
    agents keep their reset distances, hence their collision counts)."""
    need_gpu()
    V, T, N = 128, 25, 8
    w = workloads.spread(n_agents=N, n_envs=V, pop=3, hidden=256, dtype=workloads.BF16,
                         envs_per_pair=128, seed=9)
    for p in w.policies:
        p.params[:] = 0.0
        p.params[-4] = 100.0                              # b3[1]: action 1, +x
    ctx = context()
    load_population(ctx, w)
    g = rollout(ctx, w, 1, w.seed)
    ctx.close()
    assert np.all(g["action"] == 1)
    checked = 0
    for env in range(V):
        st = orc.spread_reset(N, N, env, w.seed).astype(np.float64)
        p0 = st[:4 * N].reshape(N, 4)[:, :2]
        lm = st[4 * N:6 * N].reshape(N, 2)
        d = np.hypot(*(p0[:, None, :] - p0[None, :, :]).transpose(2, 0, 1))
        if np.any(np.abs(d - 0.3) < 1e-3):
            continue                                      # too close to the collision radius
        coll = (d < 0.3).sum(axis=1) - 1
        for t in range(T):
            obs = g["obs"][0, t, env]
            np.testing.assert_allclose(obs[:, 0], 0.4 * (1 - 0.75 ** t), atol=1e-6)
            np.testing.assert_allclose(obs[:, 2:4], p0 + [0.04 * (t - 3 * (1 - 0.75 ** t)), 0.0],
                                       atol=5e-6)
            k = t + 1
            p = p0 + [0.04 * (k - 3 * (1 - 0.75 ** k)), 0.0]
            cover = sum(min(np.hypot(*(p[a] - lm[l])) for a in range(N)) for l in range(N))
            np.testing.assert_allclose(g["reward"][0, t, env], -(cover + coll), atol=1e-4)
        checked += 1
    assert checked >= 64
