"""GPU parity for the particle-spread rollout (N=3, fp32 MLP 18-64-64-5).

The GPU dumps its logits; the oracle replays the same environments with them:
observations, actions, rewards and done flags must then match bit for bit, the
observation padding must be zero, and the GPU logits must match the oracle's
within 1e-5 relative. The full 4,096-env workload is checked on sampled envs."""
import numpy as np
import pytest

import workloads
from gpu_util import context, load_population, logits_close, need_gpu, spec_of

pytestmark = pytest.mark.gpu

from paper_2106_07551_gb300 import MALIB_DUMP_LOGITS, MalibError, alloc_traj

RTOL = 1e-5


def rollout(ctx, w, n_eps, seed, n_envs=None, local_ratio=None):
    spec = spec_of(w, MALIB_DUMP_LOGITS, n_envs, local_ratio)
    traj = alloc_traj(spec, n_eps, logits=True)
    ctx.rollout(spec, w.pair_ids, n_eps, seed, traj)
    ctx.sync()
    return {k: v.cpu().numpy() for k, v in traj.items()}


def check(orc, w, g, n_eps, seed, env_lo, env_hi, local_ratio=None):
    params = [p.params for p in w.policies]
    dims = w.policies[0].dims
    sl = slice(env_lo, env_hi)
    ref = orc.spread_rollout(params, dims, w.n_agents, w.n_landmarks, w.episode_len, w.n_envs,
                             w.pair_ids, n_eps, seed, env_lo=env_lo, env_hi=env_hi,
                             ext_logits=g["logits"][:, :, sl], local_ratio=local_ratio)
    np.testing.assert_array_equal(g["obs"][:, :, sl, :, :w.obs_dim], ref["obs"])
    assert np.all(g["obs"][..., w.obs_dim:] == 0)
    np.testing.assert_array_equal(g["action"][:, :, sl].astype(np.int8), ref["action"])
    np.testing.assert_array_equal(g["reward"][:, :, sl], ref["reward"])
    done = g["done"][:, :, sl]
    assert np.all(done[:, -1] == 1) and np.all(done[:, :-1] == 0)
    n_bad, worst = logits_close(g["logits"][:, :, sl], ref["logits"], RTOL)
    assert n_bad == 0, (n_bad, worst)


@pytest.mark.parametrize("n_envs,epp,n_eps", [(512, 64, 3), (256, 128, 2), (48, 16, 5)])
def test_full_replay_parity(orc, n_envs, epp, n_eps):
    need_gpu()
    w = workloads.spread(n_agents=3, n_envs=n_envs, pop=5, envs_per_pair=epp, with_bias=True,
                         seed=300 + epp)
    ctx = context()
    load_population(ctx, w)
    g = rollout(ctx, w, n_eps, 31337)
    check(orc, w, g, n_eps, 31337, 0, n_envs)
    g2 = rollout(ctx, w, n_eps, 31337)
    for k in g:
        np.testing.assert_array_equal(g2[k], g[k])
    ctx.close()


@pytest.mark.parametrize("rho", [0.0, 0.3, 1.0])
def test_local_ratio_replay_parity(orc, rho):
    """App. B.1's local_ratio weighting of the reward: bit-exact under replay."""
    need_gpu()
    w = workloads.spread(n_agents=3, n_envs=256, pop=4, envs_per_pair=64, with_bias=True, seed=77)
    ctx = context()
    load_population(ctx, w)
    g = rollout(ctx, w, 2, 4242, local_ratio=rho)
    check(orc, w, g, 2, 4242, 0, 256, local_ratio=rho)
    ctx.close()


def test_full_workload_sampled_envs(orc):
    """4,096 envs, 32 combinations of 128 envs, population 16, 2 episodes."""
    need_gpu()
    w = workloads.config(3)
    ctx = context()
    load_population(ctx, w)
    g = rollout(ctx, w, 2, w.seed)
    for lo, hi in ((0, 40), (1000, 1030), (4090, 4096)):
        check(orc, w, g, 2, w.seed, lo, hi)
    assert np.all(g["reward"] <= 0)
    ctx.close()


def test_invalid_rollout_arguments():
    torch = need_gpu()
    w = workloads.spread(n_agents=3, n_envs=64, pop=2, envs_per_pair=16, seed=1)
    ctx = context()
    load_population(ctx, w)
    spec = spec_of(w)
    traj = alloc_traj(spec, 1)
    with pytest.raises(MalibError, match="EINVAL"):       # 64 envs over 3 combinations
        ctx.rollout(spec, w.pair_ids[:3], 1, 0, traj)
    bad = w.pair_ids.copy()
    bad[0, 0] = 7
    with pytest.raises(MalibError, match="EINVAL"):
        ctx.rollout(spec, bad, 1, 0, traj)
    t2 = dict(traj)
    t2["obs"] = traj["obs"].view(-1)[1:]                    # not 16-byte aligned
    with pytest.raises(MalibError, match="EINVAL"):
        ctx.rollout(spec, w.pair_ids, 1, 0, t2)
    with pytest.raises(MalibError, match="EUNSUPPORTED"):  # 256 envs per combination
        big = spec_of(w, n_envs=1024)
        ctx.rollout(big, w.pair_ids, 1, 0, alloc_traj(big, 1))
    ctx.rollout(spec, w.pair_ids, 0, 0, traj)              # zero episodes: no-op
    ctx.close()


def test_forced_episode_closed_form(orc):
    """Policies with zero weights and b3 = (0, 100, 0, 0, 0) push every agent +x
    in every step. From rest, after k moves v_k = 0.4 (1 - 0.75^k) and
    p_k = p_0 + 0.04 (k - 3 (1 - 0.75^k)) along x; the GPU's observations and
    rewards must follow that closed form (rewards recomputed in fp64; the
    agents keep their reset distances, hence their collision counts)."""
    need_gpu()
    V, T = 64, 25
    w = workloads.spread(n_agents=3, n_envs=V, pop=2, envs_per_pair=16, seed=6)
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
        st = orc.spread_reset(3, 3, env, w.seed).astype(np.float64)
        p0 = st[:12].reshape(3, 4)[:, :2]
        lm = st[12:18].reshape(3, 2)
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
            cover = sum(min(np.hypot(*(p[a] - lm[l])) for a in range(3)) for l in range(3))
            np.testing.assert_allclose(g["reward"][0, t, env], -(cover + coll), atol=5e-5)
        checked += 1
    assert checked >= 40
