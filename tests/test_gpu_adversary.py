"""GPU parity for the simple adversary rollout (App. B.1; 3 agents, obs 14, fp32
MLP 14-64-64-5 policies).

The GPU dumps its logits; the oracle replays the same environments with them:
observations (including the zero target slot of the adversary), actions,
rewards and done flags must then match bit for bit, the observation padding
must be zero, and the GPU logits must match the oracle's own within 1e-5
relative. The 4,096-env size is checked on sampled envs."""
import numpy as np
import pytest

import oracle
import workloads
from gpu_util import context, load_population, logits_close, need_gpu, spec_of

pytestmark = pytest.mark.gpu

from paper_2106_07551_gb300 import MALIB_DUMP_LOGITS, MalibError, alloc_traj

RTOL = 1e-5


def rollout(ctx, w, n_eps, seed, flags=MALIB_DUMP_LOGITS):
    spec = spec_of(w, flags)
    traj = alloc_traj(spec, n_eps, logits=True)
    ctx.rollout(spec, w.pair_ids, n_eps, seed, traj)
    ctx.sync()
    return {k: v.cpu().numpy() for k, v in traj.items()}


def check(w, g, n_eps, seed, env_lo, env_hi):
    params = [p.params for p in w.policies]
    dims = w.policies[0].dims
    sl = slice(env_lo, env_hi)
    ref = oracle.adversary_rollout(params, dims, w.episode_len, w.n_envs, w.pair_ids, n_eps, seed,
                                   env_lo=env_lo, env_hi=env_hi, ext_logits=g["logits"][:, :, sl])
    np.testing.assert_array_equal(g["obs"][:, :, sl, :, :14], ref["obs"])
    assert np.all(g["obs"][..., 14:] == 0)
    assert np.all(g["obs"][:, :, sl, 0, 4:6] == 0)           # the adversary is not told the target
    np.testing.assert_array_equal(g["action"][:, :, sl].astype(np.int8), ref["action"])
    np.testing.assert_array_equal(g["reward"][:, :, sl], ref["reward"])
    np.testing.assert_array_equal(g["reward"][:, :, sl, 1], g["reward"][:, :, sl, 2])
    done = g["done"][:, :, sl]
    assert np.all(done[:, -1] == 1) and np.all(done[:, :-1] == 0)
    n_bad, worst = logits_close(g["logits"][:, :, sl], ref["logits"], RTOL)
    assert n_bad == 0, (n_bad, worst)


@pytest.mark.parametrize("n_envs,epp,n_eps", [(512, 64, 3), (256, 128, 2), (48, 16, 5)])
def test_full_replay_parity(n_envs, epp, n_eps):
    need_gpu()
    w = workloads.adversary(n_envs=n_envs, pop=5, envs_per_pair=epp, with_bias=True, seed=400 + epp)
    ctx = context()
    load_population(ctx, w)
    g = rollout(ctx, w, n_eps, 2718)
    check(w, g, n_eps, 2718, 0, n_envs)
    g2 = rollout(ctx, w, n_eps, 2718)
    for k in g:
        np.testing.assert_array_equal(g2[k], g[k])
    ctx.close()


def test_4096_envs_sampled():
    need_gpu()
    w = workloads.adversary(n_envs=4096, pop=16)
    ctx = context()
    load_population(ctx, w)
    g = rollout(ctx, w, 2, w.seed)
    for lo, hi in ((0, 40), (2000, 2030), (4090, 4096)):
        check(w, g, 2, w.seed, lo, hi)
    assert np.all(g["reward"][..., 0] <= 0)
    ctx.close()


def test_invalid_adversary_arguments():
    need_gpu()
    w = workloads.adversary(n_envs=64, pop=2, envs_per_pair=16, seed=1)
    ctx = context()
    load_population(ctx, w)
    with pytest.raises(MalibError, match="EINVAL"):      # local_ratio is a spread option
        spec = spec_of(w, local_ratio=0.5)
        ctx.rollout(spec, w.pair_ids, 1, 0, alloc_traj(spec, 1))
    ctx.close()


def test_forced_episode_closed_form(orc):
    """Policies with zero weights and b3 = (0, 100, 0, 0, 0) push every agent +x
    in every step. From rest all three follow v_k = 0.4 (1 - 0.75^k),
    p_k = p_0 + 0.04 (k - 3 (1 - 0.75^k)) along x; the GPU's rewards must equal
    -d(p_0) for the adversary and -min(d(p_1), d(p_2)) + d(p_0) for both good
    agents, recomputed in fp64 from those positions."""
    need_gpu()
    V, T = 64, 25
    w = workloads.adversary(n_envs=V, pop=2, envs_per_pair=16, seed=3)
    for p in w.policies:
        p.params[:] = 0.0
        p.params[-4] = 100.0                              # b3[1]: action 1, +x
    ctx = context()
    load_population(ctx, w)
    g = rollout(ctx, w, 1, w.seed)
    ctx.close()
    assert np.all(g["action"] == 1)
    for env in range(V):
        st = orc.adversary_reset(env, w.seed).astype(np.float64)
        p0 = st[:12].reshape(3, 4)[:, :2]
        target = st[12 + 2 * int(st[16]): 14 + 2 * int(st[16])]
        for t in range(T):
            np.testing.assert_allclose(g["obs"][0, t, env, :, 0], 0.4 * (1 - 0.75 ** t), atol=1e-6)
            k = t + 1
            d = np.hypot(*(p0 + [0.04 * (k - 3 * (1 - 0.75 ** k)), 0.0] - target).T)
            good = -min(d[1], d[2]) + d[0]
            np.testing.assert_allclose(g["reward"][0, t, env], [-d[0], good, good], atol=5e-5)
