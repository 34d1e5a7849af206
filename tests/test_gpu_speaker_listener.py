"""GPU parity for the simple speaker listener rollout (App. B.1; 2 agents, obs
11, fp32 MLP 11-64-64-5 policies, the speaker's actions 3 and 4 masked).

The GPU dumps its logits; the oracle replays the same environments with them:
observations (including the speaker's one-hot target and the listener's
one-step-old message), actions, rewards and done flags must then match bit for
bit, the observation padding must be zero, the speaker must never take actions
3 or 4, and the GPU logits must match the oracle's own within 1e-5 relative.
The 4,096-env size is checked on sampled envs."""
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
    ref = oracle.sl_rollout(params, dims, w.episode_len, w.n_envs, w.pair_ids, n_eps, seed,
                            env_lo=env_lo, env_hi=env_hi, ext_logits=g["logits"][:, :, sl])
    np.testing.assert_array_equal(g["obs"][:, :, sl, :, :11], ref["obs"])
    assert np.all(g["obs"][..., 11:] == 0)
    np.testing.assert_array_equal(g["action"][:, :, sl].astype(np.int8), ref["action"])
    assert g["action"][:, :, sl, 0].max() <= 2                   # the speaker only speaks
    np.testing.assert_array_equal(g["reward"][:, :, sl], ref["reward"])
    np.testing.assert_array_equal(g["reward"][:, :, sl, 0], g["reward"][:, :, sl, 1])
    done = g["done"][:, :, sl]
    assert np.all(done[:, -1] == 1) and np.all(done[:, :-1] == 0)
    n_bad, worst = logits_close(g["logits"][:, :, sl], ref["logits"], RTOL)
    assert n_bad == 0, (n_bad, worst)


@pytest.mark.parametrize("n_envs,epp,n_eps", [(512, 64, 3), (256, 128, 2), (40, 40, 5)])
def test_full_replay_parity(n_envs, epp, n_eps):
    need_gpu()
    w = workloads.speaker_listener(n_envs=n_envs, pop=5, envs_per_pair=epp, with_bias=True,
                                   seed=600 + epp)
    ctx = context()
    load_population(ctx, w)
    g = rollout(ctx, w, n_eps, 1618)
    check(w, g, n_eps, 1618, 0, n_envs)
    g2 = rollout(ctx, w, n_eps, 1618)
    for k in g:
        np.testing.assert_array_equal(g2[k], g[k])
    ctx.close()


def test_4096_envs_sampled():
    need_gpu()
    w = workloads.speaker_listener(n_envs=4096, pop=16)
    ctx = context()
    load_population(ctx, w)
    g = rollout(ctx, w, 2, w.seed)
    for lo, hi in ((0, 40), (2000, 2030), (4090, 4096)):
        check(w, g, 2, w.seed, lo, hi)
    assert np.all(g["reward"] <= 0)
    ctx.close()


def test_invalid_speaker_listener_arguments():
    need_gpu()
    w = workloads.speaker_listener(n_envs=64, pop=2, envs_per_pair=16, seed=1)
    ctx = context()
    load_population(ctx, w)
    with pytest.raises(MalibError, match="EINVAL"):      # local_ratio is a spread option
        spec = spec_of(w, local_ratio=0.5)
        ctx.rollout(spec, w.pair_ids, 1, 0, alloc_traj(spec, 1))
    from paper_2106_07551_gb300 import make_spec
    bad = [dict(n_agents=3), dict(n_landmarks=2), dict(obs_dim=12), dict(n_envs=62)]
    for over in bad:                                     # App. B.1's 2 agents, 3 landmarks
        kw = dict(n_agents=2, obs_dim=11, n_landmarks=3, n_envs=64) | over
        spec = make_spec(w.env_kind, kw["n_agents"], kw["obs_dim"], w.n_actions, kw["n_landmarks"],
                         w.episode_len, kw["n_envs"], 0, None)
        with pytest.raises(MalibError, match="EINVAL"):
            ctx.rollout(spec, w.pair_ids, 1, 0, alloc_traj(spec, 1))
    ctx.sync()
    ctx.close()


def test_forced_episode_closed_form(orc):
    """Every policy with zero weights and b3 = (0, 0, 100, 0, 0): the speaker
    sends message 2 and the listener pushes -x in every step. From rest the
    listener follows v_k = -0.4 (1 - 0.75^k), p_k = p_0 - 0.04 (k - 3 (1 - 0.75^k))
    along x; the GPU's observations and rewards must follow that closed form
    (rewards: minus the listener's fp64 distance to the target)."""
    need_gpu()
    V, T = 64, 25
    w = workloads.speaker_listener(n_envs=V, pop=2, envs_per_pair=16, seed=4)
    for p in w.policies:
        p.params[:] = 0.0
        p.params[-3] = 100.0                              # b3[2]: message 2 / move -x
    ctx = context()
    load_population(ctx, w)
    g = rollout(ctx, w, 1, w.seed)
    ctx.close()
    assert np.all(g["action"] == 2)
    for env in range(V):
        st = orc.sl_reset(env, w.seed).astype(np.float64)
        tgt = int(st[14])
        for t in range(T):
            obs = g["obs"][0, t, env]
            np.testing.assert_array_equal(obs[0, :11], np.eye(11)[tgt])
            np.testing.assert_allclose(obs[1, 0], -0.4 * (1 - 0.75 ** t), atol=1e-6)
            np.testing.assert_array_equal(obs[1, 8:11], [0, 0, 0] if t == 0 else [0, 0, 1])
            k = t + 1
            p = st[4:6] - [0.04 * (k - 3 * (1 - 0.75 ** k)), 0.0]
            d = np.hypot(*(p - st[8 + 2 * tgt: 10 + 2 * tgt]))
            np.testing.assert_allclose(g["reward"][0, t, env], [-d, -d], atol=2e-5)
