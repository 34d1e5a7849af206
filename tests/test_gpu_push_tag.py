"""GPU parity for the simple push and simple tag rollouts (App. B.1; fp32 MLP
policies of hidden width 64), whose agents collide with the soft contact
forces, and for spread with contact forces between its agents (N = 3 on the
fp32 kernel, N = 8 on the tensor cores).

The GPU dumps its logits; the oracle replays the same environments with them:
observations, actions, rewards and done flags must then match bit for bit
(the contact forces included), the observation padding must be zero, and the
GPU logits must match the oracle's own within 1e-5 relative (fp32) or 2e-2
(bf16). The 4,096-env sizes are checked on sampled envs."""
import numpy as np
import pytest

import oracle
import workloads
from gpu_util import context, load_population, logits_close, need_gpu, spec_of

pytestmark = pytest.mark.gpu

from paper_2106_07551_gb300 import MALIB_DUMP_LOGITS, MALIB_SPREAD_CONTACT, MalibError, alloc_traj


def rollout(ctx, w, n_eps, seed, flags=MALIB_DUMP_LOGITS):
    spec = spec_of(w, flags)
    traj = alloc_traj(spec, n_eps, logits=True)
    ctx.rollout(spec, w.pair_ids, n_eps, seed, traj)
    ctx.sync()
    return {k: v.cpu().numpy() for k, v in traj.items()}


def check(replay, w, g, n_eps, seed, env_lo, env_hi, rtol=1e-5):
    params = [p.params for p in w.policies]
    dims = w.policies[0].dims
    sl = slice(env_lo, env_hi)
    ref = replay(params, dims, w.episode_len, w.n_envs, w.pair_ids, n_eps, seed,
                 env_lo=env_lo, env_hi=env_hi, ext_logits=g["logits"][:, :, sl])
    d = w.obs_dim
    np.testing.assert_array_equal(g["obs"][:, :, sl, :, :d], ref["obs"])
    assert np.all(g["obs"][..., d:] == 0)
    np.testing.assert_array_equal(g["action"][:, :, sl].astype(np.int8), ref["action"])
    np.testing.assert_array_equal(g["reward"][:, :, sl], ref["reward"])
    done = g["done"][:, :, sl]
    assert np.all(done[:, -1] == 1) and np.all(done[:, :-1] == 0)
    n_bad, worst = logits_close(g["logits"][:, :, sl], ref["logits"], rtol)
    assert n_bad == 0, (n_bad, worst)
    return ref


@pytest.mark.parametrize("n_envs,epp,n_eps", [(512, 64, 3), (256, 128, 2), (48, 16, 5)])
def test_push_replay_parity(n_envs, epp, n_eps):
    need_gpu()
    w = workloads.push(n_envs=n_envs, pop=5, envs_per_pair=epp, with_bias=True, seed=800 + epp)
    ctx = context()
    load_population(ctx, w)
    g = rollout(ctx, w, n_eps, 1618)
    check(oracle.push_rollout, w, g, n_eps, 1618, 0, n_envs)
    g2 = rollout(ctx, w, n_eps, 1618)
    for k in g:
        np.testing.assert_array_equal(g2[k], g[k])
    ctx.close()


@pytest.mark.parametrize("n_envs,epp,n_eps", [(512, 64, 3), (256, 128, 2), (48, 16, 5)])
def test_tag_replay_parity(n_envs, epp, n_eps):
    need_gpu()
    w = workloads.tag(n_envs=n_envs, pop=5, envs_per_pair=epp, with_bias=True, seed=900 + epp)
    ctx = context()
    load_population(ctx, w)
    g = rollout(ctx, w, n_eps, 31337)
    check(oracle.tag_rollout, w, g, n_eps, 31337, 0, n_envs)
    # the rewards are the hit rule's: +10 h to each adversary, -10 h to the good agent
    r = g["reward"]
    assert np.array_equal(r[..., 0], r[..., 1]) and np.array_equal(r[..., 0], r[..., 2])
    assert np.array_equal(r[..., 3], -r[..., 0]) and np.all(r[..., 0] % 10 == 0)
    g2 = rollout(ctx, w, n_eps, 31337)
    for k in g:
        np.testing.assert_array_equal(g2[k], g[k])
    ctx.close()


def test_push_tag_4096_envs_sampled():
    need_gpu()
    for make, replay in ((workloads.push, oracle.push_rollout), (workloads.tag, oracle.tag_rollout)):
        w = make(n_envs=4096, pop=16)
        ctx = context()
        load_population(ctx, w)
        g = rollout(ctx, w, 2, w.seed)
        for lo, hi in ((0, 40), (2000, 2030), (4090, 4096)):
            check(replay, w, g, 2, w.seed, lo, hi)
        ctx.close()


def contact_differs(w, n_eps, seed, replay_kwargs):
    """The oracle's own rollouts with and without contact differ somewhere (the
    workload does exercise the contact forces)."""
    params = [p.params for p in w.policies]
    a = oracle.spread_rollout(params, w.policies[0].dims, w.n_agents, w.n_landmarks, w.episode_len,
                              w.n_envs, w.pair_ids, n_eps, seed, env_hi=min(w.n_envs, 64),
                              contact=True, **replay_kwargs)
    b = oracle.spread_rollout(params, w.policies[0].dims, w.n_agents, w.n_landmarks, w.episode_len,
                              w.n_envs, w.pair_ids, n_eps, seed, env_hi=min(w.n_envs, 64), **replay_kwargs)
    return not np.array_equal(a["obs"], b["obs"])


def spread_replay(w, bf16=False):
    def replay(params, dims, T, n_envs, pairs, n_eps, seed, env_lo=0, env_hi=None, ext_logits=None):
        return oracle.spread_rollout(params, dims, w.n_agents, w.n_landmarks, T, n_envs, pairs, n_eps,
                                     seed, bf16=bf16, env_lo=env_lo, env_hi=env_hi,
                                     ext_logits=ext_logits, contact=True)
    return replay


@pytest.mark.parametrize("n_envs,epp,n_eps", [(512, 128, 2), (96, 32, 3)])
def test_spread_contact_replay_parity_fp32(n_envs, epp, n_eps):
    need_gpu()
    w = workloads.spread(n_agents=3, n_envs=n_envs, pop=5, envs_per_pair=epp, with_bias=True,
                         seed=1000 + epp)
    assert contact_differs(w, n_eps, 4242, {})
    ctx = context()
    load_population(ctx, w)
    g = rollout(ctx, w, n_eps, 4242, MALIB_DUMP_LOGITS | MALIB_SPREAD_CONTACT)
    check(spread_replay(w), w, g, n_eps, 4242, 0, n_envs)
    plain = rollout(ctx, w, n_eps, 4242)
    assert not np.array_equal(plain["obs"], g["obs"])
    ctx.close()


def test_spread_contact_replay_parity_tensor_cores():
    need_gpu()
    w = workloads.spread(n_agents=8, n_envs=256, pop=5, hidden=256, dtype=workloads.BF16,
                         envs_per_pair=128, with_bias=True, seed=1100)
    ctx = context()
    load_population(ctx, w)
    g = rollout(ctx, w, 2, 5151, MALIB_DUMP_LOGITS | MALIB_SPREAD_CONTACT)
    ref = oracle.spread_rollout([p.params for p in w.policies], w.policies[0].dims, 8, 8, w.episode_len,
                                w.n_envs, w.pair_ids, 2, 5151, bf16=True, ext_logits=g["logits"],
                                contact=True)
    np.testing.assert_array_equal(g["obs"][..., :w.obs_dim], ref["obs"])
    np.testing.assert_array_equal(g["action"].astype(np.int8), ref["action"])
    np.testing.assert_array_equal(g["reward"], ref["reward"])
    n_bad, worst = logits_close(g["logits"], ref["logits"], 2e-2)
    assert n_bad == 0, (n_bad, worst)
    plain = rollout(ctx, w, 2, 5151)
    assert not np.array_equal(plain["obs"], g["obs"])
    ctx.close()


def test_contact_flag_refused_outside_spread():
    need_gpu()
    w = workloads.push(n_envs=64, pop=2, envs_per_pair=16, seed=1)
    ctx = context()
    load_population(ctx, w)
    spec = spec_of(w, MALIB_SPREAD_CONTACT)
    with pytest.raises(MalibError, match="EINVAL"):
        ctx.rollout(spec, w.pair_ids, 1, 0, alloc_traj(spec, 1))
    ctx.close()


@pytest.mark.parametrize("n_envs,epp,n_eps,ratio", [(512, 64, 3, None), (256, 128, 2, 0.2), (48, 16, 5, 1.0)])
def test_reference_replay_parity(n_envs, epp, n_eps, ratio):
    """Simple reference (15 actions: a move and a message), with and without
    local_ratio."""
    need_gpu()
    w = workloads.reference(n_envs=n_envs, pop=5, envs_per_pair=epp, with_bias=True, seed=1200 + epp)
    ctx = context()
    load_population(ctx, w)
    spec = spec_of(w, MALIB_DUMP_LOGITS, local_ratio=ratio)
    traj = alloc_traj(spec, n_eps, logits=True)
    ctx.rollout(spec, w.pair_ids, n_eps, 777, traj)
    ctx.sync()
    g = {k: v.cpu().numpy() for k, v in traj.items()}

    def replay(params, dims, T, n_envs, pairs, n_eps, seed, env_lo=0, env_hi=None, ext_logits=None):
        return oracle.ref_rollout(params, dims, T, n_envs, pairs, n_eps, seed, env_lo=env_lo,
                                  env_hi=env_hi, ext_logits=ext_logits, local_ratio=ratio)

    check(replay, w, g, n_eps, 777, 0, n_envs)
    assert g["action"].max() >= 5                   # messages other than 0 are sent
    ctx.close()
