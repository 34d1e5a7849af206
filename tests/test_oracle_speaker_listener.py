"""Oracle pins for the simple speaker listener scenario (App. B.1: a speaker
that cannot move and a listener that cannot speak; the listener must navigate
to the target landmark, which only the speaker knows; both are rewarded by the
listener's distance to it, as in the simple reference scenario it resembles).

Checks that do not go through the oracle's own arithmetic: a hand-worked
geometry (a 3-4-5 triangle), the reward against numpy in fp64, the observation
layout element by element, the one-step delay of the message, the speaker never
moving, the listener's dynamics and the reset against the spread scenario's,
the target draw's distribution, and the rollout replaying the step function."""
import numpy as np
import pytest

import oracle
import workloads

pytestmark = pytest.mark.filterwarnings("ignore")


def make_state(pos, vel, lm, target, msg=-1):
    st = np.zeros(oracle.SL_STATE, np.float32)
    for i in range(2):
        st[4 * i:4 * i + 4] = [pos[i][0], pos[i][1], vel[i][0], vel[i][1]]
    st[8:14] = np.asarray(lm, np.float32).ravel()
    st[14] = target
    st[15] = msg
    return st


def test_hand_worked_reward():
    # listener at the origin at rest, target (landmark 1) at (0.3, 0.4): distance 0.5
    st = make_state(pos=[(0.9, 0.9), (0.0, 0.0)], vel=[(0, 0), (0, 0)],
                    lm=[(-0.5, 0.2), (0.3, 0.4), (0.7, -0.7)], target=1)
    st2, r = oracle.sl_step(st, [0, 0])
    assert abs(r[0] + 0.5) < 1e-6 and r[0] == r[1]
    np.testing.assert_array_equal(st2[:14], st[:14])      # nothing moves without force
    assert st2[15] == 0                                    # the message was sent


def test_reward_against_fp64():
    rng = np.random.default_rng(3)
    for _ in range(300):
        pos = rng.uniform(-1, 1, (2, 2))
        vel = np.array([[0, 0], rng.uniform(-0.3, 0.3, 2)])
        lm = rng.uniform(-1, 1, (3, 2))
        tgt = int(rng.integers(0, 3))
        st2, r = oracle.sl_step(make_state(pos, vel, lm, tgt), [int(rng.integers(0, 3)),
                                                             int(rng.integers(0, 5))])
        p = st2[4:6].astype(np.float64)
        d = np.linalg.norm(p - lm[tgt].astype(np.float32).astype(np.float64))
        assert abs(float(r[0]) + d) < 2e-6 and r[0] == r[1]


def test_observation_layout_and_message_delay():
    rng = np.random.default_rng(4)
    st = make_state(rng.uniform(-1, 1, (2, 2)), [(0, 0), (0.05, -0.02)], rng.uniform(-1, 1, (3, 2)),
                    target=2)
    o = oracle.sl_obs(st)
    np.testing.assert_array_equal(o[0], [0, 0, 1] + [0] * 8)          # the speaker knows the target
    np.testing.assert_array_equal(o[1, 0:2], st[6:8])                  # listener velocity
    for l in range(3):
        np.testing.assert_array_equal(o[1, 2 + 2 * l:4 + 2 * l], st[8 + 2 * l:10 + 2 * l] - st[4:6])
    np.testing.assert_array_equal(o[1, 8:11], [0, 0, 0])               # no message yet
    for m in (1, 0, 2):
        st, _ = oracle.sl_step(st, [m, 0])
        o = oracle.sl_obs(st)
        np.testing.assert_array_equal(o[1, 8:11], np.eye(3)[m])        # the message of the last step
        np.testing.assert_array_equal(o[0], [0, 0, 1] + [0] * 8)


def test_speaker_never_moves_and_listener_follows_spread_dynamics():
    rng = np.random.default_rng(5)
    st = oracle.sl_reset(11, 99)
    sp = st[:14].copy()
    for _ in range(25):
        a = [int(rng.integers(0, 3)), int(rng.integers(0, 5))]
        st2, _ = oracle.sl_step(st, a)
        np.testing.assert_array_equal(st2[0:4], st[0:4])               # speaker position, velocity
        sp, _ = oracle.spread_step(sp, 2, 3, [0, a[1]])                # the speaker at rest, noop
        np.testing.assert_array_equal(st2[:14], sp)
        st = st2


def test_reset_and_target_draw():
    seed = 2106075517
    t = []
    for g in range(3000):
        st = oracle.sl_reset(g, seed)
        if g < 50:
            np.testing.assert_array_equal(st[:14], oracle.spread_reset(2, 3, g, seed))
            np.testing.assert_array_equal(oracle.sl_reset(g, seed), st)
            assert st[15] == -1
        t.append(int(st[14]))
    cnt = np.bincount(t, minlength=3)
    chi2 = ((cnt - 1000) ** 2 / 1000).sum()
    assert chi2 < 20.0, cnt      # 2 dof, p ~ 5e-5


def test_rollout_replays_the_step_function():
    rng = np.random.default_rng(7)
    dims = (11, 16, 16, 5)
    params = []
    for _ in range(3):
        parts = []
        for fi, fo in zip(dims[:-1], dims[1:]):
            parts.append(rng.normal(0, 1 / np.sqrt(fi), (fo, fi)).astype(np.float32).ravel())
            parts.append(rng.normal(0, 0.1, fo).astype(np.float32))
        params.append(np.concatenate(parts))
    pairs = np.array([[0, 1], [2, 0]], np.int32)
    T, n_envs, n_eps, seed = 7, 8, 2, 31
    out = oracle.sl_rollout(params, dims, T, n_envs, pairs, n_eps, seed)
    assert out["action"][..., 0].max() <= 2                            # the speaker only speaks
    for ep in range(n_eps):
        for e in range(n_envs):
            st = oracle.sl_reset(ep * n_envs + e, seed)
            for t in range(T):
                np.testing.assert_array_equal(out["obs"][ep, t, e], oracle.sl_obs(st))
                st, r = oracle.sl_step(st, out["action"][ep, t, e].astype(np.int32))
                np.testing.assert_array_equal(out["reward"][ep, t, e], r)


def test_forced_episode_closed_form(orc):
    """A whole 25-step episode with forced actions: the speaker always sends
    message 2 and the listener always pushes +x. The speaker sees the target's
    one-hot at every step; from rest the listener follows v_k = 0.4 (1 - 0.75^k),
    p_k = p_0 + 0.04 (k - 3 (1 - 0.75^k)) along x; both rewards equal minus
    the listener's fp64 distance to the target; the listener sees no message
    at the first step and message 2 from then on."""
    V, T = 16, 25
    w = workloads.speaker_listener(n_envs=V, pop=2, envs_per_pair=8, seed=4)
    params = [p.params for p in w.policies]
    ext = np.zeros((1, T, V, 2, 5), np.float32)
    ext[:, :, :, 0, 2] = 100.0
    ext[:, :, :, 1, 1] = 100.0
    out = orc.sl_rollout(params, w.policies[0].dims, T, V, w.pair_ids, 1, w.seed, ext_logits=ext)
    np.testing.assert_array_equal(out["action"][0, :, :, 0], 2)
    np.testing.assert_array_equal(out["action"][0, :, :, 1], 1)
    for env in range(V):
        st = orc.sl_reset(env, w.seed).astype(np.float64)
        p1 = st[4:6]
        target = st[8 + 2 * int(st[14]): 10 + 2 * int(st[14])]
        for t in range(T):
            obs = out["obs"][0, t, env]
            np.testing.assert_array_equal(obs[0], np.eye(11)[int(st[14])])
            np.testing.assert_allclose(obs[1, 0], 0.4 * (1 - 0.75 ** t), atol=1e-6)
            assert obs[1, 1] == 0.0
            np.testing.assert_array_equal(obs[1, 8:11], [0, 0, 0] if t == 0 else [0, 0, 1])
            k = t + 1
            p = p1 + [0.04 * (k - 3 * (1 - 0.75 ** k)), 0.0]
            np.testing.assert_allclose(out["reward"][0, t, env], -np.hypot(*(p - target)), atol=2e-5)
