"""Oracle pins for the simple adversary scenario (App. B.1: one adversary and
two good agents, two landmarks of which one is the target; good agents are
rewarded for being close to the target and for the adversary being far from it,
the adversary for being close to it; the adversary is not told the target).

Checks that do not go through the oracle's own arithmetic: a hand-worked
geometry (3-4-5 triangles), the identity r_good + r_adv = -min over good agents
of the distance to the target recomputed with numpy in fp64, the observation
layout element by element, the dynamics against the spread scenario's (the
scenario reuses them), the reset against the spread reset and the target draw's
distribution, and the swap symmetry of the two good agents."""
import numpy as np
import pytest

import oracle
import workloads

pytestmark = pytest.mark.filterwarnings("ignore")


def make_state(pos, vel, lm, target):
    st = np.zeros(oracle.ADV_STATE, np.float32)
    for i in range(3):
        st[4 * i:4 * i + 4] = [pos[i][0], pos[i][1], vel[i][0], vel[i][1]]
    st[12:16] = [lm[0][0], lm[0][1], lm[1][0], lm[1][1]]
    st[16] = target
    return st


def test_hand_worked_rewards():
    # target (landmark 0) at the origin; adversary 1.0 away, good agents 0.5 and 0.9
    st = make_state(pos=[(0.6, 0.8), (0.3, 0.4), (-0.9, 0.0)], vel=[(0, 0)] * 3,
                    lm=[(0.0, 0.0), (0.9, 0.9)], target=0)
    st2, r = oracle.adversary_step(st, [0, 0, 0])
    np.testing.assert_array_equal(st2, st)                  # no force, no velocity: no move
    assert abs(r[0] - (-1.0)) < 1e-6
    assert abs(r[1] - 0.5) < 1e-6 and r[1] == r[2]
    # the same geometry around landmark 1 as the target
    st = make_state(pos=[(0.9 + 0.6, 0.9 + 0.8), (0.9 - 0.3, 0.9 - 0.4), (0.9, 0.9 - 0.9)],
                    vel=[(0, 0)] * 3, lm=[(0.0, 0.0), (0.9, 0.9)], target=1)
    _, r = oracle.adversary_step(st, [0, 0, 0])
    assert abs(r[0] - (-1.0)) < 2e-6 and abs(r[1] - 0.5) < 2e-6


def test_reward_identity_against_fp64():
    rng = np.random.default_rng(3)
    for _ in range(300):
        pos = rng.uniform(-1, 1, (3, 2))
        vel = rng.uniform(-0.3, 0.3, (3, 2))
        lm = rng.uniform(-1, 1, (2, 2))
        tgt = int(rng.integers(0, 2))
        st = make_state(pos, vel, lm, tgt)
        act = rng.integers(0, 5, 3)
        st2, r = oracle.adversary_step(st, act)
        p = st2[:12].reshape(3, 4)[:, :2].astype(np.float64)
        t = st2[12:16].reshape(2, 2)[tgt].astype(np.float64)
        d = np.linalg.norm(p - t, axis=1)
        assert abs(float(r[0]) + d[0]) < 2e-6
        assert abs(float(r[1]) - (-min(d[1], d[2]) + d[0])) < 4e-6
        assert r[1] == r[2]
        assert abs(float(r[0]) + float(r[1]) + min(d[1], d[2])) < 4e-6


def test_observation_layout():
    rng = np.random.default_rng(4)
    st = make_state(rng.uniform(-1, 1, (3, 2)), rng.uniform(-0.2, 0.2, (3, 2)),
                    rng.uniform(-1, 1, (2, 2)), 1)
    o = oracle.adversary_obs(st)
    ag = st[:12].reshape(3, 4)
    lm = st[12:16].reshape(2, 2)
    for i in range(3):
        np.testing.assert_array_equal(o[i, 0:2], ag[i, 2:4])              # velocity
        np.testing.assert_array_equal(o[i, 2:4], ag[i, 0:2])              # position
        if i == 0:
            np.testing.assert_array_equal(o[i, 4:6], [0, 0])              # target not told
        else:
            np.testing.assert_array_equal(o[i, 4:6], lm[1] - ag[i, 0:2])
            np.testing.assert_array_equal(o[i, 4:6], o[i, 8:10])          # = landmark 1's slot
        np.testing.assert_array_equal(o[i, 6:8], lm[0] - ag[i, 0:2])
        np.testing.assert_array_equal(o[i, 8:10], lm[1] - ag[i, 0:2])
        others = [j for j in range(3) if j != i]
        for k, j in enumerate(others):
            np.testing.assert_array_equal(o[i, 10 + 2 * k:12 + 2 * k], ag[j, 0:2] - ag[i, 0:2])


def test_dynamics_are_the_spread_dynamics():
    rng = np.random.default_rng(5)
    st = oracle.adversary_reset(11, 99)
    sp = np.concatenate([st[:12], st[12:16]]).astype(np.float32)
    for _ in range(25):
        act = rng.integers(0, 5, 3)
        st, _ = oracle.adversary_step(st, act)
        sp, _ = oracle.spread_step(sp, 3, 2, act)
        np.testing.assert_array_equal(st[:16], sp)


def test_reset_and_target_draw():
    seed = 2106075510
    t = []
    for g in range(4000):
        st = oracle.adversary_reset(g, seed)
        if g < 50:
            sp = oracle.spread_reset(3, 2, g, seed)
            np.testing.assert_array_equal(st[:16], sp)
            np.testing.assert_array_equal(oracle.adversary_reset(g, seed), st)   # deterministic
        assert st[16] in (0.0, 1.0)
        t.append(st[16])
    frac = float(np.mean(t))
    assert abs(frac - 0.5) < 5 * np.sqrt(0.25 / len(t))
    # the target depends on the seed too
    assert any(oracle.adversary_reset(g, 1)[16] != oracle.adversary_reset(g, 2)[16] for g in range(64))


def test_good_agents_swap_symmetry():
    rng = np.random.default_rng(6)
    for _ in range(50):
        pos = rng.uniform(-1, 1, (3, 2))
        vel = rng.uniform(-0.2, 0.2, (3, 2))
        lm = rng.uniform(-1, 1, (2, 2))
        tgt = int(rng.integers(0, 2))
        a = make_state(pos, vel, lm, tgt)
        b = make_state(pos[[0, 2, 1]], vel[[0, 2, 1]], lm, tgt)
        oa, ob = oracle.adversary_obs(a), oracle.adversary_obs(b)
        np.testing.assert_array_equal(oa[1], ob[2])
        np.testing.assert_array_equal(oa[2], ob[1])
        act = rng.integers(0, 5, 3)
        a2, ra = oracle.adversary_step(a, act)
        b2, rb = oracle.adversary_step(b, act[[0, 2, 1]])
        np.testing.assert_array_equal(ra, rb)


def test_rollout_replays_the_step_function():
    """The rollout's stored observations and rewards are those of reset + obs +
    step driven by its own actions."""
    rng = np.random.default_rng(7)
    dims = (14, 16, 16, 5)
    params = []
    for _ in range(4):
        parts = []
        for fi, fo in zip(dims[:-1], dims[1:]):
            parts.append(rng.normal(0, 1 / np.sqrt(fi), (fo, fi)).astype(np.float32).ravel())
            parts.append(rng.normal(0, 0.1, fo).astype(np.float32))
        params.append(np.concatenate(parts))
    pairs = np.array([[0, 1, 2], [3, 2, 1]], np.int32)
    T, n_envs, n_eps, seed = 6, 8, 2, 31
    out = oracle.adversary_rollout(params, dims, T, n_envs, pairs, n_eps, seed)
    for ep in range(n_eps):
        for e in range(n_envs):
            st = oracle.adversary_reset(ep * n_envs + e, seed)
            for t in range(T):
                np.testing.assert_array_equal(out["obs"][ep, t, e], oracle.adversary_obs(st))
                st, r = oracle.adversary_step(st, out["action"][ep, t, e].astype(np.int32))
                np.testing.assert_array_equal(out["reward"][ep, t, e], r)


def test_forced_episode_closed_form(orc):
    """A whole 25-step episode in which every agent pushes +x. From rest all
    three follow v_k = 0.4 (1 - 0.75^k), p_k = p_0 + 0.04 (k - 3 (1 - 0.75^k))
    along x; the rewards, recomputed in fp64 from those positions, are
    -d(p_0) for the adversary and -min(d(p_1), d(p_2)) + d(p_0) for both good
    agents, d the distance to the target landmark."""
    V, T = 16, 25
    w = workloads.adversary(n_envs=V, pop=2, envs_per_pair=8, seed=3)
    params = [p.params for p in w.policies]
    ext = np.zeros((1, T, V, 3, 5), np.float32)
    ext[..., 1] = 100.0
    out = orc.adversary_rollout(params, w.policies[0].dims, T, V, w.pair_ids, 1, w.seed,
                                ext_logits=ext)
    assert np.all(out["action"] == 1)
    for env in range(V):
        st = orc.adversary_reset(env, w.seed).astype(np.float64)
        p0 = st[:12].reshape(3, 4)[:, :2]
        target = st[12 + 2 * int(st[16]): 14 + 2 * int(st[16])]
        for t in range(T):
            np.testing.assert_allclose(out["obs"][0, t, env, :, 0], 0.4 * (1 - 0.75 ** t), atol=1e-6)
            k = t + 1
            p = p0 + [0.04 * (k - 3 * (1 - 0.75 ** k)), 0.0]
            d = np.hypot(*(p - target).T)
            want = [-d[0], -min(d[1], d[2]) + d[0], -min(d[1], d[2]) + d[0]]
            np.testing.assert_allclose(out["reward"][0, t, env], want, atol=5e-5)
