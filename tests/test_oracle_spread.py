"""Pins for the oracle's particle spread: closed-form single steps, velocity
damping, exact distances on 3-4-5 triangles, collision counting and the
observation layout, and two forced-action episodes with closed forms (at rest;
under a constant force). The return under sampled policies has no closed form
("parity unpinned" beyond these)."""
import numpy as np

import workloads

f32 = np.float32


def state(agents, landmarks):
    s = []
    for (px, py, vx, vy) in agents:
        s += [px, py, vx, vy]
    for (lx, ly) in landmarks:
        s += [lx, ly]
    return np.array(s, f32)


def test_single_step_closed_form(orc):
    st = state([(0, 0, 0, 0), (0.5, 0.5, 0.2, -0.4)], [(0.375, 0.5), (0.5, 0.5)])
    new, r = orc.spread_step(st, 2, 2, [1, 0])
    # agent 0: v = 0*0.75 + 0.1 ; p = 0 + v*0.1 (fp32)
    assert new[2] == f32(0.1) and new[3] == 0.0
    assert new[0] == f32(f32(0.1) * f32(0.1)) and new[1] == 0.0
    # agent 1, no force: v = v*0.75, p += v*0.1
    v = f32(f32(0.2) * f32(0.75)), f32(f32(-0.4) * f32(0.75))
    assert new[6] == v[0] and new[7] == v[1]
    assert new[4] == f32(f32(0.5) + f32(v[0] * f32(0.1)))
    assert new[5] == f32(f32(0.5) + f32(v[1] * f32(0.1)))
    assert r[0] == r[1] and r[0] < 0


def test_damping_geometric(orc):
    st = state([(0, 0, 1.0, -1.0)], [(0.0, 0.0)])
    for t in range(1, 12):
        st, _ = orc.spread_step(st, 1, 1, [0])
        assert st[2] == 0.75 ** t and st[3] == -(0.75 ** t)   # exact: 3^t < 2^24


def test_zero_action_zero_velocity_is_fixed(orc):
    st = state([(0.3, -0.7, 0, 0), (-0.2, 0.1, 0, 0), (0.9, 0.9, 0, 0)],
               [(0, 0), (1, 1), (-1, -1)])
    new, r = orc.spread_step(st.copy(), 3, 3, [0, 0, 0])
    np.testing.assert_array_equal(new, st)
    assert np.all(r < 0)


def test_reward_exact_distances_and_collisions(orc):
    # agents: a at (0,0); b at (0.15, 0.2) -> |a-b| = 0.25 < 0.3 (collision);
    # c at (-0.375, -0.5) -> |a-c| = 0.625. Landmarks: (0.375, 0.5) nearest a
    # (0.625) vs b: (0.225, 0.3) -> 0.375; (0, 0) -> a at 0; (-0.375,-0.5) -> c 0.
    # Positions do not move: zero velocity, zero action.
    st = state([(0, 0, 0, 0), (0.15, 0.2, 0, 0), (-0.375, -0.5, 0, 0)],
               [(0.375, 0.5), (0, 0), (-0.375, -0.5)])
    _, r = orc.spread_step(st, 3, 3, [0, 0, 0])
    # 0.375-0.15 and 0.5-0.2 are computed in fp32 by the step
    dx, dy = f32(f32(0.375) - f32(0.15)), f32(f32(0.5) - f32(0.2))
    d_b = np.sqrt(f32(dx * dx + dy * dy), dtype=f32)
    cover = f32(f32(d_b + f32(0)) + f32(0))
    assert abs(float(d_b) - 0.375) < 1e-7
    np.testing.assert_array_equal(r, -np.array([cover + 1, cover + 1, cover], f32))
    # at exactly 0.3125 apart nobody collides
    st = state([(0, 0, 0, 0), (0.1875, 0.25, 0, 0)], [(0, 0), (0.1875, 0.25)])
    _, r = orc.spread_step(st, 2, 2, [0, 0])
    assert np.all(r == 0.0)


def test_observation_layout(orc):
    st = state([(0.5, -0.25, 0.125, 0.0625), (0.0, 0.5, 0, 0), (-1.0, 0.75, 0, 0)],
               [(1, 1), (0, 0), (-0.5, 0.5)])
    o = orc.spread_obs(st, 3, 3, 18)
    want0 = [0.125, 0.0625, 0.5, -0.25, 0.5, 1.25, -0.5, 0.25, -1.0, 0.75,
             -0.5, 0.75, -1.5, 1.0, 0, 0, 0, 0]
    np.testing.assert_array_equal(o[0], np.array(want0, f32))
    want2 = [0, 0, -1.0, 0.75, 2.0, 0.25, 1.0, -0.75, 0.5, -0.25, 1.5, -1.0, 1.0, -0.25, 0, 0, 0, 0]
    np.testing.assert_array_equal(o[2], np.array(want2, f32))
    o8 = orc.spread_obs(np.zeros(4 * 8 + 16, f32), 8, 8, 34)
    assert o8.shape == (8, 34)


def test_reset_uniform(orc):
    xs = np.stack([orc.spread_reset(3, 3, g, 17) for g in range(4000)])
    pos = xs[:, [0, 1, 4, 5, 8, 9, 12, 13, 14, 15, 16, 17]]
    assert pos.min() >= -1.0 and pos.max() < 1.0
    assert abs(pos.mean()) < 0.02 and abs(pos.var() - 1 / 3) < 0.02
    assert np.all(xs[:, [2, 3, 6, 7, 10, 11]] == 0)


def test_rollout_invariants_and_replay(orc):
    w = workloads.spread(n_agents=3, n_envs=64, pop=4, envs_per_pair=16, with_bias=True,
                         n_episodes=2, seed=21)
    params = [p.params for p in w.policies]
    dims = w.policies[0].dims
    out = orc.spread_rollout(params, dims, 3, 3, 25, 64, w.pair_ids, 2, w.seed)
    r = out["reward"]
    assert np.all(r <= 0)
    # agents share the cover term; differences are whole collision counts
    # (up to the fp32 rounding of cover + count)
    d = r - r.max(axis=-1, keepdims=True)
    np.testing.assert_allclose(d, np.round(d), atol=1e-5)
    assert np.any(d < -0.5)
    # first-step observations hold zero velocity and the reset positions
    for g_env in range(4):
        st = orc.spread_reset(3, 3, g_env, w.seed)
        np.testing.assert_array_equal(out["obs"][0, 0, g_env], orc.spread_obs(st, 3, 3, 18))
    # stepping the recorded actions reproduces the recorded rewards and obs
    st = orc.spread_reset(3, 3, 64 + 5, w.seed)       # episode 1, env 5
    for t in range(25):
        np.testing.assert_array_equal(out["obs"][1, t, 5], orc.spread_obs(st, 3, 3, 18))
        st, rew = orc.spread_step(st, 3, 3, out["action"][1, t, 5].astype(np.int32))
        np.testing.assert_array_equal(out["reward"][1, t, 5], rew)
    # logits are the policy forward of the recorded observations
    row = 5 // 16
    for i in range(3):
        lg = orc.mlp_forward(params[w.pair_ids[row][i]], dims, out["obs"][1, :, 5, i])
        np.testing.assert_array_equal(lg, out["logits"][1, :, 5, i])
    # replaying the oracle's own logits reproduces everything
    rep = orc.spread_rollout(params, dims, 3, 3, 25, 64, w.pair_ids, 2, w.seed,
                             ext_logits=out["logits"])
    for k in out:
        np.testing.assert_array_equal(rep[k], out[k])
    # a slice of envs equals the same envs of the full rollout
    sl = orc.spread_rollout(params, dims, 3, 3, 25, 64, w.pair_ids, 2, w.seed, env_lo=16, env_hi=40)
    np.testing.assert_array_equal(sl["reward"], out["reward"][:, :, 16:40])


def test_local_ratio_weighting(orc):
    """App. B.1's local_ratio weights the shared cover term by 1 - rho and the
    agent's own collisions by rho. Fixed without retyping the formula: rho = 0
    leaves the same cover reward to every agent, rho = 1 leaves minus the
    collision count, rho = 1/2 halves the unweighted reward exactly (scaling by
    a power of two commutes with rounding), and any rho interpolates between
    the two ends."""
    rng = np.random.default_rng(3)
    for trial in range(40):
        N = 3 if trial % 2 else 8
        st = rng.uniform(-0.6, 0.6, 6 * N).astype(f32)
        for i in range(N):
            st[4 * i + 2:4 * i + 4] *= f32(0.1)
        acts = rng.integers(0, 5, N)
        _, r1 = orc.spread_step(st, N, N, acts)
        _, r0 = orc.spread_step(st, N, N, acts, local_ratio=0.0)
        _, rl = orc.spread_step(st, N, N, acts, local_ratio=1.0)
        _, rh = orc.spread_step(st, N, N, acts, local_ratio=0.5)
        assert np.all(r0 == r0[0]) and r0[0] <= 0
        diff = r0 - r1                                 # (cover + coll) - cover, rounded twice
        coll = np.round(diff)
        assert np.all(np.abs(diff - coll) <= 4 * np.spacing(np.abs(r1))) and np.all(coll >= 0)
        np.testing.assert_array_equal(rl, -coll)
        np.testing.assert_array_equal(rh, r1 * f32(0.5))
        _, rq = orc.spread_step(st, N, N, acts, local_ratio=0.25)
        lo, hi = np.minimum(r0, rl), np.maximum(r0, rl)
        assert np.all(rq >= lo - 1e-6) and np.all(rq <= hi + 1e-6)


def test_rollout_fixed_point_over_an_episode(orc):
    """Logits that force the no-op in every step: resets start at rest, so the
    whole 25-step episode stays at its reset state - observations and rewards
    are the same at every step (a multi-step closed form of the rollout loop)."""
    w = workloads.spread(n_agents=3, n_envs=32, pop=2, envs_per_pair=16, seed=5)
    params = [p.params for p in w.policies]
    dims = w.policies[0].dims
    T = 25
    ext = np.zeros((1, T, 32, 3, 5), np.float32)
    ext[..., 0] = 100.0                                 # probability of the no-op ~ 1 - 4 e^-100
    out = orc.spread_rollout(params, dims, 3, 3, T, 32, w.pair_ids, 1, w.seed, ext_logits=ext)
    assert np.all(out["action"] == 0)
    for env in (0, 7, 31):
        st = orc.spread_reset(3, 3, env, w.seed)
        _, r = orc.spread_step(st, 3, 3, [0, 0, 0])
        for t in range(T):
            np.testing.assert_array_equal(out["obs"][0, t, env], orc.spread_obs(st, 3, 3, 18))
            np.testing.assert_array_equal(out["reward"][0, t, env], r)


def test_rollout_constant_force_closed_form(orc):
    """Logits that force action 1 (+x) in every step. From rest, after k moves
    v_k = 0.4 (1 - 0.75^k) and p_k = p_0 + 0.04 (k - 3 (1 - 0.75^k)) along x,
    with y fixed (Sec. 3.1's rollout over the dynamics of App. B.1). All agents
    drift together, so their collision counts stay those of the reset, and the
    cover term follows from the closed-form positions. The 25-step rollout must
    agree with the fp64 closed form to within fp32 rounding."""
    V, T = 32, 25
    w = workloads.spread(n_agents=3, n_envs=V, pop=2, envs_per_pair=16, seed=6)
    params = [p.params for p in w.policies]
    ext = np.zeros((1, T, V, 3, 5), np.float32)
    ext[..., 1] = 100.0
    out = orc.spread_rollout(params, w.policies[0].dims, 3, 3, T, V, w.pair_ids, 1, w.seed,
                             ext_logits=ext)
    assert np.all(out["action"] == 1)
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
            v = 0.4 * (1 - 0.75 ** t)
            dx = 0.04 * (t - 3 * (1 - 0.75 ** t))
            obs = out["obs"][0, t, env]
            np.testing.assert_allclose(obs[:, 0], v, atol=1e-6)
            np.testing.assert_array_equal(obs[:, 1], 0.0)
            np.testing.assert_allclose(obs[:, 2:4], p0 + [dx, 0.0], atol=5e-6)
            k = t + 1                                     # the reward follows the step's move
            p = p0 + [0.04 * (k - 3 * (1 - 0.75 ** k)), 0.0]
            cover = sum(min(np.hypot(*(p[a] - lm[l])) for a in range(3)) for l in range(3))
            np.testing.assert_allclose(out["reward"][0, t, env], -(cover + coll), atol=5e-5)
        checked += 1
    assert checked >= 24
