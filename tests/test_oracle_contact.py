"""Oracle pins for the contact model and the scenarios that use it (App. B.1:
agents that collide, "obstacles block the way"; simple push, simple tag, and
spread with contact forces between its agents).

Checks that do not go through the oracle's own arithmetic: log1p against the
library routine, the contact force against its formula evaluated in fp64 with
numpy, exactly zero force beyond the margin, equal and opposite pair forces,
total velocity under contact against the closed form of the damped dynamics
(pair forces cancel), bit-identical steps with and without contact when no
pair is in range, a hand-worked push geometry, the tag speed limits against the
closed form of the capped recursion, the tag hit rule recomputed in fp64 from
the returned positions, an obstacle that pushes but does not move, the
observation layouts element by element, and the resets against the spread
reset (same chance counters)."""
import math

import numpy as np
import pytest

import oracle

pytestmark = pytest.mark.filterwarnings("ignore")

K, FC = 1e-3, 100.0          # contact margin and force scale (stated readings)


def ulp_diff(a, b):
    a = np.asarray(a, np.float32).view(np.int32).astype(np.int64)
    b = np.asarray(b, np.float32).view(np.int32).astype(np.int64)
    return np.abs(a - b)


def test_log1p_against_library():
    x = np.concatenate([np.linspace(0, 1, 20001, dtype=np.float32),
                        np.float32(2.0) ** -np.arange(1, 120, dtype=np.float32)])
    y = oracle.det_log1pf(x)
    ref = np.log1p(x.astype(np.float64)).astype(np.float32)
    assert ulp_diff(y, ref).max() <= 2
    assert y[0] == 0.0


def force64(a, b, dmin):
    d = np.subtract(a, b, dtype=np.float64)
    r = math.hypot(*d)
    pen = K * math.log1p(math.exp(-(r - dmin) / K)) if (dmin - r) / K < 30 else (dmin - r)
    return FC * pen * d / r


@pytest.mark.parametrize("a,b,dmin", [((0.0, 0.0), (0.29, 0.0), 0.3), ((0.1, -0.2), (0.2, 0.0), 0.3),
                                      ((0.5, 0.5), (0.45, 0.52), 0.125), ((0.0, 0.0), (0.3, 0.0), 0.3),
                                      ((0.0, 0.0), (0.0, 0.31), 0.3), ((0.3, 0.1), (0.1, 0.2), 0.275)])
def test_contact_force_formula(a, b, dmin):
    f, on = oracle.contact_force(a, b, dmin)
    assert on
    np.testing.assert_allclose(f, force64(a, b, dmin), rtol=2e-4, atol=1e-9)
    # equal and opposite, bit for bit
    g, on2 = oracle.contact_force(b, a, dmin)
    assert on2 and np.array_equal(g, -f)


def test_contact_force_zero_beyond_margin():
    for gap in (0.0875, 0.1, 0.5, 2.0):
        f, on = oracle.contact_force((0.0, 0.0), (0.3 + gap, 0.0), 0.3)
        assert not on and np.all(f == 0)
    # just inside the margin a (tiny) force still acts, pointing away from b
    f, on = oracle.contact_force((0.0, 0.0), (0.3 + 0.05, 0.0), 0.3)
    assert on and f[0] < 0 and f[1] == 0
    # coincident centres: no direction, no force
    f, on = oracle.contact_force((0.2, 0.2), (0.2, 0.2), 0.3)
    assert not on


def spread_state(pos, vel, lm):
    N, L = len(pos), len(lm)
    st = np.zeros(4 * N + 2 * L, np.float32)
    for i in range(N):
        st[4 * i:4 * i + 4] = [pos[i][0], pos[i][1], vel[i][0], vel[i][1]]
    for l in range(L):
        st[4 * N + 2 * l:4 * N + 2 * l + 2] = lm[l]
    return st


def test_spread_contact_reduces_to_spread_out_of_range():
    st = spread_state([(-0.8, -0.8), (0.0, 0.1), (0.7, -0.5)], [(0.1, 0.0), (0.0, -0.2), (0.05, 0.05)],
                      [(0.2, 0.2), (-0.3, 0.4), (0.9, 0.9)])
    for acts in ([0, 0, 0], [1, 2, 3], [4, 4, 1]):
        s1, r1 = oracle.spread_step(st, 3, 3, acts)
        s2, r2 = oracle.spread_step(st, 3, 3, acts, contact=True)
        assert np.array_equal(s1, s2) and np.array_equal(r1, r2)


def test_spread_contact_equal_and_opposite():
    # agents 0 and 1 overlap (0.2 < 0.3) at rest, agent 2 far away; no action
    st = spread_state([(0.0, 0.0), (0.12, 0.16), (0.9, -0.9)], [(0, 0)] * 3, [(0.5, 0.5)] * 3)
    s2, _ = oracle.spread_step(st, 3, 3, [0, 0, 0], contact=True)
    v = s2[:12].reshape(3, 4)[:, 2:]
    assert np.array_equal(v[0], -v[1]) and np.all(v[2] == 0)
    f = force64((0.0, 0.0), (0.12, 0.16), 0.3)
    np.testing.assert_allclose(v[0], 0.1 * f, rtol=2e-4)
    # pushed apart along the line of centres
    assert v[0][0] < 0 and v[0][1] < 0
    np.testing.assert_allclose(v[0][1] / v[0][0], 0.16 / 0.12, rtol=1e-5)


def test_spread_contact_total_velocity_closed_form():
    """Pair forces cancel, so sum_i v_i follows the damped recursion of the
    summed action forces alone: S_{t+1} = 0.75 S_t + 0.1 sum_i u_i(t)."""
    rng = np.random.default_rng(11)
    N = 4
    pos = rng.uniform(-0.25, 0.25, size=(N, 2))           # a crowd: many overlaps
    st = spread_state(pos, [(0, 0)] * N, [(0.0, 0.0)] * N)
    S = np.zeros(2)
    unit = {0: (0, 0), 1: (1, 0), 2: (-1, 0), 3: (0, 1), 4: (0, -1)}
    moved = False
    for t in range(30):
        acts = rng.integers(0, 5, size=N)
        st2, _ = oracle.spread_step(st, N, N, acts, contact=True)
        S = 0.75 * S + 0.1 * np.sum([unit[int(a)] for a in acts], axis=0)
        v = st2[:4 * N].reshape(N, 4)[:, 2:].astype(np.float64)
        np.testing.assert_allclose(v.sum(0), S, atol=2e-5)
        no_contact, _ = oracle.spread_step(st, N, N, acts)
        moved |= not np.array_equal(no_contact, st2)
        st = st2
    assert moved                                          # contacts did act


def test_push_hand_worked():
    # landmark at the origin; adversary 0.5 away (3-4-5), good agent 1.0 away; far apart, at rest
    st = spread_state([(0.3, 0.4), (-0.6, -0.8)], [(0, 0)] * 2, [(0.0, 0.0)])
    s2, r = oracle.push_step(st, [0, 0])
    assert np.array_equal(s2, st)
    assert abs(r[1] - (-1.0)) < 1e-6 and abs(r[0] - (1.0 - 0.5)) < 1e-6
    o = oracle.push_obs(st)
    f = np.float32
    p0, p1 = (f(0.3), f(0.4)), (f(-0.6), f(-0.8))
    np.testing.assert_array_equal(o[0], np.array([0, 0, *p0, -p0[0], -p0[1], p1[0] - p0[0], p1[1] - p0[1]], f))
    np.testing.assert_array_equal(o[1], np.array([0, 0, *p1, -p1[0], -p1[1], p0[0] - p1[0], p0[1] - p1[1]], f))


def test_push_contact_pushes_both():
    # the adversary moves into the good agent: contact acts on both, equal and opposite
    st = spread_state([(0.0, 0.0), (0.25, 0.0)], [(0.0, 0.0), (0.0, 0.0)], [(0.8, 0.0)])
    s2, r = oracle.push_step(st, [1, 0])
    v = s2[:8].reshape(2, 4)[:, 2:]
    f = force64((0.0, 0.0), (0.25, 0.0), 0.3)
    np.testing.assert_allclose(v[1], -0.1 * f, rtol=2e-4)
    np.testing.assert_allclose(v[0], 0.1 * (np.array([1.0, 0.0]) + f), rtol=2e-4)
    p = s2[:8].reshape(2, 4)[:, :2].astype(np.float64)
    d = np.hypot(*(p - [0.8, 0.0]).T)
    np.testing.assert_allclose(r, [d[1] - d[0], -d[1]], atol=1e-6)


def test_resets_are_the_spread_reset():
    for g in (0, 7, 123456789):
        np.testing.assert_array_equal(oracle.push_reset(g, 99), oracle.spread_reset(2, 1, g, 99))
        np.testing.assert_array_equal(oracle.tag_reset(g, 99), oracle.spread_reset(4, 2, g, 99))


def tag_state(pos, vel, obst):
    return spread_state(pos, vel, obst)


FAR = [(-0.9, 0.9), (-0.9, -0.9), (0.9, -0.9)]


def test_tag_speed_limits_closed_form():
    """From rest, a lone agent pushed +x each step follows v <- min(0.75 v +
    0.1 a, vmax): a = 4, vmax = 1.3 for the good agent; a = 3, vmax = 1.0 for
    an adversary (both limits are reached)."""
    for who, a, vmax in ((3, 4.0, 1.3), (0, 3.0, 1.0)):
        pos = [(-0.9, 0.5), (-0.9, -0.5), (0.9, 0.6), (0.9, -0.6)]
        pos[who] = (-3.0, 0.0)                        # far from everything, moving +x
        st = tag_state(pos, [(0, 0)] * 4, [(0.0, 3.0), (0.0, -3.0)])
        v = 0.0
        capped = False
        for t in range(12):
            acts = [0, 0, 0, 0]
            acts[who] = 1
            st, _ = oracle.tag_step(st, acts)
            v = min(0.75 * v + 0.1 * a, vmax)
            capped |= v == vmax
            assert abs(st[4 * who + 2] - v) < 2e-6 and st[4 * who + 3] == 0
        assert capped


def test_tag_speed_limit_direction_kept():
    # a diagonal velocity above the limit is scaled back along its direction
    st = tag_state([(0.0, 0.0), (-0.9, -0.9), (0.9, -0.9), (0.9, 0.9)], [(1.2, 1.2), (0, 0), (0, 0), (0, 0)],
                   [(3.0, 3.0), (-3.0, 3.0)])
    s2, _ = oracle.tag_step(st, [0, 0, 0, 0])
    vx, vy = s2[2], s2[3]
    assert abs(math.hypot(vx, vy) - 1.0) < 1e-6 and vx == vy


def test_tag_hits_and_rewards():
    # adversary 0 closes on the good agent at speed 1: 0.19 apart, after the move 0.115 < 0.125
    pos = [(-0.19, 0.0), (-0.9, 0.9), (0.9, -0.9), (0.0, 0.0)]
    st = tag_state(pos, [(1.0, 0.0), (0, 0), (0, 0), (0, 0)], [(0.0, 3.0), (0.0, -3.0)])
    s2, r = oracle.tag_step(st, [0, 0, 0, 0])
    p = s2[:16].reshape(4, 4)[:, :2].astype(np.float64)
    d = np.hypot(*(p[:3] - p[3]).T)
    hits = int(np.sum(d < 0.125))
    assert hits == 1
    np.testing.assert_array_equal(r, np.float32([10, 10, 10, -10]))
    # two adversaries on the good agent at once
    pos = [(-0.19, 0.0), (0.19, 0.0), (0.9, -0.9), (0.0, 0.0)]
    st = tag_state(pos, [(1.0, 0.0), (-1.0, 0.0), (0, 0), (0, 0)], [(0.0, 3.0), (0.0, -3.0)])
    s2, r = oracle.tag_step(st, [0, 0, 0, 0])
    p = s2[:16].reshape(4, 4)[:, :2].astype(np.float64)
    assert int(np.sum(np.hypot(*(p[:3] - p[3]).T) < 0.125)) == 2
    np.testing.assert_array_equal(r, np.float32([20, 20, 20, -20]))
    # nobody close: no reward
    st = tag_state(FAR + [(0.0, 0.0)], [(0, 0)] * 4, [(0.0, 3.0), (0.0, -3.0)])
    _, r = oracle.tag_step(st, [0, 0, 0, 0])
    assert np.all(r == 0)


def test_tag_obstacle_pushes_and_stays():
    # the good agent overlaps obstacle 0 (0.2 apart < 0.05 + 0.2), at rest, no action
    st = tag_state(FAR + [(0.2, 0.0)], [(0, 0)] * 4, [(0.0, 0.0), (0.0, 3.0)])
    s2, _ = oracle.tag_step(st, [0, 0, 0, 0])
    f = force64((0.2, 0.0), (0.0, 0.0), 0.25)
    np.testing.assert_allclose(s2[14:16], 0.1 * f, rtol=2e-4)
    assert s2[14] > 0 and s2[15] == 0                   # away from the obstacle
    np.testing.assert_array_equal(s2[16:], st[16:])     # obstacles do not move
    assert np.all(s2[:12] == st[:12])                   # the far adversaries are untouched


def test_tag_observation_layout():
    pos = [(0.1, 0.2), (-0.3, 0.4), (0.5, -0.6), (0.7, 0.8)]
    vel = [(0.01, 0.02), (0.03, 0.04), (0.05, 0.06), (0.07, 0.08)]
    ob = [(0.9, -0.1), (-0.2, -0.9)]
    o = oracle.tag_obs(tag_state(pos, vel, ob))
    f = np.float32
    for i in range(4):
        px, py = f(pos[i][0]), f(pos[i][1])
        exp = [f(vel[i][0]), f(vel[i][1]), px, py]
        for l in range(2):
            exp += [f(ob[l][0]) - px, f(ob[l][1]) - py]
        for j in range(4):
            if j != i:
                exp += [f(pos[j][0]) - px, f(pos[j][1]) - py]
        exp += [f(vel[3][0]), f(vel[3][1])] if i < 3 else [0.0, 0.0]
        np.testing.assert_array_equal(o[i], np.array(exp, np.float32))
