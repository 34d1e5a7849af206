"""Oracle pins for the simple reference scenario (App. B.1: two agents, three
landmarks; each agent's goal is known only to the other; both speak and move;
local and global distance terms weighted by local_ratio).

Checks that do not go through the oracle's own arithmetic: a hand-worked
geometry (3-4-5 triangles) for the reward at two local_ratio values, the
observation layout element by element, the one-step message delay, the move
part of an action against the spread dynamics, the reset against the spread
reset and the goal draws' distribution."""
import numpy as np
import pytest

import oracle

pytestmark = pytest.mark.filterwarnings("ignore")


def state(pos, vel, lm, goals, msgs=(-1, -1)):
    st = np.zeros(oracle.REF_STATE, np.float32)
    for i in range(2):
        st[4 * i:4 * i + 4] = [pos[i][0], pos[i][1], vel[i][0], vel[i][1]]
    for l in range(3):
        st[8 + 2 * l:10 + 2 * l] = lm[l]
    st[14:16] = goals
    st[16:18] = msgs
    return st


LM = [(0.0, 0.0), (0.6, -0.8), (-0.9, 0.9)]


@pytest.mark.parametrize("rho", [0.5, 0.2])
def test_hand_worked_rewards(rho):
    # agent 0 is 0.5 from its goal (landmark 0), agent 1 is 1.0 from its goal (landmark 1)
    st = state([(0.3, 0.4), (0.6 + 0.6, -0.8 + 0.8)], [(0, 0), (0, 0)], LM, (0, 1))
    st2, r = oracle.ref_step(st, [0, 0], rho)
    assert np.array_equal(st2[:14], st[:14])               # no force, no velocity: no move
    mean = (0.5 + 1.0) / 2
    np.testing.assert_allclose(r, [-((1 - rho) * mean + rho * 0.5), -((1 - rho) * mean + rho * 1.0)],
                               rtol=1e-6)


def test_observation_layout_and_message_delay():
    pos = [(0.1, 0.2), (-0.3, 0.4)]
    vel = [(0.01, -0.02), (0.03, 0.04)]
    st = state(pos, vel, LM, (2, 0))
    o = oracle.ref_obs(st)
    f = np.float32
    for i in range(2):
        j = 1 - i
        exp = [f(vel[i][0]), f(vel[i][1])]
        for l in range(3):
            exp += [f(LM[l][0]) - f(pos[i][0]), f(LM[l][1]) - f(pos[i][1])]
        goal = [0.0, 0.0, 0.0]
        goal[(2, 0)[j]] = 1.0
        exp += goal + [0.0, 0.0, 0.0]                       # no message before the first step
        np.testing.assert_array_equal(o[i], np.array(exp, np.float32))
    # agent 0 says 1 and moves +x; agent 1 says 2 and stays: seen one step later
    st2, _ = oracle.ref_step(st, [5 * 1 + 1, 5 * 2 + 0])
    o2 = oracle.ref_obs(st2)
    np.testing.assert_array_equal(o2[0, 11:14], [0, 0, 1])   # agent 0 hears agent 1's message 2
    np.testing.assert_array_equal(o2[1, 11:14], [0, 1, 0])   # agent 1 hears agent 0's message 1
    np.testing.assert_array_equal(o2[:, 8:11], o[:, 8:11])   # goals do not change


def test_moves_are_the_spread_dynamics():
    rng = np.random.default_rng(3)
    for _ in range(20):
        pos = rng.uniform(-1, 1, (2, 2))
        vel = rng.uniform(-0.3, 0.3, (2, 2))
        st = state(pos, vel, LM, (0, 1))
        mv = rng.integers(0, 5, 2)
        msg = rng.integers(0, 3, 2)
        st2, _ = oracle.ref_step(st, 5 * msg + mv)
        sp = np.zeros(4 * 2 + 2 * 3, np.float32)
        sp[:8] = st[:8]
        sp[8:14] = st[8:14]
        sp2, _ = oracle.spread_step(sp, 2, 3, mv)
        np.testing.assert_array_equal(st2[:8], sp2[:8])
        np.testing.assert_array_equal(st2[16:18], msg)


def test_reset_is_the_spread_reset_and_goals_are_uniform():
    counts = np.zeros((2, 3))
    for g in range(3000):
        st = oracle.ref_reset(g, 11)
        if g < 5:
            np.testing.assert_array_equal(st[:14], oracle.spread_reset(2, 3, g, 11))
            assert st[16] == -1 and st[17] == -1
        for i in range(2):
            counts[i, int(st[14 + i])] += 1
    # chi-square with 2 degrees of freedom per agent, far from its 1e-6 tail (27.6)
    chi = ((counts - 1000.0) ** 2 / 1000.0).sum(axis=1)
    assert np.all(chi < 27.6)
