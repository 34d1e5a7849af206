"""Oracle pins for the learner-side update (Sec. 3.3 independent learning;
App. C.2 training workflow: Adam, entropy coefficient).

Checks that do not go through the oracle's own arithmetic: the gradient
against central finite differences of the loss and against torch.autograd in
fp64; the loss at hand-worked points (uniform and two-action policies); the
returns-to-go of a hand-worked reward sequence; the sample gathering against
the rollout layout; Adam against its bias-corrected closed form under a
constant gradient."""
import math

import numpy as np
import pytest

from oracle import learner

DIMS = (5, 7, 6, 4)


def n_params(d):
    i, h1, h2, a = d
    return h1 * i + h1 + h2 * h1 + h2 + a * h2 + a


def tiny(seed=0, M=40):
    rng = np.random.default_rng(seed)
    p = rng.normal(0, 0.7, n_params(DIMS))
    obs = rng.normal(0, 1, (M, DIMS[0]))
    act = rng.integers(0, DIMS[3], M)
    ret = rng.normal(0, 2, M)
    return p, obs, act, ret


@pytest.mark.parametrize("beta", [0.0, 0.001, 0.5])
def test_gradient_finite_differences(beta):
    p, obs, act, ret = tiny(1)
    g, (M, b, loss, ent) = learner.pg_grad(p, DIMS, obs, act, ret, beta)
    assert M == 40 and abs(b - ret.mean()) < 1e-15
    h = 1e-6
    fd = np.zeros_like(p)
    for j in range(p.size):
        e = np.zeros_like(p)
        e[j] = h
        fd[j] = (learner.pg_loss(p + e, DIMS, obs, act, ret, beta)[0] -
                 learner.pg_loss(p - e, DIMS, obs, act, ret, beta)[0]) / (2 * h)
    np.testing.assert_allclose(g, fd, rtol=1e-5, atol=1e-8)
    assert abs(loss - learner.pg_loss(p, DIMS, obs, act, ret, beta)[0]) < 1e-12


def test_gradient_autograd():
    torch = pytest.importorskip("torch")
    p, obs, act, ret = tiny(2, M=64)
    beta = 0.01
    g, _ = learner.pg_grad(p, DIMS, obs, act, ret, beta)
    i, h1, h2, a = DIMS
    t = torch.tensor(p, dtype=torch.float64, requires_grad=True)
    o = 0
    W1 = t[o:o + h1 * i].view(h1, i); o += h1 * i
    b1 = t[o:o + h1]; o += h1
    W2 = t[o:o + h2 * h1].view(h2, h1); o += h2 * h1
    b2 = t[o:o + h2]; o += h2
    W3 = t[o:o + a * h2].view(a, h2); o += a * h2
    b3 = t[o:o + a]
    x = torch.tensor(obs)
    z = torch.relu(torch.relu(x @ W1.T + b1) @ W2.T + b2) @ W3.T + b3
    logp = torch.log_softmax(z, dim=1)
    ent = -(logp.exp() * logp).sum(1)
    A = torch.tensor(ret - ret.mean())
    loss = -(A * logp[torch.arange(len(act)), torch.tensor(act)] + beta * ent).mean()
    loss.backward()
    np.testing.assert_allclose(g, t.grad.numpy(), rtol=1e-10, atol=1e-13)


def zero_params(b3):
    p = np.zeros(n_params(DIMS))
    p[-DIMS[3]:] = b3
    return p


def test_loss_hand_worked():
    # zero weights and biases: uniform policy over 4 actions, entropy log 4
    obs = np.ones((2, DIMS[0]))
    loss, ent, b = learner.pg_loss(zero_params([0, 0, 0, 0]), DIMS, obs, np.array([0, 3]),
                                   np.array([1.0, 3.0]), 0.1)
    # advantages -1 and +1 cancel against equal log-probabilities
    assert abs(b - 2.0) < 1e-15 and abs(ent - math.log(4)) < 1e-15
    assert abs(loss - (-0.1 * math.log(4))) < 1e-15
    # b3 = (log 2, 0, 0, 0): pi = (2/5, 1/5, 1/5, 1/5)
    loss, ent, _ = learner.pg_loss(zero_params([math.log(2), 0, 0, 0]), DIMS, obs, np.array([0, 3]),
                                   np.array([1.0, 3.0]), 0.0)
    # -(1/2)[(-1) log(2/5) + (+1) log(1/5)] = -(1/2) log(1/2)
    assert abs(loss - (-0.5 * math.log(0.5))) < 1e-14
    H = -(0.4 * math.log(0.4) + 3 * 0.2 * math.log(0.2))
    assert abs(ent - H) < 1e-14


def test_logit_gradient_hand_worked():
    # one sample at b3 = (log 2, 0, 0, 0): dL/db3 = (1/M) A (pi - onehot) + beta pi (log pi + H), A = 0
    p = zero_params([math.log(2), 0, 0, 0])
    g, _ = learner.pg_grad(p, DIMS, np.ones((1, DIMS[0])), np.array([1]), np.array([5.0]), 0.3)
    pi = np.array([0.4, 0.2, 0.2, 0.2])
    H = -(pi * np.log(pi)).sum()
    np.testing.assert_allclose(g[-4:], 0.3 * pi * (np.log(pi) + H), rtol=1e-13, atol=1e-16)
    assert np.all(g[:-4] == 0)                        # no hidden unit is active


def test_returns_to_go_hand_worked():
    r = np.zeros((1, 3, 1, 2))
    r[0, :, 0, 0] = [1.0, 2.0, 3.0]
    r[0, :, 0, 1] = [0.0, 0.0, 4.0]
    G = learner.returns_to_go(r, 0.5)
    np.testing.assert_allclose(G[0, :, 0, 0], [2.75, 3.5, 3.0])
    np.testing.assert_allclose(G[0, :, 0, 1], [1.0, 2.0, 4.0])
    np.testing.assert_allclose(learner.returns_to_go(r, 0.0)[0, :, 0, 0], [1.0, 2.0, 3.0])


def test_gather_follows_the_rollout_layout():
    E, T, n_envs, N, od = 2, 3, 8, 3, 4
    pairs = np.array([[1, 0, 1], [2, 1, 0]], np.int32)       # 2 combinations of 4 envs
    rng = np.random.default_rng(5)
    traj = {"obs": rng.normal(size=(E, T, n_envs, N, od + 2)).astype(np.float32),
            "action": rng.integers(0, 5, (E, T, n_envs, N)).astype(np.uint8),
            "reward": rng.normal(size=(E, T, n_envs, N)).astype(np.float32)}
    obs, act, ret = learner.gather(traj, pairs, n_envs, N, od, 1, 0.9)
    slots = [(0, 0), (0, 2), (1, 1)]
    assert learner.samples(pairs, n_envs, N, 1) == slots
    assert obs.shape == (len(slots) * E * T * 4, od)
    G = learner.returns_to_go(traj["reward"], 0.9)
    j = 0
    for c, k in slots:
        for e in range(E):
            for t in range(T):
                for v in range(c * 4, c * 4 + 4):
                    assert np.array_equal(obs[j], traj["obs"][e, t, v, k, :od].astype(np.float64))
                    assert act[j] == traj["action"][e, t, v, k] and ret[j] == G[e, t, v, k]
                    j += 1


def test_adam_closed_form():
    # constant gradient: m_hat = g and v_hat = g^2 at every step, so each step
    # moves every parameter by -lr g / (|g| + eps)
    g = np.array([0.5, -2.0, 1e-3, 0.0])
    p = np.array([1.0, 1.0, 1.0, 1.0])
    m = np.zeros(4)
    v = np.zeros(4)
    lr, eps = 1e-2, 1e-8
    for step in range(1, 6):
        p, m, v = learner.adam(p, g, m, v, step, lr, eps=eps)
        np.testing.assert_allclose(p, 1.0 - step * lr * g / (np.abs(g) + eps), rtol=1e-12)
    # a changing scalar gradient against the recursion iterated by hand
    p, m, v = np.array([0.0]), np.zeros(1), np.zeros(1)
    p, m, v = learner.adam(p, [1.0], m, v, 1, 0.1)
    p, m, v = learner.adam(p, [-1.0], m, v, 2, 0.1)
    m2 = 0.9 * 0.1 - 0.1                                   # -0.01
    v2 = 0.999 * 0.001 + 0.001                             # 0.001999
    step2 = 0.1 * (m2 / (1 - 0.81)) / (math.sqrt(v2 / (1 - 0.999 ** 2)) + 1e-8)
    assert abs(p[0] - (-0.1 / (1 + 1e-8) - step2)) < 1e-12


# ---- the PPO variant: clipped surrogate against the behavior policy's logits

def ppo_case(seed, M=48, spread=0.6):
    """A policy, its samples and behavior logits near the policy's own, drawn
    until every ratio is at least 1e-3 from a clip edge (so that central
    differences do not cross a kink)."""
    for s in range(seed, seed + 50):
        p, obs, act, ret = tiny(s, M)
        rng = np.random.default_rng(1000 + s)
        W1, b1, W2, b2, W3, b3 = learner.unpack(p, DIMS)
        z = np.maximum(np.maximum(obs @ W1.T + b1, 0) @ W2.T + b2, 0) @ W3.T + b3
        blog = z + rng.normal(0, spread, z.shape)
        if learner.ppo_margin(p, DIMS, obs, act, blog, 0.2) > 1e-3:
            return p, obs, act, ret, blog
    raise AssertionError("no case with a clear margin")


@pytest.mark.parametrize("beta", [0.0, 0.01])
def test_ppo_gradient_finite_differences(beta):
    p, obs, act, ret, blog = ppo_case(3)
    g, (M, b, loss, ent) = learner.ppo_grad(p, DIMS, obs, act, ret, blog, beta, 0.2)
    h = 1e-6
    fd = np.zeros_like(p)
    for j in range(p.size):
        e = np.zeros_like(p)
        e[j] = h
        fd[j] = (learner.ppo_loss(p + e, DIMS, obs, act, ret, blog, beta, 0.2) -
                 learner.ppo_loss(p - e, DIMS, obs, act, ret, blog, beta, 0.2)) / (2 * h)
    np.testing.assert_allclose(g, fd, rtol=1e-5, atol=1e-8)
    assert abs(loss - learner.ppo_loss(p, DIMS, obs, act, ret, blog, beta, 0.2)) < 1e-12


def test_ppo_some_samples_clipped_both_ways():
    """The case above really exercises both branches of the min."""
    p, obs, act, ret, blog = ppo_case(3)
    W1, b1, W2, b2, W3, b3 = learner.unpack(p, DIMS)
    z = np.maximum(np.maximum(obs @ W1.T + b1, 0) @ W2.T + b2, 0) @ W3.T + b3
    idx = np.arange(obs.shape[0])
    rho = np.exp(learner.log_softmax(z)[idx, act] - learner.log_softmax(blog)[idx, act])
    A = ret - ret.mean()
    assert ((rho > 1.2) & (A > 0)).any() and ((rho < 0.8) & (A < 0)).any()
    assert ((rho < 1.2) & (rho > 0.8)).any()


def test_ppo_on_policy_is_the_policy_gradient():
    """mu = pi: every ratio is 1, the unclipped term is active, and the
    gradient is the policy gradient's; the loss is the entropy term alone
    (the advantages sum to zero)."""
    p, obs, act, ret = tiny(5, M=64)
    W1, b1, W2, b2, W3, b3 = learner.unpack(p, DIMS)
    z = np.maximum(np.maximum(obs @ W1.T + b1, 0) @ W2.T + b2, 0) @ W3.T + b3
    g_ppo, st_ppo = learner.ppo_grad(p, DIMS, obs, act, ret, z, 0.01, 0.2)
    g_pg, st_pg = learner.pg_grad(p, DIMS, obs, act, ret, 0.01)
    np.testing.assert_allclose(g_ppo, g_pg, rtol=1e-12, atol=1e-15)
    assert abs(st_ppo[2] + 0.01 * st_ppo[3]) < 1e-12 and st_ppo[3] == st_pg[3]


def test_ppo_all_clipped_leaves_the_entropy_term():
    """Behavior logits that make every ratio leave the clip range on the side
    where the clipped term is the minimum: the surrogate is constant, so the
    gradient is the entropy bonus's alone (the policy gradient with a zero
    advantage)."""
    p, obs, act, ret = tiny(6, M=40)
    A = ret - ret.mean()
    blog = np.zeros((obs.shape[0], DIMS[3]))
    # A > 0: make mu(a) tiny (rho >> 1 + eps); A < 0: make mu(a) ~ 1 (rho << 1 - eps)
    for i in range(obs.shape[0]):
        blog[i, act[i]] = -40.0 if A[i] > 0 else 40.0
    g, _ = learner.ppo_grad(p, DIMS, obs, act, ret, blog, 0.05, 0.2)
    g_ent, _ = learner.pg_grad(p, DIMS, obs, act, np.zeros_like(ret), 0.05)
    np.testing.assert_allclose(g, g_ent, rtol=1e-12, atol=1e-15)


def test_ppo_gradient_autograd():
    torch = pytest.importorskip("torch")
    p, obs, act, ret, blog = ppo_case(7, M=64)
    beta, eps = 0.01, 0.2
    g, _ = learner.ppo_grad(p, DIMS, obs, act, ret, blog, beta, eps)
    i, h1, h2, a = DIMS
    t = torch.tensor(p, dtype=torch.float64, requires_grad=True)
    o = 0
    W1 = t[o:o + h1 * i].view(h1, i); o += h1 * i
    b1 = t[o:o + h1]; o += h1
    W2 = t[o:o + h2 * h1].view(h2, h1); o += h2 * h1
    b2 = t[o:o + h2]; o += h2
    W3 = t[o:o + a * h2].view(a, h2); o += a * h2
    b3 = t[o:o + a]
    x = torch.tensor(obs)
    lp = torch.log_softmax(torch.relu(torch.relu(x @ W1.T + b1) @ W2.T + b2) @ W3.T + b3, dim=1)
    ent = -(lp.exp() * lp).sum(1)
    at = torch.tensor(act)
    lmu = torch.log_softmax(torch.tensor(blog), dim=1)[torch.arange(len(act)), at]
    rho = torch.exp(lp[torch.arange(len(act)), at] - lmu)
    A = torch.tensor(ret - ret.mean())
    surr = torch.minimum(rho * A, torch.clamp(rho, 1 - eps, 1 + eps) * A)
    (-(surr + beta * ent).mean()).backward()
    np.testing.assert_allclose(g, t.grad.numpy(), rtol=1e-10, atol=1e-13)


def test_gather_logits_order():
    """gather_logits follows gather's sample order: slot, then episode, step, env."""
    E, T, n_envs, N, A = 2, 3, 4, 2, 5
    lg = np.arange(E * T * n_envs * N * A, dtype=np.float64).reshape(E, T, n_envs, N, A)
    pairs = np.array([[0, 1], [1, 0]], np.int32)           # 2 combinations of 2 envs each
    out = learner.gather_logits({"logits": lg}, pairs, n_envs, N, 1)
    exp = np.concatenate([lg[:, :, 0:2, 1, :].reshape(-1, A), lg[:, :, 2:4, 0, :].reshape(-1, A)])
    np.testing.assert_array_equal(out, exp)
