"""CPU oracle of the learner-side update: one independent learner's
policy-gradient step on the samples a rollout wrote, and the Adam update.

TEST INFRASTRUCTURE ONLY: a plain, slow fp64 numpy restatement, used to check
the GPU path. Only the tests, the smoke check and the benchmark's CPU-baseline
leg may import it; it shares no code with the CUDA path.

What it follows:
 * Sec. 3.3 "Independent Learning": one learner per policy, trained only on its
   own agents' experience (the policy-gradient family of the paper's Table 2).
 * App. C.2, the training workflow: rollout episodes are sampled into a batch
   and the learner's optimize() runs Adam with lr 1e-4 and an entropy
   coefficient of 0.001 (its training_config).
 * Readings (stated, the paper gives no loss): the loss of policy p over its
   samples S_p (every (episode, step, environment, agent) whose combination
   gives that agent policy p) is
       L = -(1/M) sum_i [ (G_i - b) log pi(a_i | o_i) + beta H(pi(. | o_i)) ],
   M = |S_p|, G_i the discounted return-to-go of sample i within its episode
   (G_t = r_t + gamma G_{t+1}, G after the last step 0), b = the mean of G
   over S_p (a baseline), H the entropy of the softmax over all actions.
   Adam as in Kingma and Ba (2015), with bias correction.

The PPO variant (the paper's learners are PPO/A2C-style; it prints no loss):
Schulman et al. (2017)'s clipped surrogate with the same advantage A = G - b,
       L = -(1/M) sum_i [ min(rho_i A_i, clip(rho_i, 1 - eps, 1 + eps) A_i)
                          + beta H(pi(. | o_i)) ],
rho_i = pi(a_i | o_i) / mu(a_i | o_i), mu the behavior policy that acted in the
rollout, known from the logits the rollout recorded. At rho = 1 (the first
epoch on fresh samples) its gradient is the policy gradient's.

Parity status: the gradients are pinned by central finite differences of the
losses and by torch.autograd in fp64 (tests/test_oracle_learner.py); the PPO
gradient also by its two limits, the policy gradient at mu = pi and the
entropy term alone when every sample is clipped; Adam by its first-step closed
form and a hand-iterated scalar sequence.
"""
from __future__ import annotations

import numpy as np


def unpack(params: np.ndarray, dims):
    """W1 [h1][in], b1, W2 [h2][h1], b2, W3 [a][h2], b3 (fp64 views)."""
    i, h1, h2, a = dims
    p = np.asarray(params, np.float64)
    o = 0
    W1 = p[o:o + h1 * i].reshape(h1, i); o += h1 * i
    b1 = p[o:o + h1]; o += h1
    W2 = p[o:o + h2 * h1].reshape(h2, h1); o += h2 * h1
    b2 = p[o:o + h2]; o += h2
    W3 = p[o:o + a * h2].reshape(a, h2); o += a * h2
    b3 = p[o:o + a]; o += a
    assert o == p.size
    return W1, b1, W2, b2, W3, b3


def samples(pairs: np.ndarray, n_envs: int, n_agents: int, policy_id: int):
    """The (combination, agent) slots that act with policy_id, ascending."""
    pairs = np.asarray(pairs).reshape(-1, n_agents)
    return [(c, k) for c in range(pairs.shape[0]) for k in range(n_agents) if pairs[c, k] == policy_id]


def returns_to_go(reward: np.ndarray, gamma: float) -> np.ndarray:
    """reward [E][T][n_envs][N] -> G of the same shape: G_t = r_t + gamma G_{t+1}."""
    r = np.asarray(reward, np.float64)
    G = np.zeros_like(r)
    run = np.zeros(r.shape[:1] + r.shape[2:])
    for t in range(r.shape[1] - 1, -1, -1):
        run = r[:, t] + gamma * run
        G[:, t] = run
    return G


def gather(traj: dict, pairs, n_envs: int, n_agents: int, obs_dim: int, policy_id: int, gamma: float):
    """Observations [M][obs_dim], actions [M], returns [M] of policy_id's
    samples, in slot order (combination, agent), then episode, step, env."""
    slots = samples(pairs, n_envs, n_agents, policy_id)
    n_pairs = np.asarray(pairs).reshape(-1, n_agents).shape[0]
    epp = n_envs // n_pairs
    G = returns_to_go(traj["reward"], gamma)
    obs, act, ret = [], [], []
    for c, k in slots:
        envs = slice(c * epp, (c + 1) * epp)
        obs.append(np.asarray(traj["obs"], np.float64)[:, :, envs, k, :obs_dim].reshape(-1, obs_dim))
        act.append(np.asarray(traj["action"])[:, :, envs, k].reshape(-1).astype(np.int64))
        ret.append(G[:, :, envs, k].reshape(-1))
    if not slots:
        return np.zeros((0, obs_dim)), np.zeros(0, np.int64), np.zeros(0)
    return np.concatenate(obs), np.concatenate(act), np.concatenate(ret)


def gather_logits(traj: dict, pairs, n_envs: int, n_agents: int, policy_id: int):
    """The behavior logits [M][A] that the rollout recorded for policy_id's
    samples (traj["logits"] [E][T][n_envs][N][A]), in gather()'s order."""
    slots = samples(pairs, n_envs, n_agents, policy_id)
    n_pairs = np.asarray(pairs).reshape(-1, n_agents).shape[0]
    epp = n_envs // n_pairs
    lg = np.asarray(traj["logits"], np.float64)
    if not slots:
        return np.zeros((0, lg.shape[-1]))
    return np.concatenate([lg[:, :, c * epp:(c + 1) * epp, k, :].reshape(-1, lg.shape[-1]) for c, k in slots])


def log_softmax(z: np.ndarray) -> np.ndarray:
    """Row-wise log pi of logits z [M][A] (fp64, max-shifted)."""
    z = np.asarray(z, np.float64)
    zmax = z.max(axis=1, keepdims=True)
    return z - zmax - np.log(np.exp(z - zmax).sum(axis=1, keepdims=True))


def pg_loss(params, dims, obs, act, ret, beta: float):
    """The loss L above and (mean entropy, baseline)."""
    W1, b1, W2, b2, W3, b3 = unpack(params, dims)
    M = obs.shape[0]
    if M == 0:
        return 0.0, 0.0, 0.0
    h1 = np.maximum(obs @ W1.T + b1, 0.0)
    h2 = np.maximum(h1 @ W2.T + b2, 0.0)
    z = h2 @ W3.T + b3
    zmax = z.max(axis=1, keepdims=True)
    logp = z - zmax - np.log(np.exp(z - zmax).sum(axis=1, keepdims=True))
    pi = np.exp(logp)
    H = -(pi * logp).sum(axis=1)
    b = ret.mean()
    A = ret - b
    loss = -(A * logp[np.arange(M), act] + beta * H).sum() / M
    return loss, H.mean(), b


def pg_grad(params, dims, obs, act, ret, beta: float):
    """dL/dparams in the params layout (fp64), by the chain rule written out:
    dL/dz_j = (1/M) [ (G - b)(pi_j - [j = a]) + beta pi_j (log pi_j + H) ],
    then back through W3, the second ReLU (pre-activation > 0), W2, the first
    ReLU and W1. Also returns (M, baseline, loss, mean entropy)."""
    W1, b1, W2, b2, W3, b3 = unpack(params, dims)
    M = obs.shape[0]
    grad = np.zeros(np.asarray(params).size)
    if M == 0:
        return grad, (0, 0.0, 0.0, 0.0)
    pre1 = obs @ W1.T + b1
    h1 = np.maximum(pre1, 0.0)
    pre2 = h1 @ W2.T + b2
    h2 = np.maximum(pre2, 0.0)
    z = h2 @ W3.T + b3
    zmax = z.max(axis=1, keepdims=True)
    logp = z - zmax - np.log(np.exp(z - zmax).sum(axis=1, keepdims=True))
    pi = np.exp(logp)
    H = -(pi * logp).sum(axis=1)
    b = ret.mean()
    A = ret - b
    onehot = np.zeros_like(pi)
    onehot[np.arange(M), act] = 1.0
    dz = (A[:, None] * (pi - onehot) + beta * pi * (logp + H[:, None])) / M
    dW3 = dz.T @ h2
    db3 = dz.sum(0)
    d2 = (dz @ W3) * (pre2 > 0)
    dW2 = d2.T @ h1
    db2 = d2.sum(0)
    d1 = (d2 @ W2) * (pre1 > 0)
    dW1 = d1.T @ obs
    db1 = d1.sum(0)
    grad[:] = np.concatenate([dW1.ravel(), db1, dW2.ravel(), db2, dW3.ravel(), db3])
    loss = -(A * logp[np.arange(M), act] + beta * H).sum() / M
    return grad, (M, b, loss, H.mean())


def ppo_loss(params, dims, obs, act, ret, blogits, beta: float, eps: float):
    """The clipped-surrogate loss L of the PPO variant above (fp64)."""
    W1, b1, W2, b2, W3, b3 = unpack(params, dims)
    M = obs.shape[0]
    if M == 0:
        return 0.0
    h1 = np.maximum(obs @ W1.T + b1, 0.0)
    h2 = np.maximum(h1 @ W2.T + b2, 0.0)
    logp = log_softmax(h2 @ W3.T + b3)
    H = -(np.exp(logp) * logp).sum(axis=1)
    A = ret - ret.mean()
    idx = np.arange(M)
    rho = np.exp(logp[idx, act] - log_softmax(blogits)[idx, act])
    surr = np.minimum(rho * A, np.clip(rho, 1.0 - eps, 1.0 + eps) * A)
    return -(surr + beta * H).sum() / M


def ppo_grad(params, dims, obs, act, ret, blogits, beta: float, eps: float):
    """dL/dparams of the clipped surrogate (fp64), with the chain rule written
    out. The unclipped term is the minimum, and carries the gradient, when
    rho A <= clip(rho) A (ties go to it); the clipped one is constant in the
    parameters. So
      dL/dz_j = (1/M) [ active A rho (pi_j - [j = a]) + beta pi_j (log pi_j + H) ],
    then back through the layers as in pg_grad. Also returns (M, baseline,
    loss, mean entropy)."""
    W1, b1, W2, b2, W3, b3 = unpack(params, dims)
    M = obs.shape[0]
    grad = np.zeros(np.asarray(params).size)
    if M == 0:
        return grad, (0, 0.0, 0.0, 0.0)
    pre1 = obs @ W1.T + b1
    h1 = np.maximum(pre1, 0.0)
    pre2 = h1 @ W2.T + b2
    h2 = np.maximum(pre2, 0.0)
    logp = log_softmax(h2 @ W3.T + b3)
    pi = np.exp(logp)
    H = -(pi * logp).sum(axis=1)
    b = ret.mean()
    A = ret - b
    idx = np.arange(M)
    rho = np.exp(logp[idx, act] - log_softmax(blogits)[idx, act])
    clipped = np.clip(rho, 1.0 - eps, 1.0 + eps) * A
    active = rho * A <= clipped
    onehot = np.zeros_like(pi)
    onehot[idx, act] = 1.0
    dz = (np.where(active, A * rho, 0.0)[:, None] * (pi - onehot) + beta * pi * (logp + H[:, None])) / M
    dW3 = dz.T @ h2
    db3 = dz.sum(0)
    d2 = (dz @ W3) * (pre2 > 0)
    dW2 = d2.T @ h1
    db2 = d2.sum(0)
    d1 = (d2 @ W2) * (pre1 > 0)
    dW1 = d1.T @ obs
    db1 = d1.sum(0)
    grad[:] = np.concatenate([dW1.ravel(), db1, dW2.ravel(), db2, dW3.ravel(), db3])
    loss = -(np.minimum(rho * A, clipped) + beta * H).sum() / M
    return grad, (M, b, loss, H.mean())


def ppo_margin(params, dims, obs, act, blogits, eps: float) -> float:
    """The smallest distance of any sample's ratio to a clip edge 1 -/+ eps:
    where it is tiny, fp32 and fp64 may take that sample's branch differently."""
    W1, b1, W2, b2, W3, b3 = unpack(params, dims)
    if obs.shape[0] == 0:
        return np.inf
    h1 = np.maximum(obs @ W1.T + b1, 0.0)
    h2 = np.maximum(h1 @ W2.T + b2, 0.0)
    idx = np.arange(obs.shape[0])
    rho = np.exp(log_softmax(h2 @ W3.T + b3)[idx, act] - log_softmax(blogits)[idx, act])
    return float(np.minimum(np.abs(rho - (1.0 - eps)), np.abs(rho - (1.0 + eps))).min())


def adam(params, grad, m, v, step: int, lr: float, beta1: float = 0.9, beta2: float = 0.999,
         eps: float = 1e-8):
    """One Adam step (Kingma and Ba): m <- beta1 m + (1 - beta1) g,
    v <- beta2 v + (1 - beta2) g^2, p <- p - lr m_hat / (sqrt(v_hat) + eps),
    m_hat = m / (1 - beta1^step), v_hat = v / (1 - beta2^step); step >= 1."""
    g = np.asarray(grad, np.float64)
    m = beta1 * np.asarray(m, np.float64) + (1 - beta1) * g
    v = beta2 * np.asarray(v, np.float64) + (1 - beta2) * g * g
    mh = m / (1 - beta1 ** step)
    vh = v / (1 - beta2 ** step)
    p = np.asarray(params, np.float64) - lr * mh / (np.sqrt(vh) + eps)
    return p, m, v
