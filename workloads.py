"""Seeded synthetic workloads for the rollout / payoff-evaluation path.

This module only draws inputs: populations (tabular behaviour policies and MLP
weights), policy combinations, and seeds. It holds none of the method's
arithmetic (no environment step, no policy forward, no sampling); both the CUDA
path and the CPU oracle consume exactly the arrays produced here.

The five workloads follow the paper's evaluation set-up (population of policies
per agent, policy combinations formed by picking one policy per agent, Sec. 3.1
"Defining the Task Graph"; Monte-Carlo simulations per combination, Sec. 4.2
Leduc PSRO) with the shapes listed below. The paper's own environments (MA-Atari,
SMAC, the MPE binaries) are not available, so these synthetic inputs stand in.

Parameter layout of one MLP policy (fp32, row-major, all layers back to back):
    W1[h1][in], b1[h1], W2[h2][h1], b2[h2], W3[out][h2], b3[out]
Weights ~ N(0, 1/fan_in); biases are 0 in the named workloads and
N(0, 0.1^2) when ``with_bias=True`` (used by tests so a dropped bias is caught).
Tabular Kuhn policies hold P(bet) for 6 infosets, ~ Uniform(0, 1) fp32.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

SEED_BASE = 2106075510

ENV_KUHN, ENV_LEDUC, ENV_SPREAD, ENV_ADVERSARY = 1, 2, 3, 4
ENV_SPEAKER_LISTENER, ENV_PUSH, ENV_TAG, ENV_REFERENCE = 5, 6, 7, 8
POL_TABULAR, POL_MLP = 1, 2
F32, BF16 = 0, 1


@dataclass
class Policy:
    kind: int            # POL_TABULAR or POL_MLP
    dtype: int           # F32 or BF16 (weights; accumulation is fp32 on the GPU)
    seat: int            # owning seat for poker populations, -1 for a shared pool
    dims: tuple          # (in, h1, h2, out) for MLP; (n_infosets, 0, 0, 1) tabular
    params: np.ndarray   # flat float32


@dataclass
class Workload:
    name: str
    env_kind: int
    n_agents: int
    n_landmarks: int
    obs_dim: int
    n_actions: int
    episode_len: int
    n_envs: int
    policies: list = field(default_factory=list)
    pair_ids: np.ndarray | None = None   # int32 [n_pairs][n_agents] (indices into policies)
    n_episodes: int = 1
    seed: int = 0
    rows: int = 0        # poker: seat-0 population size
    cols: int = 0        # poker: seat-1 population size

    @property
    def n_pairs(self) -> int:
        return 0 if self.pair_ids is None else int(self.pair_ids.shape[0])


def mlp_param_count(dims) -> int:
    i, h1, h2, o = dims
    return h1 * i + h1 + h2 * h1 + h2 + o * h2 + o


def random_mlp(rng: np.random.Generator, dims, with_bias: bool = False) -> np.ndarray:
    """Draw one MLP parameter vector in the layout of the module docstring."""
    i, h1, h2, o = dims
    parts = []
    for fan_in, fan_out in ((i, h1), (h1, h2), (h2, o)):
        w = rng.standard_normal((fan_out, fan_in), dtype=np.float32)
        w *= np.float32(1.0 / np.sqrt(fan_in))
        if with_bias:
            b = (rng.standard_normal(fan_out, dtype=np.float32) * np.float32(0.1))
        else:
            b = np.zeros(fan_out, dtype=np.float32)
        parts += [w.reshape(-1), b]
    out = np.concatenate(parts).astype(np.float32)
    assert out.size == mlp_param_count(dims)
    return out


def cartesian_pairs(rows: int, cols: int, row_offset: int = 0, col_offset: int = 0) -> np.ndarray:
    """All (seat-0 policy, seat-1 policy) combinations, row-major."""
    r = np.repeat(np.arange(rows, dtype=np.int32), cols) + row_offset
    c = np.tile(np.arange(cols, dtype=np.int32), rows) + col_offset
    return np.stack([r, c], axis=1).astype(np.int32)


def kuhn(pop: int = 4, n_episodes: int = 10_000, seed: int = SEED_BASE + 1) -> Workload:
    """Kuhn poker, `pop` tabular policies per seat, all pop x pop pairs."""
    rng = np.random.default_rng(seed)
    w = Workload("kuhn_4x4_tabular", ENV_KUHN, 2, 0, 0, 2, 0, 0, n_episodes=n_episodes,
                 seed=seed, rows=pop, cols=pop)
    for seat in (0, 1):
        for _ in range(pop):
            p = rng.random(6, dtype=np.float32)
            w.policies.append(Policy(POL_TABULAR, F32, seat, (6, 0, 0, 1), p))
    w.pair_ids = cartesian_pairs(pop, pop, 0, pop)
    return w


def leduc(pop: int = 8, hidden: int = 128, dtype: int = F32, n_episodes: int = 65_536,
          seed: int = SEED_BASE + 2, with_bias: bool = False, name: str | None = None) -> Workload:
    """Leduc hold'em, `pop` MLP policies 17->hidden->hidden->3 per seat, all pairs."""
    rng = np.random.default_rng(seed)
    dims = (17, hidden, hidden, 3)
    w = Workload(name or f"leduc_{pop}x{pop}_mlp{hidden}_{'bf16' if dtype == BF16 else 'f32'}",
                 ENV_LEDUC, 2, 0, 17, 3, 0, 0, n_episodes=n_episodes, seed=seed,
                 rows=pop, cols=pop)
    for seat in (0, 1):
        for _ in range(pop):
            w.policies.append(Policy(POL_MLP, dtype, seat, dims, random_mlp(rng, dims, with_bias)))
    w.pair_ids = cartesian_pairs(pop, pop, 0, pop)
    return w


def spread(n_agents: int = 3, n_envs: int = 4096, pop: int = 16, hidden: int = 64,
           obs_dim: int | None = None, dtype: int = F32, n_episodes: int = 1,
           episode_len: int = 25, envs_per_pair: int = 128, seed: int = SEED_BASE + 3,
           with_bias: bool = False, name: str | None = None) -> Workload:
    """Cooperative particle spread: N agents, N landmarks, shared population.

    Agents are assigned to policies by the seed, one policy per (block of
    `envs_per_pair` envs, agent slot): pair_ids[n_envs // envs_per_pair][N].
    """
    if obs_dim is None:
        obs_dim = 18 if n_agents == 3 else 4 + 2 * n_agents + 2 * (n_agents - 1)
    rng = np.random.default_rng(seed)
    dims = (obs_dim, hidden, hidden, 5)
    w = Workload(name or f"spread_n{n_agents}_{n_envs}env_mlp{hidden}_{'bf16' if dtype == BF16 else 'f32'}",
                 ENV_SPREAD, n_agents, n_agents, obs_dim, 5, episode_len, n_envs,
                 n_episodes=n_episodes, seed=seed)
    for _ in range(pop):
        w.policies.append(Policy(POL_MLP, dtype, -1, dims, random_mlp(rng, dims, with_bias)))
    n_pairs = max(1, n_envs // envs_per_pair)
    w.pair_ids = rng.integers(0, pop, size=(n_pairs, n_agents)).astype(np.int32)
    return w


def adversary(n_envs: int = 4096, pop: int = 16, hidden: int = 64, n_episodes: int = 1,
              episode_len: int = 25, envs_per_pair: int = 128, seed: int = SEED_BASE + 6,
              with_bias: bool = False, name: str | None = None) -> Workload:
    """Simple adversary (App. B.1): agent 0 the adversary, agents 1, 2 good,
    two landmarks; MLP 14-hidden-hidden-5 fp32 policies from one shared pool,
    assigned by the seed per (block of envs_per_pair envs, agent slot)."""
    rng = np.random.default_rng(seed)
    dims = (14, hidden, hidden, 5)
    w = Workload(name or f"adversary_{n_envs}env_mlp{hidden}_f32", ENV_ADVERSARY, 3, 2, 14, 5,
                 episode_len, n_envs, n_episodes=n_episodes, seed=seed)
    for _ in range(pop):
        w.policies.append(Policy(POL_MLP, F32, -1, dims, random_mlp(rng, dims, with_bias)))
    n_pairs = max(1, n_envs // envs_per_pair)
    w.pair_ids = rng.integers(0, pop, size=(n_pairs, 3)).astype(np.int32)
    return w


def speaker_listener(n_envs: int = 4096, pop: int = 16, hidden: int = 64, n_episodes: int = 1,
                     episode_len: int = 25, envs_per_pair: int = 128, seed: int = SEED_BASE + 7,
                     with_bias: bool = False, name: str | None = None) -> Workload:
    """Simple speaker listener (App. B.1): agent 0 the speaker, agent 1 the
    listener, three landmarks; MLP 11-hidden-hidden-5 fp32 policies from one
    shared pool, assigned by the seed per (block of envs_per_pair envs, agent
    slot)."""
    rng = np.random.default_rng(seed)
    dims = (11, hidden, hidden, 5)
    w = Workload(name or f"speaker_listener_{n_envs}env_mlp{hidden}_f32", ENV_SPEAKER_LISTENER, 2, 3,
                 11, 5, episode_len, n_envs, n_episodes=n_episodes, seed=seed)
    for _ in range(pop):
        w.policies.append(Policy(POL_MLP, F32, -1, dims, random_mlp(rng, dims, with_bias)))
    n_pairs = max(1, n_envs // envs_per_pair)
    w.pair_ids = rng.integers(0, pop, size=(n_pairs, 2)).astype(np.int32)
    return w


def push(n_envs: int = 4096, pop: int = 16, hidden: int = 64, n_episodes: int = 1,
         episode_len: int = 25, envs_per_pair: int = 128, seed: int = SEED_BASE + 8,
         with_bias: bool = False, name: str | None = None) -> Workload:
    """Simple push (App. B.1): agent 0 the adversary, agent 1 the good agent,
    one landmark, contact forces between the agents; MLP 8-hidden-hidden-5
    fp32 policies from one shared pool, assigned by the seed per (block of
    envs_per_pair envs, agent slot)."""
    rng = np.random.default_rng(seed)
    dims = (8, hidden, hidden, 5)
    w = Workload(name or f"push_{n_envs}env_mlp{hidden}_f32", ENV_PUSH, 2, 1, 8, 5,
                 episode_len, n_envs, n_episodes=n_episodes, seed=seed)
    for _ in range(pop):
        w.policies.append(Policy(POL_MLP, F32, -1, dims, random_mlp(rng, dims, with_bias)))
    n_pairs = max(1, n_envs // envs_per_pair)
    w.pair_ids = rng.integers(0, pop, size=(n_pairs, 2)).astype(np.int32)
    return w


def tag(n_envs: int = 4096, pop: int = 16, hidden: int = 64, n_episodes: int = 1,
        episode_len: int = 25, envs_per_pair: int = 128, seed: int = SEED_BASE + 9,
        with_bias: bool = False, name: str | None = None) -> Workload:
    """Simple tag (App. B.1): agents 0..2 the adversaries, agent 3 the good
    agent, two obstacles, contact forces among all of them; MLP
    16-hidden-hidden-5 fp32 policies from one shared pool, assigned by the seed
    per (block of envs_per_pair envs, agent slot)."""
    rng = np.random.default_rng(seed)
    dims = (16, hidden, hidden, 5)
    w = Workload(name or f"tag_{n_envs}env_mlp{hidden}_f32", ENV_TAG, 4, 2, 16, 5,
                 episode_len, n_envs, n_episodes=n_episodes, seed=seed)
    for _ in range(pop):
        w.policies.append(Policy(POL_MLP, F32, -1, dims, random_mlp(rng, dims, with_bias)))
    n_pairs = max(1, n_envs // envs_per_pair)
    w.pair_ids = rng.integers(0, pop, size=(n_pairs, 4)).astype(np.int32)
    return w


def reference(n_envs: int = 4096, pop: int = 16, hidden: int = 64, n_episodes: int = 1,
              episode_len: int = 25, envs_per_pair: int = 128, seed: int = SEED_BASE + 10,
              with_bias: bool = False, name: str | None = None) -> Workload:
    """Simple reference (App. B.1): 2 agents that speak and move, three
    landmarks; MLP 14-hidden-hidden-15 fp32 policies (15 = 5 moves x 3
    messages) from one shared pool, assigned by the seed per (block of
    envs_per_pair envs, agent slot)."""
    rng = np.random.default_rng(seed)
    dims = (14, hidden, hidden, 15)
    w = Workload(name or f"reference_{n_envs}env_mlp{hidden}_f32", ENV_REFERENCE, 2, 3, 14, 15,
                 episode_len, n_envs, n_episodes=n_episodes, seed=seed)
    for _ in range(pop):
        w.policies.append(Policy(POL_MLP, F32, -1, dims, random_mlp(rng, dims, with_bias)))
    n_pairs = max(1, n_envs // envs_per_pair)
    w.pair_ids = rng.integers(0, pop, size=(n_pairs, 2)).astype(np.int32)
    return w


def config(k: int, **over) -> Workload:
    """The five named workloads, 1-indexed:

    1 Kuhn 4x4 tabular x 10,000 episodes per pair
    2 Leduc 8x8 MLP 17-128-128-3 fp32 x 65,536 episodes per pair
    3 spread N=3, 4,096 envs, population 16, MLP 18-64-64-5 fp32
    4 spread N=8, 65,536 envs, population 32, MLP 34-256-256-5 bf16
    5 Leduc 64x64 MLP 17-256-256-3 bf16 x 16,384 episodes per pair
    """
    if k == 1:
        return kuhn(**over)
    if k == 2:
        return leduc(**over)
    if k == 3:
        return spread(**{"n_agents": 3, "n_envs": 4096, "pop": 16, "hidden": 64, **over})
    if k == 4:
        return spread(**{"n_agents": 8, "n_envs": 65_536, "pop": 32, "hidden": 256,
                         "dtype": BF16, "seed": SEED_BASE + 4, **over})
    if k == 5:
        return leduc(**{"pop": 64, "hidden": 256, "dtype": BF16, "n_episodes": 16_384,
                        "seed": SEED_BASE + 5, **over})
    raise ValueError(f"no workload {k}")
