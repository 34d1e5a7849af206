"""The library's two quick-start uses, written as a user would: a Leduc payoff
table between 8 + 8 fp32 MLP policies, and a particle-spread rollout of 3
agents over 4,096 environments in 32 blocks of 128 with their own policy
combinations. Checks the shapes and invariants of what comes back."""
import numpy as np
import pytest

from gpu_util import need_gpu

pytestmark = pytest.mark.gpu


def _mlp(rng, dims):
    """Row-major W[out][in] then b[out], per layer, fp32."""
    parts = []
    for fi, fo in zip(dims[:-1], dims[1:]):
        parts += [rng.normal(0, fi ** -0.5, (fo, fi)).astype(np.float32).ravel(),
                  np.zeros(fo, np.float32)]
    return np.concatenate(parts)


def test_quick_start_payoff_table_and_rollout():
    need_gpu()
    import __graft_entry__
    __graft_entry__.build()
    from paper_2106_07551_gb300 import (MALIB_ENV_LEDUC, MALIB_ENV_SPREAD, MALIB_F32,
                                        MALIB_POL_MLP, Context, alloc_traj, make_spec,
                                        policy_desc)
    rng = np.random.default_rng(0)
    dims = (17, 128, 128, 3)
    params = [_mlp(rng, dims) for _ in range(16)]
    seats = [0] * 8 + [1] * 8
    spec = make_spec(MALIB_ENV_LEDUC, 2, 17, 3)
    with Context(0) as ctx:
        ids = ctx.pop_load(spec, [policy_desc(MALIB_POL_MLP, MALIB_F32, s, dims, p)
                                  for s, p in zip(seats, params)])
        pairs = np.array([[i, j] for i in ids[:8] for j in ids[8:]], np.int32)
        table = ctx.eval_payoff(pairs, 65536, 1)
    assert table.shape == (64, 4)
    assert np.all(np.isfinite(table)) and np.all(table[:, 1] > 0)
    assert np.all(np.abs(table[:, 0]) <= 13)

    dims = (18, 64, 64, 5)
    params = [_mlp(rng, dims) for _ in range(16)]
    spec = make_spec(MALIB_ENV_SPREAD, 3, 18, 5, n_landmarks=3, episode_len=25, n_envs=4096)
    with Context(0) as ctx:
        ids = ctx.pop_load(spec, [policy_desc(MALIB_POL_MLP, MALIB_F32, -1, dims, p)
                                  for p in params])
        combos = rng.integers(0, 16, (32, 3)).astype(np.int32)
        traj = alloc_traj(spec, 2)
        ctx.rollout(spec, combos, 2, 7, traj)
        ctx.sync()
    obs = traj["obs"].cpu().numpy()
    assert obs.shape == (2, 25, 4096, 3, 20)
    assert traj["action"].cpu().numpy().max() <= 4
    done = traj["done"].cpu().numpy()
    assert np.all(done[:, -1] == 1) and np.all(done[:, :-1] == 0)
    assert np.all(traj["reward"].cpu().numpy() <= 0)


def test_quick_start_learner_loop():
    """rollout -> policy gradient -> Adam -> population update, as a user would
    write it; the loss statistics are finite and the next rollout runs."""
    torch = need_gpu()
    import __graft_entry__
    __graft_entry__.build()
    from paper_2106_07551_gb300 import (MALIB_ENV_SPREAD, MALIB_F32, MALIB_POL_MLP, Context, alloc_traj,
                                        make_spec, policy_desc)
    rng = np.random.default_rng(0)
    dims = (18, 64, 64, 5)
    params = [_mlp(rng, dims) for _ in range(16)]
    spec = make_spec(MALIB_ENV_SPREAD, 3, 18, 5, n_landmarks=3, episode_len=25, n_envs=4096)
    with Context(0) as ctx:
        ids = ctx.pop_load(spec, [policy_desc(MALIB_POL_MLP, MALIB_F32, -1, dims, p) for p in params])
        combos = rng.integers(0, 16, (32, 3)).astype(np.int32)
        combos[0, 0] = 0                                  # policy 0 acts somewhere
        traj = alloc_traj(spec, 2)
        ctx.rollout(spec, combos, 2, 7, traj)
        P = params[0].size
        grad = torch.zeros(P, device="cuda")
        stats = torch.zeros(4, dtype=torch.float64, device="cuda")
        ctx.learn_pg(spec, combos, 2, traj, 0, 0.95, 0.001, grad, stats)
        # every policy at once, on the same weights and trajectory
        grads = torch.zeros((len(params), P), device="cuda")
        ctx.learn_pg_batch(spec, combos, 2, traj, list(range(len(params))), 0.95, 0.001, grads)
        w = torch.from_numpy(params[0]).cuda()
        m, v = torch.zeros_like(w), torch.zeros_like(w)
        ctx.adam_step(w, grad, m, v, 1, 1e-4)
        ctx.pop_update(int(ids[0]), w)
        ctx.rollout(spec, combos, 2, 8, traj)
        ctx.sync()
        # the batched call's row 0 is the single call's gradient up to the order of
        # its partial sums (the CTAs' shares of the tiles differ)
        assert (grads[0] - grad).abs().max() <= 1e-4 * grad.abs().max()
        st = stats.cpu().numpy()
        assert st[0] == (combos == 0).sum() * 128 * 2 * 25 and np.all(np.isfinite(st))
        assert torch.isfinite(grad).all() and grad.abs().max() > 0
        assert np.all(traj["done"][:, -1].cpu().numpy() == 1)
