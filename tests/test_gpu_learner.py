"""GPU parity for the learner-side update (Sec. 3.3 independent learning; App.
C.2 training workflow): the policy-gradient step of one policy on a GPU
rollout's samples, Adam, and the population update that closes the loop.

The oracle (oracle/learner.py, fp64) gathers the same samples from the
trajectory the GPU wrote and computes the gradient; the GPU's fp32 gradient
must match per parameter block within 1e-4 of the block's largest magnitude
(fp32 forward and fp32 per-CTA sums of a few thousand terms, summed across
CTAs in fp64: relative errors of order 1e-6), M exactly, the baseline and
mean entropy within 1e-5 relative, the loss (a mean of cancelling terms)
within 1e-5 of the terms' scale. Adam matches the fp64 recursion within
1e-6 relative. After pop_update, the next rollout replays bit for bit against
the oracle's rollout of the updated parameters."""
import numpy as np
import pytest

import oracle
import workloads
from oracle import learner
from gpu_util import context, load_population, logits_close, need_gpu, spec_of

pytestmark = pytest.mark.gpu

from paper_2106_07551_gb300 import MALIB_DUMP_LOGITS, MalibError, alloc_traj


def rollout(ctx, w, n_eps, seed, flags=0):
    spec = spec_of(w, flags)
    traj = alloc_traj(spec, n_eps, logits=bool(flags & MALIB_DUMP_LOGITS))
    ctx.rollout(spec, w.pair_ids, n_eps, seed, traj)
    ctx.sync()
    return spec, traj


def blocks(dims):
    i, h1, h2, a = dims
    sizes = [h1 * i, h1, h2 * h1, h2, a * h2, a]
    return np.cumsum([0] + sizes)


def check_grad(g, o, dims):
    cut = blocks(dims)
    for lo, hi in zip(cut[:-1], cut[1:]):
        scale = np.abs(o[lo:hi]).max()
        np.testing.assert_allclose(g[lo:hi], o[lo:hi], rtol=0, atol=1e-4 * scale + 1e-12)


def learn(ctx, w, spec, traj, n_eps, pid, gamma, beta, device_out=False):
    torch = need_gpu()
    P = int(blocks(w.policies[0].dims)[-1])
    if device_out:
        g = torch.zeros(P, dtype=torch.float32, device="cuda")
        st = torch.zeros(4, dtype=torch.float64, device="cuda")
        ctx.learn_pg(spec, w.pair_ids, n_eps, traj, pid, gamma, beta, g, st)
        ctx.sync()
        return g.cpu().numpy(), st.cpu().numpy()
    g = np.zeros(P, np.float32)
    st = np.zeros(4, np.float64)
    ctx.learn_pg(spec, w.pair_ids, n_eps, traj, pid, gamma, beta, g, st)
    return g, st


def host(traj):
    return {k: v.cpu().numpy() for k, v in traj.items()}


def oracle_grad(w, tr, pid, gamma, beta):
    obs, act, ret = learner.gather(tr, w.pair_ids, w.n_envs, w.n_agents, w.obs_dim, pid, gamma)
    return learner.pg_grad(w.policies[pid].params, w.policies[pid].dims, obs, act, ret, beta)


@pytest.mark.parametrize("make,kw", [(workloads.spread, dict(n_agents=3, n_envs=1024, pop=6)),
                                     (workloads.tag, dict(n_envs=512, pop=5)),
                                     (workloads.push, dict(n_envs=384, pop=4, envs_per_pair=64))])
def test_policy_gradient_parity(make, kw):
    need_gpu()
    w = make(with_bias=True, seed=77, **kw)
    ctx = context()
    load_population(ctx, w)
    spec, traj = rollout(ctx, w, 2, 99)
    tr = host(traj)
    for pid, gamma, beta, dev in ((0, 0.95, 0.001, False), (1, 0.0, 0.0, True), (2, 1.0, 0.1, False)):
        g, st = learn(ctx, w, spec, traj, 2, pid, gamma, beta, dev)
        o, (M, b, loss, ent) = oracle_grad(w, tr, pid, gamma, beta)
        assert st[0] == M and M > 0
        np.testing.assert_allclose([st[1], st[3]], [b, ent], rtol=1e-5, atol=1e-7)
        # the loss is a mean of terms of order |G - b| |log pi| that cancel: an
        # absolute bound relative to those terms, not to the (small) mean
        assert abs(st[2] - loss) <= 1e-5 * (1.0 + np.abs(tr["reward"]).max() * w.episode_len)
        check_grad(g, o, w.policies[pid].dims)
        # deterministic
        g2, st2 = learn(ctx, w, spec, traj, 2, pid, gamma, beta, dev)
        assert np.array_equal(g, g2) and np.array_equal(st, st2)
    ctx.close()


def test_policy_gradient_batch():
    """Every policy of a population in one call (including policies without
    samples) against the oracle, and against the single-policy entry point."""
    torch = need_gpu()
    w = workloads.spread(n_agents=3, n_envs=1024, pop=9, with_bias=True, seed=88)
    w.pair_ids[w.pair_ids == 8] = 7                      # policy 8 never acts
    ctx = context()
    load_population(ctx, w)
    spec, traj = rollout(ctx, w, 2, 5)
    tr = host(traj)
    P = int(blocks(w.policies[0].dims)[-1])
    ids = np.array([3, 8, 0, 1, 2, 4, 5, 6, 7], np.int32)
    g = torch.zeros((len(ids), P), device="cuda")
    st = torch.zeros((len(ids), 4), dtype=torch.float64, device="cuda")
    ctx.learn_pg_batch(spec, w.pair_ids, 2, traj, ids, 0.9, 0.01, g, st)
    ctx.sync()
    g, st = g.cpu().numpy(), st.cpu().numpy()
    for row, pid in enumerate(ids):
        o, (M, b, loss, ent) = oracle_grad(w, tr, int(pid), 0.9, 0.01)
        assert st[row, 0] == M
        if M == 0:
            assert np.all(g[row] == 0) and np.all(st[row] == 0)
            continue
        np.testing.assert_allclose([st[row, 1], st[row, 3]], [b, ent], rtol=1e-5, atol=1e-7)
        check_grad(g[row], o, w.policies[pid].dims)
        g1, st1 = learn(ctx, w, spec, traj, 2, int(pid), 0.9, 0.01)
        check_grad(g[row], g1.astype(np.float64), w.policies[pid].dims)
    with pytest.raises(MalibError, match="EINVAL"):
        ctx.learn_pg_batch(spec, w.pair_ids, 2, traj, np.array([1, 2, 1], np.int32), 0.9, 0.0,
                           np.zeros((3, P), np.float32))
    ctx.close()


def test_policy_without_samples():
    need_gpu()
    w = workloads.spread(n_agents=3, n_envs=256, pop=6, seed=5)
    w.pair_ids[:] = np.array([0, 1, 2], np.int32)              # policies 3..5 never act
    ctx = context()
    load_population(ctx, w)
    spec, traj = rollout(ctx, w, 1, 3)
    g, st = learn(ctx, w, spec, traj, 1, 4, 0.9, 0.01)
    assert np.all(g == 0) and np.all(st == 0)
    ctx.close()


def test_adam_parity():
    torch = need_gpu()
    rng = np.random.default_rng(8)
    n = 10_000
    p0 = rng.normal(size=n).astype(np.float32)
    ctx = context()
    p = torch.from_numpy(p0.copy()).cuda()
    m = torch.zeros(n, device="cuda")
    v = torch.zeros(n, device="cuda")
    rp, rm, rv = p0.astype(np.float64), np.zeros(n), np.zeros(n)
    for step in range(1, 6):
        gr = rng.normal(size=n).astype(np.float32)
        ctx.adam_step(p, torch.from_numpy(gr).cuda(), m, v, step, 1e-3)
        rp, rm, rv = learner.adam(rp, gr, rm, rv, step, 1e-3)
        ctx.sync()
        np.testing.assert_allclose(p.cpu().numpy(), rp, rtol=1e-6, atol=1e-7)
        # m is a running sum of terms of order 0.1 |g| that can cancel: absolute
        np.testing.assert_allclose(m.cpu().numpy(), rm, rtol=1e-5, atol=1e-7)
    ctx.close()


def test_training_loop_closes():
    """rollout -> policy gradient -> Adam -> pop_update -> rollout: the second
    rollout replays bit for bit against the oracle with the updated policy."""
    torch = need_gpu()
    w = workloads.spread(n_agents=3, n_envs=512, pop=4, with_bias=True, seed=21)
    ctx = context()
    load_population(ctx, w)
    spec, traj = rollout(ctx, w, 1, 11)
    pid = int(w.pair_ids[0, 0])
    P = int(blocks(w.policies[pid].dims)[-1])
    g = torch.zeros(P, device="cuda")
    ctx.learn_pg(spec, w.pair_ids, 1, traj, pid, 0.95, 0.001, g)
    params = torch.from_numpy(w.policies[pid].params.astype(np.float32)).cuda()
    m = torch.zeros(P, device="cuda")
    v = torch.zeros(P, device="cuda")
    ctx.adam_step(params, g, m, v, 1, 1e-2)
    ctx.pop_update(pid, params)
    new = params.cpu().numpy()
    assert not np.array_equal(new, w.policies[pid].params)
    w.policies[pid].params = new
    spec, traj2 = rollout(ctx, w, 1, 12, MALIB_DUMP_LOGITS)
    tr = host(traj2)
    ref = oracle.spread_rollout([p.params for p in w.policies], w.policies[0].dims, 3, 3, w.episode_len,
                                w.n_envs, w.pair_ids, 1, 12, ext_logits=tr["logits"])
    np.testing.assert_array_equal(tr["obs"][..., :w.obs_dim], ref["obs"])
    np.testing.assert_array_equal(tr["action"].astype(np.int8), ref["action"])
    n_bad, worst = logits_close(tr["logits"], ref["logits"], 1e-5)
    assert n_bad == 0, (n_bad, worst)
    # a host buffer works as well, and restores the old parameters
    old = np.asarray(workloads.spread(n_agents=3, n_envs=512, pop=4, with_bias=True, seed=21)
                     .policies[pid].params, np.float32)
    ctx.pop_update(pid, old)
    ctx.close()


def test_learner_refusals():
    torch = need_gpu()
    w = workloads.spread(n_agents=3, n_envs=256, pop=3, seed=2)
    ctx = context()
    load_population(ctx, w)
    spec, traj = rollout(ctx, w, 1, 1)
    g = np.zeros(int(blocks(w.policies[0].dims)[-1]), np.float32)
    for pid, gamma, beta in ((3, 0.9, 0.0), (-1, 0.9, 0.0), (0, 1.5, 0.0), (0, 0.9, -1.0)):
        with pytest.raises(MalibError, match="EINVAL"):
            ctx.learn_pg(spec, w.pair_ids, 1, traj, pid, gamma, beta, g)
    with pytest.raises(MalibError, match="EINVAL"):
        ctx.pop_update(0, np.zeros(5, np.float32))
    with pytest.raises(MalibError, match="EINVAL"):
        ctx.adam_step(torch.zeros(4, device="cuda"), np.zeros(4, np.float32), torch.zeros(4, device="cuda"),
                      torch.zeros(4, device="cuda"), 1, 1e-3)
    ctx.close()
    # a bf16 (tensor-core) population has no learner kernel
    wb = workloads.spread(n_agents=8, n_envs=128, pop=2, hidden=256, dtype=workloads.BF16, seed=3)
    ctx = context()
    load_population(ctx, wb)
    spec, traj = rollout(ctx, wb, 1, 1)
    with pytest.raises(MalibError, match="EUNSUPPORTED"):
        ctx.learn_pg(spec, wb.pair_ids, 1, traj, 0, 0.9, 0.0, np.zeros(100, np.float32))
    ctx.close()


# ---- PPO: the clipped surrogate against the behavior logits the rollout recorded

def perturbed(w, pids, scale, seed):
    """New parameters for the policies pids (the behavior policies stay in w)."""
    rng = np.random.default_rng(seed)
    return {pid: (w.policies[pid].params + rng.normal(0, scale, w.policies[pid].params.shape)).astype(np.float32)
            for pid in pids}


def ppo_oracle(w, tr, pid, params, gamma, beta, eps):
    obs, act, ret = learner.gather(tr, w.pair_ids, w.n_envs, w.n_agents, w.obs_dim, pid, gamma)
    blog = learner.gather_logits(tr, w.pair_ids, w.n_envs, w.n_agents, pid)
    dims = w.policies[pid].dims
    return (learner.ppo_grad(params, dims, obs, act, ret, blog, beta, eps),
            learner.ppo_margin(params, dims, obs, act, blog, eps), (obs, act, ret, blog))


@pytest.mark.parametrize("make,kw", [(workloads.spread, dict(n_agents=3, n_envs=256, pop=6)),
                                     (workloads.tag, dict(n_envs=256, pop=5))])
def test_ppo_parity(make, kw):
    """Policies moved away from the ones that acted: the GPU's clipped-surrogate
    gradient against the oracle's. A sample whose ratio lies within the fp32
    error (a few 1e-6) of a clip edge may take the other branch on the GPU, so
    the clip range is chosen among nearby values as one that leaves every
    ratio at least 2e-5 from both edges; samples are clipped on both sides."""
    torch = need_gpu()
    w = make(with_bias=True, seed=71, **kw)
    ctx = context()
    load_population(ctx, w)
    spec, traj = rollout(ctx, w, 2, 41, MALIB_DUMP_LOGITS)
    tr = host(traj)
    ids, counts = np.unique(w.pair_ids, return_counts=True)
    pids = [int(p) for p in ids[np.argsort(-counts, kind="stable")][:2]]   # the two busiest policies
    new = perturbed(w, pids, 0.05, 5)
    gamma, beta = 0.95, 0.01
    for eps in np.linspace(0.15, 0.25, 21):
        eps = float(eps)
        res = {pid: ppo_oracle(w, tr, pid, new[pid], gamma, beta, eps) for pid in pids}
        if min(r[1] for r in res.values()) > 2e-5:
            break
    else:
        pytest.fail("no clip range with a clear margin")
    # both branches are exercised
    obs, act, ret, blog = res[pids[0]][2]
    dims = w.policies[0].dims
    W1, b1, W2, b2, W3, b3 = learner.unpack(new[pids[0]], dims)
    z = np.maximum(np.maximum(obs @ W1.T + b1, 0) @ W2.T + b2, 0) @ W3.T + b3
    idx = np.arange(obs.shape[0])
    rho = np.exp(learner.log_softmax(z)[idx, act] - learner.log_softmax(blog)[idx, act])
    assert (rho > 1 + eps).any() and (rho < 1 - eps).any() and (np.abs(rho - 1) < eps).any()
    for pid in pids:
        ctx.pop_update(pid, new[pid])
    P = int(blocks(dims)[-1])
    g = torch.zeros((len(pids), P), device="cuda")
    st = torch.zeros((len(pids), 4), dtype=torch.float64, device="cuda")
    ctx.learn_ppo_batch(spec, w.pair_ids, 2, traj, pids, gamma, beta, eps, g, st)
    ctx.sync()
    g, st = g.cpu().numpy(), st.cpu().numpy()
    for row, pid in enumerate(pids):
        o, (M, b, loss, ent) = res[pid][0]
        assert st[row, 0] == M and M > 0
        np.testing.assert_allclose([st[row, 1], st[row, 3]], [b, ent], rtol=1e-5, atol=1e-7)
        assert abs(st[row, 2] - loss) <= 1e-5 * (1.0 + np.abs(tr["reward"]).max() * w.episode_len)
        check_grad(g[row], o, dims)
    # deterministic
    g2 = torch.zeros((len(pids), P), device="cuda")
    ctx.learn_ppo_batch(spec, w.pair_ids, 2, traj, pids, gamma, beta, eps, g2)
    ctx.sync()
    assert np.array_equal(g, g2.cpu().numpy())
    ctx.close()


def test_ppo_on_policy_is_the_policy_gradient():
    """The policies that acted, unchanged: every ratio is 1 up to rounding, and
    the PPO gradient is the policy gradient's."""
    torch = need_gpu()
    w = workloads.spread(n_agents=3, n_envs=1024, pop=6, with_bias=True, seed=72)
    ctx = context()
    load_population(ctx, w)
    spec, traj = rollout(ctx, w, 2, 43, MALIB_DUMP_LOGITS)
    P = int(blocks(w.policies[0].dims)[-1])
    ids = [0, 3, 5]
    g_ppo = torch.zeros((3, P), device="cuda")
    g_pg = torch.zeros((3, P), device="cuda")
    ctx.learn_ppo_batch(spec, w.pair_ids, 2, traj, ids, 0.9, 0.001, 0.2, g_ppo)
    ctx.learn_pg_batch(spec, w.pair_ids, 2, traj, ids, 0.9, 0.001, g_pg)
    ctx.sync()
    for row, pid in enumerate(ids):
        check_grad(g_ppo[row].cpu().numpy(), g_pg[row].cpu().numpy().astype(np.float64), w.policies[pid].dims)
    ctx.close()


def test_ppo_refusals():
    torch = need_gpu()
    w = workloads.spread(n_agents=3, n_envs=256, pop=3, seed=73)
    ctx = context()
    load_population(ctx, w)
    spec, traj = rollout(ctx, w, 1, 3)                       # no logits recorded
    P = int(blocks(w.policies[0].dims)[-1])
    g = torch.zeros((1, P), device="cuda")
    with pytest.raises(MalibError, match="EINVAL"):
        ctx.learn_ppo_batch(spec, w.pair_ids, 1, traj, [0], 0.9, 0.0, 0.2, g)
    spec, traj = rollout(ctx, w, 1, 3, MALIB_DUMP_LOGITS)
    for eps in (0.0, -0.1, 1.0, float("nan")):
        with pytest.raises(MalibError, match="EINVAL"):
            ctx.learn_ppo_batch(spec, w.pair_ids, 1, traj, [0], 0.9, 0.0, eps, g)
    ctx.learn_ppo_batch(spec, w.pair_ids, 1, traj, [0], 0.9, 0.0, 0.2, g)
    ctx.sync()
    assert torch.isfinite(g).all()
    ctx.close()


def test_ppo_batch_with_an_idle_policy_and_push():
    """PPO over every policy of a push population, one of which never acts (its
    row and statistics stay zero), after one Adam-free perturbation of the
    others; each row against the oracle."""
    torch = need_gpu()
    w = workloads.push(n_envs=384, pop=4, envs_per_pair=64, with_bias=True, seed=74)
    w.pair_ids[w.pair_ids == 3] = 2                      # policy 3 never acts
    ctx = context()
    load_population(ctx, w)
    spec, traj = rollout(ctx, w, 2, 47, MALIB_DUMP_LOGITS)
    tr = host(traj)
    pids = [0, 1, 2]
    new = perturbed(w, pids, 0.03, 9)
    for eps in np.linspace(0.15, 0.25, 21):
        eps = float(eps)
        res = {pid: ppo_oracle(w, tr, pid, new[pid], 0.9, 0.005, eps) for pid in pids}
        if min(r[1] for r in res.values()) > 2e-5:
            break
    else:
        pytest.fail("no clip range with a clear margin")
    for pid in pids:
        ctx.pop_update(pid, new[pid])
    dims = w.policies[0].dims
    P = int(blocks(dims)[-1])
    ids = [3, 0, 1, 2]
    g = torch.zeros((4, P), device="cuda")
    st = torch.zeros((4, 4), dtype=torch.float64, device="cuda")
    ctx.learn_ppo_batch(spec, w.pair_ids, 2, traj, ids, 0.9, 0.005, eps, g, st)
    ctx.sync()
    g, st = g.cpu().numpy(), st.cpu().numpy()
    assert np.all(g[0] == 0) and np.all(st[0] == 0)
    for row, pid in enumerate(ids[1:], start=1):
        o, (M, b, loss, ent) = res[pid][0]
        assert st[row, 0] == M and M > 0
        np.testing.assert_allclose([st[row, 1], st[row, 3]], [b, ent], rtol=1e-5, atol=1e-7)
        check_grad(g[row], o, dims)
    ctx.close()
