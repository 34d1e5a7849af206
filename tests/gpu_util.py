"""Helpers shared by the GPU parity tests (no method arithmetic here)."""
import numpy as np
import pytest

import workloads


def need_gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return torch


def context():
    torch = need_gpu()
    import __graft_entry__
    __graft_entry__.build()
    from paper_2106_07551_gb300 import Context
    return Context(0, torch.cuda.current_stream(0))


def spec_of(w: workloads.Workload, flags: int = 0, n_envs: int | None = None, local_ratio=None):
    from paper_2106_07551_gb300 import make_spec
    return make_spec(w.env_kind, w.n_agents, w.obs_dim, w.n_actions, w.n_landmarks,
                     w.episode_len, w.n_envs if n_envs is None else n_envs, flags, local_ratio)


def load_population(ctx, w: workloads.Workload):
    from paper_2106_07551_gb300 import policy_desc
    descs = [policy_desc(p.kind, p.dtype, p.seat, p.dims, p.params) for p in w.policies]
    ids = ctx.pop_load(spec_of(w), descs)
    assert list(ids) == list(range(len(w.policies)))
    return ids


def logits_close(gpu, ref, rtol):
    """|g - o| <= rtol * max(|o|, rms(o over the row)) for every entry."""
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    rms = np.sqrt(np.mean(ref ** 2, axis=-1, keepdims=True))
    scale = np.maximum(np.abs(ref), rms)
    bad = np.abs(gpu - ref) > rtol * scale + 1e-30
    return int(bad.sum()), float((np.abs(gpu - ref) / np.maximum(scale, 1e-30)).max(initial=0.0))


def four_se_rule(mean, se, exact):
    """At most 3 entries beyond 4 standard errors and none beyond 5."""
    z = np.abs(np.asarray(mean) - np.asarray(exact)) / np.maximum(np.asarray(se), 1e-12)
    return int((z > 4).sum()), float(z.max(initial=0.0))
