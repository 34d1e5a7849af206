"""The allocation-free payoff evaluation (malib_eval_payoff_noalloc).

It exists for callers that cannot allocate device memory while they evaluate:
a framework that has reserved the GPU's memory in its own pool, or a
latency-critical loop where cudaMalloc / cudaFree would synchronise the device.
Its scratch is a fixed device array inside the library, so this test checks,
through the C ABI, that two calls in a row give exactly the table of the
ordinary allocating entry point (integer sums bit-exact, mean and SE to 1e-12),
that the shared scratch is cleared between calls, that the call leaves the
device's free memory unchanged on a context that has never evaluated, that
exactly 8192 pairs are served while more, host buffers and bf16 (tensor-core)
Leduc populations are refused. This file is collected last.
"""
import ctypes as C

import numpy as np
import pytest

import workloads
from gpu_util import context, load_population, need_gpu

pytestmark = pytest.mark.gpu


def _noalloc(ctx, pairs, n_eps, seed, out):
    from paper_2106_07551_gb300 import _abi
    lib = _abi.load()
    return lib.malib_eval_payoff_noalloc(ctx.handle, C.c_void_p(pairs.data_ptr()),
                                         int(pairs.shape[0]), n_eps, seed,
                                         C.c_void_p(out.data_ptr()))


@pytest.mark.parametrize("kind", ["leduc", "kuhn"])
def test_noalloc_matches_allocating_entry_point(kind):
    torch = need_gpu()
    w = (workloads.leduc(pop=4, with_bias=True, seed=77) if kind == "leduc"
         else workloads.kuhn())
    n_eps = 3000 if kind == "leduc" else 10_000
    ctx = context()
    load_population(ctx, w)
    d_pairs = torch.from_numpy(w.pair_ids).cuda()
    for seed in (5, 6):
        ref = ctx.eval_payoff(w.pair_ids, n_eps, seed)
        for _ in range(2):   # two calls in a row share (and must clear) the scratch
            out = torch.full((w.n_pairs, 4), -1.0, dtype=torch.float64, device="cuda")
            assert _noalloc(ctx, d_pairs, n_eps, seed, out) == 0, ctx.last_error()
            ctx.sync()
            got = out.cpu().numpy()
            np.testing.assert_array_equal(got[:, 2:], ref[:, 2:])
            np.testing.assert_allclose(got[:, :2], ref[:, :2], rtol=1e-12, atol=1e-15)
    # a smaller table after a larger one: stale sums must not leak in
    out = torch.zeros((3, 4), dtype=torch.float64, device="cuda")
    assert _noalloc(ctx, d_pairs[:3].contiguous(), n_eps, 9, out) == 0
    ctx.sync()
    ref = ctx.eval_payoff(w.pair_ids[:3].copy(), n_eps, 9)
    np.testing.assert_array_equal(out.cpu().numpy()[:, 2:], ref[:, 2:])
    ctx.close()


def test_noalloc_refuses_oversize_and_host_buffers():
    torch = need_gpu()
    from paper_2106_07551_gb300 import _abi
    w = workloads.kuhn()
    ctx = context()
    load_population(ctx, w)
    tiled = np.tile(w.pair_ids, (8193 // w.n_pairs + 1, 1))
    big = torch.from_numpy(tiled[:8193].copy()).cuda()
    out = torch.zeros((8193, 4), dtype=torch.float64, device="cuda")
    assert _noalloc(ctx, big, 10, 0, out) == _abi.MALIB_EINVAL
    assert "8192" in ctx.last_error()
    # exactly the capacity is served, with the ordinary entry point's table
    edge = torch.from_numpy(tiled[:8192].copy()).cuda()
    out = torch.full((8192, 4), -1.0, dtype=torch.float64, device="cuda")
    assert _noalloc(ctx, edge, 10, 3, out) == 0, ctx.last_error()
    ctx.sync()
    ref = ctx.eval_payoff(tiled[:8192].copy(), 10, 3)
    np.testing.assert_array_equal(out.cpu().numpy()[:, 2:], ref[:, 2:])
    lib = _abi.load()
    h_out = np.zeros((w.n_pairs, 4), np.float64)
    d_pairs = torch.from_numpy(w.pair_ids).cuda()
    code = lib.malib_eval_payoff_noalloc(ctx.handle, C.c_void_p(d_pairs.data_ptr()), w.n_pairs,
                                         10, 0, h_out.ctypes.data_as(C.c_void_p))
    assert code == _abi.MALIB_EINVAL
    ctx.close()
    # bf16 Leduc populations run on the tensor-core kernel, which this entry
    # point does not serve
    wb = workloads.leduc(pop=2, hidden=256, dtype=workloads.BF16, seed=79)
    ctx = context()
    load_population(ctx, wb)
    d_pairs = torch.from_numpy(wb.pair_ids).cuda()
    out = torch.zeros((wb.n_pairs, 4), dtype=torch.float64, device="cuda")
    assert _noalloc(ctx, d_pairs, 10, 0, out) == _abi.MALIB_EUNSUPPORTED
    ctx.close()


@pytest.mark.parametrize("kind", ["kuhn", "leduc"])
def test_noalloc_leaves_free_memory_unchanged(kind):
    """On a context that has never evaluated (so none of its evaluation
    buffers exists), two calls change the device's free memory by nothing. The
    kernels and the library's scratch array are loaded first on another
    context, so lazy module loading does not count."""
    torch = need_gpu()
    w = (workloads.leduc(pop=3, with_bias=True, seed=80) if kind == "leduc" else workloads.kuhn())
    n_eps = 2000 if kind == "leduc" else 10_000
    d_pairs = torch.from_numpy(w.pair_ids).cuda()
    out = torch.zeros((w.n_pairs, 4), dtype=torch.float64, device="cuda")
    warm = context()
    load_population(warm, w)
    ref = warm.eval_payoff(w.pair_ids, n_eps, 4)
    assert _noalloc(warm, d_pairs, n_eps, 4, out) == 0, warm.last_error()
    warm.sync()
    warm.close()
    out.fill_(-1.0)                            # torch's own kernel loaded before the window
    ctx = context()
    load_population(ctx, w)
    ctx.sync()
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(2):
        out.fill_(-1.0)
        assert _noalloc(ctx, d_pairs, n_eps, 4, out) == 0, ctx.last_error()
        ctx.sync()
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0, (free0, free1)
    np.testing.assert_array_equal(out.cpu().numpy()[:, 2:], ref[:, 2:])
    ctx.close()


@pytest.mark.parametrize("kind", ["kuhn", "leduc"])
def test_noalloc_captured_in_a_cuda_graph(kind):
    """The allocation-free call can be captured into a CUDA graph (zero, main
    and finalize kernels as graph nodes) and replayed: every replay gives the
    table of the ordinary entry point."""
    torch = need_gpu()
    import __graft_entry__
    __graft_entry__.build()
    from paper_2106_07551_gb300 import Context
    w = (workloads.leduc(pop=3, with_bias=True, seed=78) if kind == "leduc" else workloads.kuhn())
    n_eps = 2000 if kind == "leduc" else 10_000
    s = torch.cuda.Stream()
    ctx = Context(0, s)                      # every call of this context is ordered on s
    load_population(ctx, w)
    ref = ctx.eval_payoff(w.pair_ids, n_eps, 12)
    d_pairs = torch.from_numpy(w.pair_ids).cuda()
    out = torch.zeros((w.n_pairs, 4), dtype=torch.float64, device="cuda")
    with torch.cuda.stream(s):               # warm-up outside the capture
        assert _noalloc(ctx, d_pairs, n_eps, 12, out) == 0, ctx.last_error()
    s.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        assert _noalloc(ctx, d_pairs, n_eps, 12, out) == 0, ctx.last_error()
    for _ in range(3):
        out.fill_(-1.0)
        g.replay()
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        np.testing.assert_array_equal(got[:, 2:], ref[:, 2:])
        np.testing.assert_allclose(got[:, :2], ref[:, :2], rtol=1e-12, atol=1e-15)
    ctx.sync()
    ctx.close()
