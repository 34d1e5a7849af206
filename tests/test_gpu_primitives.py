"""GPU parity of the sampling primitives every kernel uses: Philox4x32-10,
the deterministic exp and the masked inverse-CDF draw, bit for bit against the
oracle; the deterministic exp also against CUDA's expf within 2 ulp."""
import numpy as np
import pytest

from gpu_util import context, need_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    c = context()
    yield c
    c.close()


@pytest.mark.parametrize("seed", [0, 2106075512, 0xDEADBEEFCAFEF00D])
def test_philox_bit_exact(ctx, orc, seed):
    torch = need_gpu()
    rng = np.random.default_rng(seed & 0xFFFF)
    n = 1 << 20
    ctr = rng.integers(0, 2**32, size=(n, 4), dtype=np.uint64).astype(np.uint32)
    ctr[:8] = [[0, 0, 0, 0], [0xFFFFFFFF] * 4, [1, 0, 0, 0], [0, 0, 0, 0xFFFFFFFF],
               [5, 0, 7, 0xFFFFFFFF], [2**31, 1, 24, 7], [0, 0, 0x80000003, 0xFFFFFFFF],
               [123, 0, 0, 1]]
    d_ctr = torch.from_numpy(ctr.view(np.int32)).cuda()
    d_out = torch.empty_like(d_ctr)
    ctx.selftest_philox(d_ctr, seed, d_out)
    ctx.sync()
    got = d_out.cpu().numpy().view(np.uint32)
    np.testing.assert_array_equal(got, orc.philox(ctr, seed))


@pytest.mark.parametrize("n,calls", [(1, 0), (1000, 7), (4099, 33)])
def test_philox_digest(ctx, orc, n, calls):
    """The throughput probe folds exactly the oracle's Philox words."""
    torch = need_gpu()
    seed = 0x0123456789ABCDEF
    d_out = torch.zeros(n, dtype=torch.int32, device="cuda")
    ctx.philox_digest(seed, calls, d_out)
    ctx.sync()
    got = d_out.cpu().numpy().view(np.uint32)
    t = np.arange(n, dtype=np.uint64)
    want = np.zeros(n, np.uint32)
    for i in range(calls):
        ctr = np.stack([(t & 0xFFFFFFFF).astype(np.uint32), (t >> 32).astype(np.uint32),
                        np.full(n, i, np.uint32), np.zeros(n, np.uint32)], axis=1)
        r = orc.philox(ctr, seed)
        want ^= r[:, 0] ^ r[:, 1] ^ r[:, 2] ^ r[:, 3]
    np.testing.assert_array_equal(got, want)


def test_det_expf_bit_exact_and_near_expf(ctx, orc):
    torch = need_gpu()
    x = np.concatenate([np.linspace(-90, 89, 2_000_001, dtype=np.float32),
                        np.float32([0.0, -0.0, -87.0, -86.99999, 88.0, 88.5, -1e-30, np.nan])])
    x = x.astype(np.float32)
    d_x = torch.from_numpy(x).cuda()
    d_y = torch.empty_like(d_x)
    ctx.selftest_det_expf(d_x, d_y)
    ctx.sync()
    got = d_y.cpu().numpy()
    ref = orc.det_expf(x)
    np.testing.assert_array_equal(got.view(np.uint32), ref.view(np.uint32))
    # against CUDA's own expf (torch.exp on the device), inside the domain
    m = (x > -86.9) & (x < 88.0)
    cu = torch.exp(d_x).cpu().numpy()
    ulp = np.spacing(np.abs(cu[m]))
    assert (np.abs(got[m].astype(np.float64) - cu[m]) / ulp).max() <= 2.0


@pytest.mark.parametrize("A", [2, 3, 5])
def test_sample_bit_exact(ctx, orc, A):
    torch = need_gpu()
    rng = np.random.default_rng(A)
    n = 1 << 18
    lg = (rng.standard_normal((n, A)) * rng.choice([0.1, 1, 10, 60], size=(n, 1))).astype(np.float32)
    lg[: n // 8] = np.round(lg[: n // 8])           # many exact ties
    legal = (rng.random((n, A)) < 0.75).astype(np.uint8)
    legal[np.arange(n), rng.integers(0, A, n)] = 1
    u = ((rng.integers(0, 1 << 24, n)) * 2.0 ** -24).astype(np.float32)
    u[:16] = [0.0, 1 - 2 ** -24] * 8
    d = [torch.from_numpy(a).cuda() for a in (lg, legal, u)]
    out = torch.empty(n, dtype=torch.int32, device="cuda")
    ctx.selftest_sample(d[0], d[1], d[2], out)
    ctx.sync()
    np.testing.assert_array_equal(out.cpu().numpy(), orc.sample(lg, legal, u))


@pytest.mark.parametrize("dtype,N,K", [("bf16", 256, 256), ("bf16", 16, 16), ("bf16", 128, 48),
                                       ("tf32", 256, 128), ("tf32", 64, 24)])
def test_tensor_core_gemm(ctx, dtype, N, K):
    """tcgen05 MMA with the kernels' operand layout against an fp64 matmul of
    the same (bf16 / tf32-truncated) operands."""
    torch = need_gpu()
    from paper_2106_07551_gb300 import MALIB_BF16, MALIB_F32
    g = torch.Generator().manual_seed(N * 1000 + K)
    A = torch.randn(128, K, generator=g)
    B = torch.randn(N, K, generator=g)
    if dtype == "bf16":
        Ab, Bb = A.to(torch.bfloat16), B.to(torch.bfloat16)
        ref = Ab.double() @ Bb.double().T
        dA, dB = Ab.view(torch.int16).cuda(), Bb.view(torch.int16).cuda()
        code = MALIB_BF16
    else:
        mask = torch.tensor(-8192, dtype=torch.int32)      # keep 19 high bits (tf32)
        At = (A.view(torch.int32) & mask).view(torch.float32)
        Bt = (B.view(torch.int32) & mask).view(torch.float32)
        ref = At.double() @ Bt.double().T
        dA, dB = A.cuda(), B.cuda()
        code = MALIB_F32
    D = torch.full((128, N), float("nan"), device="cuda")
    ctx.selftest_mma(code, dA, dB, D)
    ctx.sync()
    got = D.cpu().double()
    scale = ref.abs().max().item()
    err = (got - ref).abs().max().item()
    # tf32 inputs may be rounded rather than truncated by the unit: allow 2^-10
    tol = (1e-5 if dtype == "bf16" else 2e-3) * scale
    assert err <= tol, (err, scale)
