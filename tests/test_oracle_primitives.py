"""Pins for the oracle's primitives: Philox4x32-10, det_expf, masked sampling,
bf16 rounding and the MLP forward. Each is checked against something other than
itself: an independent library implementation, the mathematics, or exact
special cases."""
import math
import os
import subprocess
import sys
import textwrap

import numpy as np
import pytest


# ----------------------------------------------------------------- Philox
_TRITON_SCRIPT = textwrap.dedent("""
    import os, sys
    os.environ["TRITON_INTERPRET"] = "1"
    import numpy as np, torch, triton, triton.language as tl

    @triton.jit
    def k(out, seed, c0p, c1p, c2p, c3p, N: tl.constexpr):
        o = tl.arange(0, N)
        a, b, c, d = tl.philox(seed, tl.load(c0p + o), tl.load(c1p + o), tl.load(c2p + o),
                               tl.load(c3p + o), 10)
        tl.store(out + o * 4 + 0, a); tl.store(out + o * 4 + 1, b)
        tl.store(out + o * 4 + 2, c); tl.store(out + o * 4 + 3, d)

    ctr = np.load(sys.argv[1]); seed = int(sys.argv[2]); N = ctr.shape[0]
    cs = [torch.from_numpy(ctr[:, i].astype(np.int64)).to(torch.uint32) for i in range(4)]
    out = torch.zeros(N * 4, dtype=torch.uint32)
    k[(1,)](out, seed, *cs, N=N)
    np.save(sys.argv[3], out.view(torch.int32).numpy().view(np.uint32).reshape(N, 4))
""")


@pytest.mark.parametrize("seed", [0, 12345, 2106075512, 0xFFFFFFFF, 0x123456789ABCDEF0])
def test_philox_matches_triton_interpreter(orc, tmp_path, seed):
    """Triton's CPU interpreter carries its own Philox4x32-10 (key = seed lo, hi)."""
    pytest.importorskip("triton")
    pytest.importorskip("torch")
    rng = np.random.default_rng(seed & 0xFFFF)
    ctr = rng.integers(0, 2**32, size=(256, 4), dtype=np.uint64).astype(np.uint32)
    ctr[:4] = [[0, 0, 0, 0], [0xFFFFFFFF] * 4, [1, 0, 0, 0], [0, 0, 0, 0xFFFFFFFF]]
    np.save(tmp_path / "ctr.npy", ctr)
    script = tmp_path / "tp.py"
    script.write_text(_TRITON_SCRIPT)
    env = dict(os.environ, TRITON_INTERPRET="1")
    r = subprocess.run([sys.executable, str(script), str(tmp_path / "ctr.npy"), str(seed),
                        str(tmp_path / "out.npy")], env=env, capture_output=True, text=True,
                       timeout=600)
    if r.returncode != 0:
        pytest.skip(f"triton interpreter unavailable: {r.stderr[-300:]}")
    ref = np.load(tmp_path / "out.npy")
    np.testing.assert_array_equal(orc.philox(ctr, seed), ref)


def test_philox_uniformity_and_key_sensitivity(orc):
    n = 1 << 16
    ctr = np.zeros((n, 4), np.uint32)
    ctr[:, 0] = np.arange(n, dtype=np.uint32)
    ctr[:, 2] = 7
    out = orc.philox(ctr, 99)
    # chi-square of the top 4 bits of every word, 16 cells
    for w in range(4):
        cnt = np.bincount(out[:, w] >> 28, minlength=16)
        chi2 = ((cnt - n / 16) ** 2 / (n / 16)).sum()
        assert chi2 < 50.0, chi2     # 15 dof, p ~ 1e-5
    # bit balance
    bits = np.unpackbits(out.view(np.uint8)).mean()
    assert abs(bits - 0.5) < 0.005
    assert len(np.unique(out[:, 0])) > n - 5
    assert not np.array_equal(orc.philox(ctr[:16], 99), orc.philox(ctr[:16], 100))
    assert not np.array_equal(orc.philox(ctr[:16], 99), orc.philox(ctr[:16], 99 + (1 << 32)))


# ----------------------------------------------------------------- det_expf
def _ulp_err(y, ref):
    y = y.astype(np.float64)
    ulp = np.spacing(np.abs(ref).astype(np.float32)).astype(np.float64)
    return np.abs(y - ref) / ulp


def test_det_expf_accuracy(orc):
    x = np.concatenate([np.linspace(-86.9, 88.0, 400_001, dtype=np.float32),
                        np.float32(-np.logspace(-8, 1.9, 20_000))]).astype(np.float32)
    y = orc.det_expf(x)
    ref = np.exp(x.astype(np.float64))
    assert _ulp_err(y, ref).max() <= 2.0


def test_det_expf_special_values(orc):
    assert orc.det_expf(np.array([0.0], np.float32))[0] == 1.0
    y = orc.det_expf(np.array([-87.0, -100.0, -1e30, -np.inf], np.float32))
    assert np.all(y == 0.0)
    # exact powers of two: exp(k ln2) within 1 ulp of 2^k
    k = np.arange(-120, 120)
    y = orc.det_expf((k * np.log(2.0)).astype(np.float32))
    ref = np.exp((k * np.log(2.0)).astype(np.float32).astype(np.float64))
    assert _ulp_err(y, ref).max() <= 1.5


# ----------------------------------------------------------------- sampling
def test_sample_inverse_cdf_fractions(orc):
    """Over a uniform grid of u, action a is drawn for a fraction of the grid
    equal to its softmax probability (to the grid resolution)."""
    rng = np.random.default_rng(3)
    for A in (3, 5):
        for _ in range(5):
            lg = rng.standard_normal(A).astype(np.float32) * 2
            legal = (rng.random(A) < 0.7).astype(np.uint8)
            legal[rng.integers(A)] = 1
            u = (np.arange(1 << 16, dtype=np.float64) / (1 << 16)).astype(np.float32)
            acts = orc.sample(np.tile(lg, (u.size, 1)), np.tile(legal, (u.size, 1)), u)
            assert np.all(legal[acts] == 1)
            p = np.where(legal == 1, np.exp(lg.astype(np.float64) - lg[legal == 1].max()), 0.0)
            p /= p.sum()
            frac = np.bincount(acts, minlength=A) / u.size
            np.testing.assert_allclose(frac, p, atol=2.0 / u.size + 1e-6)


def test_sample_special_cases(orc):
    lg = np.array([[0.3, -1.0, 2.0]] * 4, np.float32)
    # single legal action is always taken
    legal = np.array([[0, 1, 0]] * 4, np.uint8)
    u = np.array([0.0, 0.5, 0.999, 1 - 2**-24], np.float32)
    assert list(orc.sample(lg, legal, u)) == [1, 1, 1, 1]
    # u = 0 picks the first legal action; u -> 1 the last
    legal = np.array([[1, 1, 1]] * 2, np.uint8)
    assert list(orc.sample(lg[:2], legal, np.array([0.0, 1 - 2**-24], np.float32))) == [0, 2]
    # equal logits split u into equal thirds
    lg3 = np.zeros((3, 3), np.float32)
    acts = orc.sample(lg3, np.ones((3, 3), np.uint8), np.array([0.30, 0.40, 0.70], np.float32))
    assert list(acts) == [0, 1, 2]
    # a masked action never wins, even with a huge logit
    lg = np.array([[50.0, 0.0, 0.0]], np.float32)
    assert orc.sample(lg, np.array([[0, 1, 1]], np.uint8), np.array([0.1], np.float32))[0] == 1


# ----------------------------------------------------------------- bf16
def test_bf16_round_matches_torch(orc):
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(5)
    x = np.concatenate([rng.standard_normal(4000).astype(np.float32) * 10,
                        np.float32([1 + 2**-8, 1 + 3 * 2**-8, -1 - 2**-8, 0.0, 1e-30, 3e38])])
    ours = np.array([orc.bf16_round(v) for v in x], np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()
    np.testing.assert_array_equal(ours, ref)
    assert orc.bf16_round(1 + 2**-8) == 1.0               # tie to even (down)
    assert orc.bf16_round(1 + 3 * 2**-8) == 1 + 2**-6     # tie to even (up)


# ----------------------------------------------------------------- MLP
def _unpack(params, dims):
    i, h1, h2, o = dims
    k = 0
    out = []
    for fi, fo in ((i, h1), (h1, h2), (h2, o)):
        W = params[k:k + fi * fo].reshape(fo, fi); k += fi * fo
        b = params[k:k + fo]; k += fo
        out += [W.astype(np.float64), b.astype(np.float64)]
    return out


def test_mlp_forward_against_numpy(orc):
    import workloads
    rng = np.random.default_rng(11)
    for dims in ((17, 128, 128, 3), (18, 64, 64, 5), (34, 256, 256, 5)):
        p = workloads.random_mlp(rng, dims, with_bias=True)
        x = rng.standard_normal((64, dims[0])).astype(np.float32)
        W1, b1, W2, b2, W3, b3 = _unpack(p, dims)
        h = np.maximum(x.astype(np.float64) @ W1.T + b1, 0)
        h = np.maximum(h @ W2.T + b2, 0)
        ref = h @ W3.T + b3
        got = orc.mlp_forward(p, dims, x)
        np.testing.assert_allclose(got, ref.astype(np.float32), rtol=1e-6, atol=1e-6)


def test_mlp_forward_hand_case(orc):
    """2 -> 2 -> 2 -> 2 net whose ReLUs clip one unit per layer."""
    dims = (2, 2, 2, 2)
    W1 = [[1, 0], [0, -1]]; b1 = [0.5, 0.0]
    W2 = [[2, 0], [1, 1]]; b2 = [0.0, -10.0]
    W3 = [[1, 1], [-1, 3]]; b3 = [0.25, 0.0]
    p = np.array(sum([sum(W1, []), b1, sum(W2, []), b2, sum(W3, []), b3], []), np.float32)
    x = np.array([[1.0, 2.0]], np.float32)
    # h1 = relu([1.5, -2]) = [1.5, 0]; h2 = relu([3, 1.5 - 10]) = [3, 0]; out = [3.25, -3]
    np.testing.assert_array_equal(orc.mlp_forward(p, dims, x), [[3.25, -3.0]])


def test_mlp_forward_bf16_emulation(orc):
    torch = pytest.importorskip("torch")
    import workloads
    rng = np.random.default_rng(12)
    dims = (17, 256, 256, 3)
    p = workloads.random_mlp(rng, dims, with_bias=True)
    x = rng.standard_normal((32, 17)).astype(np.float32)

    def bf(a):
        return torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(torch.bfloat16).to(
            torch.float32).numpy().astype(np.float64)

    W1, b1, W2, b2, W3, b3 = _unpack(p, dims)
    h = bf(np.maximum(bf(x) @ bf(W1).T + b1, 0))
    h = bf(np.maximum(h @ bf(W2).T + b2, 0))
    ref = h @ bf(W3).T + b3
    got = orc.mlp_forward(p, dims, x, bf16=True)
    np.testing.assert_allclose(got, ref, rtol=2e-3, atol=2e-3)
    # and it differs from the fp32 forward by more than rounding noise
    assert np.abs(got - orc.mlp_forward(p, dims, x)).max() > 1e-4
