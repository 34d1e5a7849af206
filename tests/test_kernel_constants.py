"""Host-side checks of numeric facts the kernels rely on (no GPU needed)."""
import os
import re

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_collision_threshold_is_exact():
    """The spread kernels test |p_i - p_j| < 0.3 on the squared distance: with
    the correctly rounded fp32 square root, fl(sqrt(s)) < 0.3f  <=>  s < T.
    T must be the smallest fp32 value whose rounded root reaches 0.3f."""
    src = open(os.path.join(ROOT, "paper_2106_07551_gb300", "csrc", "spread_env.cuh")).read()
    lit = re.search(r"kCollideSq\s*=\s*(0x[0-9a-fA-Fp.+-]+)f;", src).group(1)
    T = np.float32(float.fromhex(lit))
    c = np.float32(0.3)
    assert np.sqrt(T) >= c
    assert np.sqrt(np.nextafter(T, np.float32(0))) < c
    bits = int(np.float32(T).view(np.uint32))
    s = np.arange(bits - 1_000_000, bits + 1_000_000, dtype=np.int64).astype(np.uint32).view(np.float32)
    np.testing.assert_array_equal(np.sqrt(s) < c, s < T)


def test_min_of_rounded_roots_is_root_of_min():
    """fl(sqrt(.)) is monotone, so min_a fl(sqrt(x_a)) == fl(sqrt(min_a x_a))
    (the kernels take one root per landmark)."""
    rng = np.random.default_rng(0)
    x = (rng.random((200_000, 8)) * 8).astype(np.float32)
    np.testing.assert_array_equal(np.sqrt(x).min(axis=1), np.sqrt(x.min(axis=1)))
