"""Pins of the oracle's random-number layer (not the GPU).

Philox4x32-10 is pinned against cuRAND's host-side Philox generator (a
library run on the CPU): its output block i, after a generator offset of 4*j
words, is Philox4x32-10 with key = (seed lo, seed hi) and counter
(b // 65536 mod 2^32, b // 2^48, b mod 65536, 0) for b = i + j.  Every
counter the method uses has c3 = 0, so the whole space it draws from is
covered.  Box-Muller is pinned by special cases with closed forms and by a
Kolmogorov-Smirnov test against scipy's normal CDF; the bounded draw by range
and uniformity checks.
"""
import ctypes
import ctypes.util
import math
import os

import numpy as np
import pytest

CURAND_RNG_PSEUDO_PHILOX4_32_10 = 161


def _curand():
    for name in ("/usr/local/cuda/lib64/libcurand.so", ctypes.util.find_library("curand")):
        if name and (os.path.exists(name) or not name.startswith("/")):
            try:
                return ctypes.CDLL(name)
            except OSError:
                continue
    return None


def curand_blocks(seed, block0, n_blocks):
    lib = _curand()
    if lib is None:
        pytest.skip("libcurand not available")
    gen = ctypes.c_void_p()
    assert lib.curandCreateGeneratorHost(ctypes.byref(gen), CURAND_RNG_PSEUDO_PHILOX4_32_10) == 0
    try:
        assert lib.curandSetPseudoRandomGeneratorSeed(gen, ctypes.c_ulonglong(seed)) == 0
        assert lib.curandSetGeneratorOffset(gen, ctypes.c_ulonglong((4 * block0) % 2**64)) == 0
        out = np.zeros(4 * n_blocks, dtype=np.uint32)
        assert lib.curandGenerate(gen, out.ctypes.data_as(ctypes.c_void_p),
                                  ctypes.c_size_t(out.size)) == 0
    finally:
        lib.curandDestroyGenerator(gen)
    return out.reshape(n_blocks, 4)


def _ctr_of(b):
    return (b // 65536) % 2**32, b // 2**48, b % 65536


@pytest.mark.parametrize("seed", [0, 1, 0x123456789ABCDEF0, 2**64 - 1])
def test_philox_matches_curand_first_blocks(orc, seed):
    ref = curand_blocks(seed, 0, 300)
    for b in range(300):
        c0, c1, c2 = _ctr_of(b)
        got = orc.philox_words(seed, c1, c2, 0, c0, 1)
        assert list(got) == list(ref[b]), b


@pytest.mark.parametrize("c0,c1,c2", [
    (1, 0, 5), (3, 1, 7), (0x1234, 0x55, 0xFFF0), (0xFFFFFFFF, 7, 65535),
    (262143, 4095, 8), (17, 16383, 4 * 323 + 3), (5, 9999, 4 * 7 + 3),
])
def test_philox_matches_curand_far_counters(orc, c0, c1, c2):
    """Counters with large c0 and nonzero c1 (segment ids, aux purposes)."""
    if c2 >= 65536:
        pytest.skip("c2 beyond cuRAND's subsequence range")
    seed = 0xFEDCBA9876543210
    b = ((c1 << 32 | c0) * 65536) + c2
    ref = curand_blocks(seed, b, 1)[0]
    got = orc.philox_words(seed, c1, c2, 0, c0, 1)
    assert list(got) == list(ref)


def test_philox_words_block_order(orc):
    """philox_words(first, n) is block-major with counter word 0 = first + i."""
    w = orc.philox_words(7, 11, 13, 0, 100, 5).reshape(5, 4)
    for i in range(5):
        assert list(w[i]) == list(orc.philox4x32_10([100 + i, 11, 13, 0], [7, 0]))


def test_philox_bits_balanced(orc):
    w = orc.philox_words(42, 0, 0, 0, 0, 1 << 14)
    bits = np.unpackbits(w.view(np.uint8))
    n = bits.size
    assert abs(bits.mean() - 0.5) < 5 * 0.5 / math.sqrt(n)
    counts = np.bincount(w.view(np.uint8), minlength=256)
    exp = w.size * 4 / 256
    chi2 = ((counts - exp) ** 2 / exp).sum()
    assert chi2 < 255 + 6 * math.sqrt(2 * 255)


# --------------------------------------------------------------------------
# Box-Muller

def test_box_muller_special_cases(orc):
    # u1 = 1 (x0 >> 8 = 2^24 - 1): radius 0, both normals are zero
    z0, z1 = orc.box_muller(0xFFFFFFFF, 0x12345678)
    assert z0 == 0.0 and z1 == 0.0
    # u1 = 1/2 (x0 >> 8 = 2^23 - 1): radius sqrt(2 ln 2) = 1.1774100225154747
    r = 1.1774100225154747
    z0, z1 = orc.box_muller((2**23 - 1) << 8, 0)   # u2 = 0: cos = 1, sin = 0
    assert z0 == pytest.approx(r, rel=1e-15) and z1 == 0.0
    z0, z1 = orc.box_muller((2**23 - 1) << 8, (2**22) << 8)   # u2 = 1/4
    assert abs(z0) < 1e-15 and z1 == pytest.approx(r, rel=1e-15)
    z0, z1 = orc.box_muller((2**23 - 1) << 8, (2**23) << 8)   # u2 = 1/2
    assert z0 == pytest.approx(-r, rel=1e-15) and abs(z1) < 1e-15
    # the low 8 bits of each word are ignored
    assert orc.box_muller(0xABCDEF00, 0x13579B00) == orc.box_muller(0xABCDEFFF, 0x13579BFF)
    # u1 = 2^-24 (x0 >> 8 = 0): largest radius sqrt(48 ln 2)
    z0, _ = orc.box_muller(0, 0)
    assert z0 == pytest.approx(math.sqrt(48 * math.log(2)), rel=1e-15)


def test_box_muller_pairs_is_the_pairwise_transform(orc):
    """The array form used by the exhaustive device sweep is the scalar
    transform applied pair by pair."""
    rng = np.random.default_rng(5)
    w = rng.integers(0, 2**32, size=(257, 2), dtype=np.uint64).astype(np.uint32)
    w[0] = (0xFFFFFFFF, 0)
    z = orc.box_muller_pairs(w)
    for i in range(w.shape[0]):
        assert tuple(z[i]) == orc.box_muller(int(w[i, 0]), int(w[i, 1]))


def test_normals_distribution(orc):
    stats = pytest.importorskip("scipy.stats")
    z = orc.philox_normals(2024, 3, 4, 0, 0, 1 << 16)
    n = z.size
    assert abs(z.mean()) < 5 / math.sqrt(n)
    assert abs(z.var() - 1.0) < 5 * math.sqrt(2.0 / n)
    assert stats.kstest(z, stats.norm.cdf).pvalue > 1e-4
    pairs = z.reshape(-1, 2)
    assert abs(np.corrcoef(pairs[:, 0], pairs[:, 1])[0, 1]) < 5 / math.sqrt(pairs.shape[0])


def test_normals_layout(orc):
    """Element 4q + j of a stream is normal j of block q: (x0, x1) -> 0, 1; (x2, x3) -> 2, 3."""
    w = orc.philox_words(9, 1, 2, 0, 5, 1)
    z = orc.philox_normals(9, 1, 2, 0, 5, 1)
    assert tuple(z[:2]) == orc.box_muller(w[0], w[1])
    assert tuple(z[2:]) == orc.box_muller(w[2], w[3])


# --------------------------------------------------------------------------
# Lemire bounded draws

@pytest.mark.parametrize("n", [1, 2, 3, 7, 1000, 8192, 2**31 + 1, 2**32 - 1])
def test_bounded_range_and_uniformity(orc, n):
    v = orc.aux_bounded(77, 1, 0, 0, n, 4000).astype(np.int64)
    assert v.min() >= 0 and v.max() < n
    if n == 1:
        assert (v == 0).all()
        return
    k = min(n, 8)
    bins = (v * k) // n
    counts = np.bincount(bins, minlength=k)
    # bins of [0, n) by floor(v*k/n) hold floor or ceil of n/k values
    exp = v.size / k
    assert ((counts - exp) ** 2 / exp).sum() < (k - 1) + 8 * math.sqrt(2 * (k - 1))


def test_bounded_first_draw_is_multiply_shift(orc):
    """Without rejection the draw is floor(x * n / 2^32) of the next word."""
    n = 1000
    words = orc.philox_words(5, (1 << 24) | 0, 4 * 9 + 3, 0, 0, 2)
    v = orc.aux_bounded(5, 1, 0, 9, n, 8)
    for i in range(8):
        x = int(words[i])
        assert (x * n) % 2**32 >= (2**32 - n) % n   # no rejection for this seed
        assert v[i] == (x * n) >> 32
