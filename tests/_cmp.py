"""Comparison helpers for the GPU-vs-oracle parity tests (tolerances stated here).

Tolerances:
  - integers (Philox words, labels, U counts): bit-exact;
  - A-hat: bit-exact (the same IEEE operations on the same exact integers);
  - fp16 live activations: within 1 fp16 ulp (the GPU rounds fp32 -> fp16,
    the oracle fp64 -> fp16);
  - normals and references: |g - o| <= 2^-20 max(|o|, 2^-6) (8 fp32 ulp of the
    larger of |o| and 1/64; logf, sqrtf and sincospif are each within a couple
    of ulp);
  - rel_l2: within 1e-5 relative of the fp64 oracle on the same bytes;
  - max_abs: equal to the oracle's fp64 maximum rounded to fp32;
  - cos_dev: |g - o| <= 1e-5 max(o, m^2 / 2) + 1e-12: the GPU forms it from
    fp32-accumulated sums whose error scales with m^2 / 2 (it is near zero for
    a pure rescale, where any fp32 sum error dominates the true value).
"""
import numpy as np

NORMAL_RTOL = 2.0 ** -20
NORMAL_FLOOR = 2.0 ** -6
REL_L2_RTOL = 1e-5
COS_RTOL = 1e-5


def ordered_half(bits):
    b = np.asarray(bits).view(np.uint16).astype(np.int64)
    return np.where(b & 0x8000, -(b & 0x7FFF), b & 0x7FFF)


def half_ulp_distance(a_bits, b_bits):
    return np.abs(ordered_half(a_bits) - ordered_half(b_bits))


def assert_normals_close(g, o, scale=1.0, what="normals"):
    g = np.asarray(g, np.float64)
    o = np.asarray(o, np.float64)
    tol = NORMAL_RTOL * np.maximum(np.abs(o), NORMAL_FLOOR * scale)
    bad = np.abs(g - o) > tol
    assert not bad.any(), (f"{what}: {bad.sum()} of {bad.size} outside tolerance; "
                           f"worst {np.max(np.abs(g - o) / np.maximum(np.abs(o), NORMAL_FLOOR * scale))}")


def assert_scores_close(g, o, what="scores"):
    """g: float32 [3][...] from the GPU; o: float64 [3][...] from the oracle."""
    g = np.asarray(g)
    o = np.asarray(o)
    rel_g, rel_o = g[0].astype(np.float64), o[0]
    fin = np.isfinite(rel_o)
    assert np.array_equal(np.isnan(rel_g), np.isnan(rel_o)), f"{what}: rel_l2 NaN pattern"
    assert np.array_equal(np.isinf(rel_g), np.isinf(rel_o)), f"{what}: rel_l2 inf pattern"
    err = np.abs(rel_g[fin] - rel_o[fin])
    lim = REL_L2_RTOL * np.abs(rel_o[fin])
    assert np.all(err <= lim), f"{what}: rel_l2 worst rel err {np.max(err / np.maximum(np.abs(rel_o[fin]), 1e-300))}"
    assert np.array_equal(g[1], o[1].astype(np.float32)), f"{what}: max_abs not exact"
    cos_g, cos_o = g[2].astype(np.float64), o[2]
    fin = np.isfinite(cos_o)
    assert np.array_equal(np.isnan(cos_g), np.isnan(cos_o)), f"{what}: cos_dev NaN pattern"
    m2 = np.where(np.isfinite(rel_o), rel_o, 0.0) ** 2 / 2
    lim = COS_RTOL * np.maximum(cos_o, m2) + 1e-12
    err = np.abs(cos_g - cos_o)
    assert np.all(err[fin] <= lim[fin]), f"{what}: cos_dev worst {np.max(err[fin] / lim[fin])} of tolerance"
