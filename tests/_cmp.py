"""Comparison helpers for the GPU-vs-oracle parity tests (tolerances stated here).

Tolerances:
  - integers (Philox words, labels, U counts): bit-exact;
  - A-hat: bit-exact (the same IEEE operations on the same exact integers);
  - fp16 live activations (assert_live_close): |g - o| <= one fp16 step at
    the larger of the two + 2 |a_g - a_o| + 2^-15 |o - a| + 2^-20 (|a| + |c|),
    with a = a_o the oracle's reference, a_g the GPU's (within the normals
    tolerance below) and c the segment's coefficient (sigma_s mu of Eq. 2,
    or eps ||a|| / ||g|| of the Gaussian tamper).  The GPU evaluates
    v = a_g + c z in fp32 (one fused multiply-add, 2^-24 |v|; the relative
    form a (1 + sigma z) takes three roundings and scales a_g - a_o by
    1 + sigma z) with a normal z within 2^-20 max(|z|, 2^-6) of the exact
    one and a coefficient formed from fp32 partial sums of at most 256 terms
    per thread (relative error below 2^-16); the oracle evaluates it in fp64
    from a_o; each then rounds to fp16 once, which adds at most one step.
    So the bound holds with |c z| taken as |o - a|.  Away from a cancellation
    a + c z ~ 0 it is one fp16 step; near one the fp16 step is far below
    the fp32 evaluation error of a and c z, and the bound is that error;
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
LIVE_DIFF_RTOL = 2.0 ** -15     # of |o - a| = |c z|: the coefficient's and the normal's error
LIVE_ABS_RTOL = 2.0 ** -20      # of |a| + |c|: the fused rounding and the normals' 2^-6 floor
FP16_MAX_STEP = 65536.0         # where binary16 overflows to infinity


def ordered_half(bits):
    b = np.asarray(bits).view(np.uint16).astype(np.int64)
    return np.where(b & 0x8000, -(b & 0x7FFF), b & 0x7FFF)


def half_ulp_distance(a_bits, b_bits):
    return np.abs(ordered_half(a_bits) - ordered_half(b_bits))


def fp16_step(x):
    """Spacing of binary16 at |x|: 2^(floor(log2 |x|) - 10), and 2^-24 in the
    subnormal range."""
    ax = np.abs(np.asarray(x, np.float64))
    return np.exp2(np.floor(np.log2(np.maximum(ax, 2.0 ** -14))) - 10.0)


def assert_live_close(g_bits, o_bits, g_refs, o_refs, coef=0.0, what="live values"):
    """fp16 live values (binary16 bits) from the GPU against the oracle's,
    with both sides' references; coef broadcasts against the leading axes
    (one per segment).  Returns the largest distance in fp16 steps, for
    reporting."""
    g_bits = np.asarray(g_bits).view(np.uint16)
    o_bits = np.asarray(o_bits).view(np.uint16)
    g = g_bits.view(np.float16).astype(np.float64)
    o = o_bits.view(np.float16).astype(np.float64)
    a = np.asarray(o_refs, np.float64)
    da = np.abs(np.asarray(g_refs, np.float64) - a)
    c = np.abs(np.asarray(coef, np.float64))
    if c.ndim:
        c = c.reshape(c.shape + (1,) * (a.ndim - c.ndim))
    assert np.array_equal(np.isnan(g), np.isnan(o)), f"{what}: NaN pattern"
    # an overflow is the step above 65504: it rounds from 65520 up
    gv = np.where(np.isinf(g), np.sign(g) * FP16_MAX_STEP, g)
    ov = np.where(np.isinf(o), np.sign(o) * FP16_MAX_STEP, o)
    with np.errstate(invalid="ignore"):
        err = np.abs(gv - ov)
    tol = (fp16_step(np.maximum(np.abs(gv), np.abs(ov))) + 2.0 * da
           + LIVE_DIFF_RTOL * np.abs(ov - a) + LIVE_ABS_RTOL * (np.abs(a) + c))
    bad = err > tol
    bad &= ~np.isnan(err)
    assert not bad.any(), (f"{what}: {int(bad.sum())} of {bad.size} outside the bound; worst "
                           f"{float(np.max(err[bad] / tol[bad])):.3g} of it")
    return int(half_ulp_distance(g_bits, o_bits).max())


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
