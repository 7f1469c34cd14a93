"""Pins of the oracle's fp16 rounding and drift statistics (not the GPU).

fp16 rounding is checked against numpy's float64 -> float16 conversion (a
correctly rounded library routine); the drift statistics against hand-worked
values (tests/golden/drift_handworked.json), closed forms of Eq. 4 and the
cosine ablation, and numpy's fp64 norms and dot products.
"""
import json
import math
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_half_from_double_matches_numpy(orc):
    rng = np.random.Generator(np.random.PCG64(1))
    xs = [0.0, -0.0, 1.0, -1.0, 65504.0, 65519.999, 65520.0, -65520.0, 1e9,
          2.0**-24, 2.0**-25, 3 * 2.0**-26, 2.0**-14, 2.0**-14 - 2.0**-25, 5.960464477539063e-08,
          float("inf"), float("-inf")]
    # every fp16 midpoint around a sample of values: ties go to even
    for h in rng.integers(0, 0x7BFF, size=2000):
        lo = float(np.uint16(h).view(np.float16))
        hi = float(np.uint16(h + 1).view(np.float16))
        xs += [lo, (lo + hi) / 2, -(lo + hi) / 2, np.nextafter((lo + hi) / 2, 0.0),
               np.nextafter((lo + hi) / 2, 1e9)]
    xs += list(rng.standard_normal(2000) * 10.0 ** rng.uniform(-9, 5, 2000))
    for x in xs:
        with np.errstate(over="ignore"):
            want = int(np.float64(x).astype(np.float16).view(np.uint16))
        assert orc.half_from_double(x) == want, x
    assert orc.half_from_double(float("nan")) & 0x7C00 == 0x7C00


def test_half_to_double_all_patterns(orc):
    for h in range(0, 65536, 7):
        want = float(np.uint16(h).view(np.float16))
        got = orc.half_to_double(h)
        if math.isnan(want):
            assert math.isnan(got)
        else:
            assert got == want and math.copysign(1, got) == math.copysign(1, want)


def _h(values):
    return np.asarray(values, dtype=np.float16).view(np.uint16)


def test_drift_handworked(orc):
    cases = json.load(open(os.path.join(GOLDEN, "drift_handworked.json")))["cases"]
    for c in cases:
        out, _ = orc.drift_segment(_h(c["h"]), np.asarray(c["a"], np.float32))
        assert out[0] == pytest.approx(c["rel_l2"], rel=1e-14, abs=1e-300)
        assert out[1] == c["max_abs"]
        assert out[2] == pytest.approx(c["cos_dev"], rel=1e-13, abs=1e-15)


def test_drift_closed_forms(orc):
    rng = np.random.Generator(np.random.PCG64(3))
    a16 = rng.standard_normal(4096).astype(np.float16)          # fp16-exact reference
    a = a16.astype(np.float32)
    # h = a: every statistic is zero
    out, _ = orc.drift_segment(a16.view(np.uint16), a)
    assert list(out) == [0.0, 0.0, 0.0]
    # h = 2a (exact in fp16 here): m = 1, cosine 0
    out, _ = orc.drift_segment((2 * a16).view(np.uint16), a)
    assert out[0] == pytest.approx(1.0, rel=1e-14) and out[2] == pytest.approx(0.0, abs=1e-15)
    # h = -a: m = 2, cosine deviation 2
    out, _ = orc.drift_segment((-a16).view(np.uint16), a)
    assert out[0] == pytest.approx(2.0, rel=1e-14) and out[2] == pytest.approx(2.0, rel=1e-14)
    assert out[1] == 2 * np.abs(a).max()
    # zero reference: m = 0 when h = 0, +inf otherwise; cosine defined as 0
    z = np.zeros(16, np.float32)
    out, _ = orc.drift_segment(_h(np.zeros(16)), z)
    assert list(out) == [0.0, 0.0, 0.0]
    out, _ = orc.drift_segment(_h(np.ones(16)), z)
    assert out[0] == math.inf and out[1] == 1.0 and out[2] == 0.0
    # zero live tensor against a nonzero reference: m = 1, cosine 0 by convention
    out, _ = orc.drift_segment(_h(np.zeros(16)), np.ones(16, np.float32))
    assert out[0] == 1.0 and out[2] == 0.0


def test_drift_matches_numpy_norms(orc):
    """Random segments: Eq. 4 and the cosine mismatch via numpy's fp64 routines."""
    import seeded_inputs as SI
    acts, refs = SI.drift_arrays(3, 5, 1000, seed=11)
    for s in range(3):
        for n in range(5):
            h = acts[s, n].view(np.float16).astype(np.float64)
            a = refs[s, n].astype(np.float64)
            out, sums = orc.drift_segment(acts[s, n], refs[s, n])
            na, nh = np.linalg.norm(a), np.linalg.norm(h)
            nd = np.linalg.norm(h - a)
            if na > 0:
                assert out[0] == pytest.approx(nd / na, rel=1e-12)
            assert out[1] == (np.abs(h - a).max() if h.size else 0.0)
            if na > 0 and nh > 0:
                cos = float(np.dot(h, a)) / (nh * na)
                # 1 - cos loses digits near cos = 1; compare to its own precision
                assert out[2] == pytest.approx(1.0 - cos, abs=1e-12)
                assert sums[0] == pytest.approx(nd * nd, rel=1e-12)


def test_drift_scores_layout(orc):
    """scores[stat][n][s] of segment (s, n) of acts [S][N][L]."""
    import seeded_inputs as SI
    S, N, L = 3, 4, 37
    acts, refs = SI.drift_arrays(S, N, L, seed=5)
    sc = orc.drift_scores(acts, refs, S, N)
    for s in range(S):
        for n in range(N):
            out, _ = orc.drift_segment(acts[s, n], refs[s, n])
            assert list(sc[:, n, s]) == list(out)


def test_drift_nan_propagates(orc):
    h = _h([1.0, float("nan"), 2.0])
    a = np.array([1.0, 1.0, 1.0], np.float32)
    out, _ = orc.drift_segment(h, a)
    assert math.isnan(out[0]) and math.isnan(out[2]) and out[1] == 1.0
