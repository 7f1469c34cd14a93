"""Pins of the oracle's propagating pipeline (Eq. 2 recursion with the
block's response to an upstream deviation linearised as a gain), not the GPU.

gain = 0 reproduces the hop-local pipeline byte for byte; a stage after the
first inherits gain x the previous stage's fp16 deviation (checked element by
element for a sign flip, where tau is exact); benign deviations accumulate
like a geometric series, sigma^2 (1 + g^2 + g^4 + ...) in the mismatch
squared; with gain < 1 the tamper origin keeps the largest mismatch."""
import math

import numpy as np
import pytest

import seeded_inputs as SI


def cfg(**kw):
    base = SI.shrink(SI.PAPER_SHAPE, n_canaries=4, tokens=8, hidden=256)
    base.update(kw)
    return base


def test_gain_zero_is_hop_local(orc):
    c = cfg()
    D = orc.desc_from_dict(c)
    a0, r0, _ = orc.generate_pipeline(D)
    a1, r1 = orc.generate_propagating(D, 0.0)
    assert np.array_equal(a0, a1) and np.array_equal(r0, r1)


def test_sign_flip_inherits_scaled_deviation(orc):
    """Stage i* = 5 negates v = a + g (h_4 - a_4); check h_5 = fp16(-v) exactly."""
    c = cfg(tamper=SI.TAMPER_SIGNFLIP_FULL)
    D = orc.desc_from_dict(c)
    g = 0.5
    acts, refs = orc.generate_propagating(D, g)
    h4 = acts[4].view(np.float16).astype(np.float64)
    v5 = refs[5].astype(np.float64) + float(np.float32(g)) * (h4 - refs[4].astype(np.float64))
    assert np.array_equal(acts[5], (-v5).astype(np.float16).view(np.uint16))


def test_benign_deviation_accumulates(orc):
    """With Eq. 2 noise at sigma and gain g on every stage, stage s's mismatch
    squared tends to sigma_eff^2 (1 - g^(2(s+1))) / (1 - g^2)."""
    c = cfg(malicious=(), benign_sigma=1e-2, hidden=1024, tokens=16, n_canaries=2)
    D = orc.desc_from_dict(c)
    g = 0.8
    acts, refs = orc.generate_propagating(D, g)
    S = c["n_shards"]
    m = orc.drift_scores(acts, refs, S, 2)[0].mean(axis=0)
    base = m[0]
    for s in (3, 7, 11):
        expect = base * math.sqrt((1 - g ** (2 * (s + 1))) / (1 - g * g))
        assert m[s] == pytest.approx(expect, rel=0.05)


def test_attenuating_blocks_keep_origin_highest(orc):
    """gain < 1: downstream stages carry gain^k of the tamper, so the tampering
    stage keeps the largest mismatch and A-hat = 1; with gain > 1 it does not."""
    for g, expect_one in [(0.5, True), (1.5, False)]:
        c = cfg(malicious=(3,), tamper_param=0.05)
        D = orc.desc_from_dict(c)
        acts, refs = orc.generate_propagating(D, g)
        sc = orc.drift_scores(acts, refs, c["n_shards"], c["n_canaries"])[0].astype(np.float32)
        labels = np.zeros((c["n_canaries"], c["n_shards"]), np.int8)
        labels[:, 3] = 1
        A = orc.auroc(sc[None], labels[None])["auroc"][0]
        assert (A == 1.0) == expect_one, (g, A)
