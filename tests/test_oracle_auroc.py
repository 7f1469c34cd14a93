"""Pins of the oracle's ranking test (Eq. 5, Eq. 6) and the scrambled-label
control (Sec. 4.5), not the GPU.

The counts are checked against an independent pure-Python pair count and
scipy's Mann-Whitney U; A-hat against exact rational arithmetic (fractions);
plus the invariants of a rank statistic and the expectations of the random
baseline and the control, whose printed ranges are in
tests/golden/paper_values.json.
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import seeded_inputs as SI

PAPER = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_values.json")))


def brute(scores, labels):
    C, N, S = scores.shape
    u2 = np.zeros((C, N), np.int64)
    A = []
    for c in range(C):
        terms = []
        for n in range(N):
            m, l = scores[c, n].tolist(), labels[c, n].tolist()
            mal = [m[i] for i in range(S) if l[i] == 1]
            ben = [m[j] for j in range(S) if l[j] == 0]
            u = sum(2 if x > y else (1 if x == y else 0) for x in mal for y in ben)
            u2[c, n] = u
            if mal and ben:
                terms.append(Fraction(u, 2 * len(mal) * len(ben)))
        A.append(sum(terms) / len(terms) if terms else None)
    return u2, A


@pytest.mark.parametrize("n_mal,excluded,ties", [(1, 0, None), (1, 0, 3), (2, 1, 4), (3, 0, 2)])
def test_counts_match_pair_enumeration(orc, n_mal, excluded, ties):
    scores, labels = SI.score_arrays(4, 9, 7, seed=n_mal * 10 + excluded, n_malicious=n_mal,
                                     tie_levels=ties, excluded=excluded)
    res = orc.auroc(scores, labels)
    u2, A = brute(scores, labels)
    assert np.array_equal(res["u2"], u2)
    assert np.array_equal(res["u2"], 2 * res["gt"] + res["eq"])
    for c in range(4):
        assert res["auroc"][c] == float(A[c])   # correctly rounded exact mean


def test_nonuniform_pair_counts(orc):
    scores, labels = SI.score_arrays(3, 6, 9, seed=4, n_malicious=2, tie_levels=5)
    labels[:, ::2, 8] = -1           # some canaries lose a benign stage
    labels[1, 3, :] = 0              # one canary with no malicious stage: skipped
    res = orc.auroc(scores, labels)
    u2, A = brute(scores, labels)
    assert np.array_equal(res["u2"], u2)
    for c in range(3):
        assert res["auroc"][c] == pytest.approx(float(A[c]), rel=4e-16)


def test_matches_scipy_mannwhitney(orc):
    stats = pytest.importorskip("scipy.stats")
    rng = np.random.Generator(np.random.PCG64(8))
    for _ in range(20):
        S = int(rng.integers(3, 33))
        c = int(rng.integers(1, S))
        m = (rng.integers(0, 6, size=S) / 4).astype(np.float32)
        lab = np.zeros(S, np.int8)
        lab[rng.permutation(S)[:c]] = 1
        res = orc.auroc(m[None, None], lab[None, None])
        U = stats.mannwhitneyu(m[lab == 1], m[lab == 0], alternative="two-sided").statistic
        assert res["u2"][0, 0] == round(2 * U)


def test_invariants(orc):
    scores, labels = SI.score_arrays(5, 8, 6, seed=2, n_malicious=2)
    base = orc.auroc(scores, labels)["auroc"]
    # separated: every malicious above every benign -> 1, below -> 0
    sep = np.where(labels == 1, scores + 2.0, scores).astype(np.float32)
    assert np.all(orc.auroc(sep, labels)["auroc"] == 1.0)
    sep = np.where(labels == 1, scores - 2.0, scores).astype(np.float32)
    assert np.all(orc.auroc(sep, labels)["auroc"] == 0.0)
    # all equal -> 0.5
    assert np.all(orc.auroc(np.ones_like(scores), labels)["auroc"] == 0.5)
    # AUROC(-s) = 1 - AUROC(s), exactly (uniform pair counts)
    neg = orc.auroc(-scores, labels)
    assert np.array_equal(neg["u2"], 2 * (2 * 4) - orc.auroc(scores, labels)["u2"])   # 2c(S-c) - 2U
    assert np.all(neg["auroc"] == 1.0 - base)
    # strictly increasing transform and a permutation of stages leave it unchanged
    assert np.array_equal(orc.auroc(np.exp(3 * scores).astype(np.float32), labels)["auroc"], base)
    perm = np.random.Generator(np.random.PCG64(0)).permutation(6)
    assert np.array_equal(orc.auroc(scores[:, :, perm], labels[:, :, perm])["auroc"], base)


def test_single_malicious_is_eq5(orc):
    """c = 1 and no ties: A^(t) is the fraction of benign stages ranked below (Eq. 5)."""
    scores, labels = SI.score_arrays(1, 1, 10, seed=3)
    res = orc.auroc(scores, labels)
    m, l = scores[0, 0], labels[0, 0]
    i = int(np.flatnonzero(l == 1)[0])
    expect = sum(m[i] > m[j] for j in range(10) if j != i) / 9
    assert res["auroc"][0] == expect


def test_nan_score_is_an_error(orc):
    from oracle.oracle import OracleError
    scores, labels = SI.score_arrays(1, 2, 4, seed=0)
    scores[0, 1, 2] = np.nan
    with pytest.raises(OracleError):
        orc.auroc(scores, labels)


def test_random_baseline_distribution(orc):
    """Uniform(0,1) scores (Sec. 4.5): E[A-hat] = 0.5 and, with c = 1 and no
    ties, A^(t) is uniform on {0, 1/(S-1), ..., 1}, so Var[A-hat] =
    (S+1) / (12 (S-1) N).  For S = 4, N = 100 this is sd 0.037, in line with
    the printed range of the random baseline."""
    S, N, R = 4, 100, 400
    scores, labels = SI.score_arrays(R, N, S, seed=99)
    A = orc.auroc(scores, labels)["auroc"]
    sd = math.sqrt((S + 1) / (12 * (S - 1) * N))
    assert abs(A.mean() - PAPER["random_baseline"]["mean"]) < 5 * sd / math.sqrt(R)
    assert A.std() == pytest.approx(sd, rel=0.15)
    lo, hi = PAPER["random_baseline"]["range"]
    assert 0.5 - lo < 3 * sd and hi - 0.5 < 3 * sd


def test_control_labels_structure(orc):
    labels = np.zeros((3, 50, 8), np.int8)
    labels[:, :, 3] = 1
    labels[2, :, 5] = 1
    ctrl = orc.control_labels(labels, seed=17, config_id0=40)
    assert np.all((ctrl == 1).sum(axis=2) == 1)
    assert np.all(ctrl[labels == 1] == -1)
    assert np.all(ctrl[labels == 0] >= 0)
    # j* is the r-th benign stage, r the first bounded draw of the canary's stream
    for c in range(3):
        benign = [s for s in range(8) if labels[c, 0, s] == 0]
        for n in range(50):
            r = orc.aux_bounded(17, orc.AUX_CONTROL, n, 40 + c, len(benign), 1)[0]
            assert ctrl[c, n, benign[r]] == 1


def test_control_uniform_over_benign(orc):
    labels = np.zeros((1, 7000, 8), np.int8)
    labels[0, :, 2] = 1
    ctrl = orc.control_labels(labels, seed=5)
    js = np.argmax(ctrl[0] == 1, axis=1)
    counts = np.bincount(js, minlength=8)
    assert counts[2] == 0
    exp = 7000 / 7
    assert ((counts[counts > 0] - exp) ** 2 / exp).sum() < 6 + 8 * math.sqrt(12)


def test_control_auroc_near_half(orc):
    """On real mismatches the scrambled control collapses to chance (Sec. 5)."""
    D = orc.desc_from_dict(SI.shrink(SI.TINY, n_canaries=64, hidden=128, tokens=16))
    acts, refs, labels = orc.generate_pipeline(D)
    sc = orc.drift_scores(acts, refs, 4, 64)[0].astype(np.float32)
    vals = []
    for cid in range(40):
        ctrl = orc.control_labels(labels[None], seed=1000 + cid)
        vals.append(orc.auroc(sc[None], ctrl)["auroc"][0])
    lo, hi = PAPER["control_acceptance"]["interval"]
    assert lo <= float(np.mean(vals)) <= hi
    assert orc.auroc(sc[None], labels[None])["auroc"][0] == 1.0


# --------------------------------------------------------------------------
# Pooled Mann-Whitney (all canaries of a configuration in one pool)

def test_pooled_matches_scipy_and_pairs(orc):
    stats = pytest.importorskip("scipy.stats")
    for seed, ties, nm, ex in [(1, None, 1, 0), (2, 4, 2, 1), (3, 3, 3, 0)]:
        scores, labels = SI.score_arrays(3, 11, 7, seed=seed, n_malicious=nm, tie_levels=ties,
                                         excluded=ex)
        res = orc.auroc_pooled(scores, labels)
        for c in range(3):
            m, l = scores[c].ravel(), labels[c].ravel()
            U = stats.mannwhitneyu(m[l == 1], m[l == 0], alternative="two-sided").statistic
            assert res["u2"][c] == round(2 * U)
            assert res["n_mal"][c] == (l == 1).sum() and res["n_ben"][c] == (l == 0).sum()
            exact = Fraction(int(res["u2"][c]), 2 * int(res["n_mal"][c]) * int(res["n_ben"][c]))
            assert res["auroc"][c] == float(exact)


def test_pooled_equals_per_canary_when_one_canary(orc):
    scores, labels = SI.score_arrays(4, 1, 9, seed=8, n_malicious=2, tie_levels=3)
    assert np.array_equal(orc.auroc_pooled(scores, labels)["u2"],
                          orc.auroc(scores, labels)["u2"][:, 0])


def test_pooled_invariants(orc):
    scores, labels = SI.score_arrays(3, 5, 6, seed=4, n_malicious=1)
    base = orc.auroc_pooled(scores, labels)
    neg = orc.auroc_pooled(-scores, labels)
    assert np.array_equal(neg["u2"], 2 * base["n_mal"] * base["n_ben"] - base["u2"])
    assert np.allclose(neg["auroc"], 1.0 - base["auroc"], rtol=0, atol=1e-15)
    sep = np.where(labels == 1, scores + 2.0, scores).astype(np.float32)
    assert np.all(orc.auroc_pooled(sep, labels)["auroc"] == 1.0)
    nan = scores.copy()
    nan[0, 0, 0] = np.nan
    with pytest.raises(Exception):
        orc.auroc_pooled(nan, labels)
