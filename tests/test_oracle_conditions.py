"""Pins of the oracle's reference conditions (Sec. 4.5) and the
noisy-reference ablation (Sec. 4.4), not the GPU.

Random baseline: each score is the top 24 bits of one Philox word scaled by
2^-24 (checked word by word), E[A-hat] = 0.5 with Var = (S+1)/(12(S-1)N).
Recompute: replica 0 reproduces the live benign draw exactly; a replica r
draws its noise from counter word c3 = r; against an independent replica a
benign stage's mismatch is sqrt(2) times its live mismatch against the clean
reference, and the full detector's ceiling is 1.000 (Table 1, 'Ceil.')."""
import json
import math
import os

import numpy as np
import pytest

import seeded_inputs as SI

PAPER = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_values.json")))


def test_random_scores_are_philox_words(orc):
    sc = orc.random_scores(77, 3, 5, 6, config_id0=10)
    for c in range(3):
        for n in range(5):
            w = orc.philox_words(77, (orc.AUX_RANDOM << 24) | n, 4 * (10 + c) + 3, 0, 0, 2)
            expect = (w[:6] >> 8).astype(np.float64) * 2.0 ** -24
            assert np.array_equal(sc[c, n].astype(np.float64), expect)


def test_random_baseline_auroc(orc):
    S, N, R = 4, 100, 300
    sc = orc.random_scores(5, R, N, S)
    labels = np.zeros((R, N, S), np.int8)
    labels[:, :, 2] = 1
    A = orc.auroc(sc, labels)["auroc"]
    sd = math.sqrt((S + 1) / (12 * (S - 1) * N))
    assert abs(A.mean() - PAPER["random_baseline"]["mean"]) < 5 * sd / math.sqrt(R)
    assert A.std() == pytest.approx(sd, rel=0.15)


def _desc(orc, **kw):
    cfg = SI.shrink(SI.PAPER_SHAPE, n_canaries=6, tokens=8, **kw)
    return cfg, orc.desc_from_dict(cfg)


def test_recompute_replica0_is_live_draw(orc):
    cfg, D = _desc(orc)
    acts, refs, labels = orc.generate_pipeline(D)
    rec = orc.generate_recompute(D, 0)
    live = acts.view(np.float16).astype(np.float32)
    benign = [s for s in range(cfg["n_shards"]) if s not in cfg["malicious"]]
    assert np.array_equal(rec[benign], live[benign])
    mal = cfg["malicious"][0]
    assert not np.array_equal(rec[mal], live[mal])      # the recompute is honest


def test_recompute_replica_noise_counter(orc):
    cfg, D = _desc(orc, noise=orc.NOISE_MULT)
    rec = orc.generate_recompute(D, 3)
    _, _, _, _ = orc.generate_segment(D, 2, 1)
    refs, _, _, _ = orc.generate_segment(D, 2, 1)
    L = refs.size
    z = orc.philox_normals(cfg["seed"], 2 * 6 + 1, 4 * cfg["config_id"] + 1, 3, 0, L // 4)
    sig = float(np.float32(cfg["benign_sigma"]))
    expect = (refs.astype(np.float64) * (1.0 + sig * z)).astype(np.float16).astype(np.float32)
    assert np.array_equal(rec[2, 1], expect)


def test_recompute_mismatch_scale_and_ceiling(orc):
    """Benign: m(live, recompute) ~ sqrt(2) m(live, clean reference); the
    malicious stage still stands out, so the ceiling's A-hat is 1."""
    cfg = SI.shrink(SI.PAPER_SHAPE, n_canaries=8, tokens=16)
    D = orc.desc_from_dict(cfg)
    acts, refs, labels = orc.generate_pipeline(D)
    rec = orc.generate_recompute(D, 1)
    S, N = cfg["n_shards"], cfg["n_canaries"]
    clean = orc.drift_scores(acts, refs, S, N)[0]
    noisy = orc.drift_scores(acts, rec, S, N)[0]
    benign = [s for s in range(S) if s not in cfg["malicious"]]
    ratio = noisy[:, benign].mean() / clean[:, benign].mean()
    assert ratio == pytest.approx(math.sqrt(2), rel=0.05)
    A = orc.auroc(noisy.astype(np.float32)[None], labels[None])["auroc"][0]
    assert A == PAPER["full_detector_auroc"]["value"]
