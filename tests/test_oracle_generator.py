"""Pins of the oracle's synthetic pipeline generator (not the GPU).

The generator simulates Eq. 2 (benign stages) and Eq. 3 with the three tamper
strategies of Sec. 3.2 at every hop.  Its pins are the constructions' exact
properties (the Gaussian tamper has relative norm exactly eps before fp16
rounding, the rescale has mismatch exactly |beta - 1|, the sign flip exactly
2, a channel flip 2 sqrt(sum_C a^2 / sum a^2)), numpy's fp16 rounding of the
pre-rounding values, the counter layout of every element, and the expected
magnitudes of benign drift (m_benign = O(sigma_hw), Sec. 3.4).
"""
import math

import numpy as np
import pytest

import seeded_inputs as SI


def desc(orc, **kw):
    base = dict(n_shards=4, hidden=64, n_canaries=3, tokens=8, malicious=(1,),
                noise=orc.NOISE_PAPER, benign_sigma=1e-3, tamper=orc.TAMPER_ADDITIVE,
                tamper_param=0.05, seed=123, config_id=7)
    base.update(kw)
    return orc.make_desc(**base)


def rel(pre, a):
    a = a.astype(np.float64)
    return np.linalg.norm(pre - a) / np.linalg.norm(a)


def test_reference_counter_layout(orc):
    """Reference element e of segment (s, n) is normal e of stream
    (c1 = s*N + n, c2 = 4*config_id + 0), times the outlier scale on outlier channels."""
    D = desc(orc, n_outlier=3, outlier_scale=20.0)
    outl, _, _ = orc.config_tables(D)
    assert len(set(outl.tolist())) == 3 and outl.max() < 64
    L = 8 * 64
    for s, n in [(0, 0), (2, 1), (3, 2)]:
        refs, _, _, _ = orc.generate_segment(D, s, n)
        z = orc.philox_normals(123, s * 3 + n, 4 * 7 + 0, 0, 0, L // 4)
        scale = np.ones(L)
        scale[np.isin(np.arange(L) % 64, outl)] = np.float32(20.0)
        assert np.array_equal(refs, (z * scale).astype(np.float32))


def test_outlier_channels_are_the_first_distinct_draws(orc):
    D = desc(orc, n_outlier=5)
    outl, _, _ = orc.config_tables(D)
    draws = orc.aux_bounded(123, orc.AUX_OUTLIER, 0, 7, 64, 40)
    firsts = []
    for v in draws:
        if v not in firsts:
            firsts.append(int(v))
    assert outl.tolist() == firsts[:5]


def test_mult_noise_construction(orc):
    D = desc(orc, noise=orc.NOISE_MULT, benign_sigma=1e-3)
    refs, pre, acts, coef = orc.generate_segment(D, 2, 1)
    z = orc.philox_normals(123, 2 * 3 + 1, 4 * 7 + 1, 0, 0, refs.size // 4)
    sig = float(np.float32(1e-3))
    assert np.allclose(pre, refs.astype(np.float64) * (1.0 + sig * z), rtol=0, atol=1e-15)
    assert np.array_equal(acts, pre.astype(np.float16).view(np.uint16))
    assert coef == 0.0


def test_paper_noise_construction(orc):
    """Eq. 2: delta ~ N(0, sigma^2 mu^2), mu = ||a||_1 / (T d)."""
    D = desc(orc, benign_sigma=2e-3)
    refs, pre, acts, coef = orc.generate_segment(D, 0, 2)
    mu = np.abs(refs.astype(np.float64)).mean()
    sig = float(np.float32(2e-3))
    assert coef == pytest.approx(sig * mu, rel=1e-13)
    z = orc.philox_normals(123, 0 * 3 + 2, 4 * 7 + 1, 0, 0, refs.size // 4)
    assert np.allclose(pre - refs.astype(np.float64), coef * z, rtol=0, atol=1e-14)
    assert np.array_equal(acts, pre.astype(np.float16).view(np.uint16))


def test_benign_drift_magnitude(orc):
    """m_benign = O(sigma_hw) (Sec. 3.4): about sigma for the relative noise,
    sigma * mean|a| / rms(a) = sigma sqrt(2/pi) for Eq. 2 without outliers."""
    for noise, expect in [(orc.NOISE_MULT, 1.0), (orc.NOISE_PAPER, math.sqrt(2 / math.pi))]:
        D = desc(orc, hidden=1024, tokens=64, noise=noise, benign_sigma=1e-2)
        refs, pre, _, _ = orc.generate_segment(D, 0, 0)
        assert rel(pre, refs) == pytest.approx(1e-2 * expect, rel=0.03)


def test_gaussian_tamper_exact_norm(orc):
    """tau(v) = v + eps ||v|| U, U = g/||g||: relative norm exactly eps."""
    for eps in (1e-3, 0.02, 0.05, 0.2):
        D = desc(orc, tamper_param=eps)
        refs, pre, acts, coef = orc.generate_segment(D, 1, 2)
        e = float(np.float32(eps))
        assert rel(pre, refs) == pytest.approx(e, rel=1e-12)
        g = orc.philox_normals(123, 1 * 3 + 2, 4 * 7 + 2, 0, 0, refs.size // 4)
        d = pre - refs.astype(np.float64)
        assert np.allclose(d / np.linalg.norm(d), g / np.linalg.norm(g), atol=1e-12)
        assert np.array_equal(acts, pre.astype(np.float16).view(np.uint16))


def test_sign_flip_and_rescale(orc):
    D = desc(orc, tamper=orc.TAMPER_SIGNFLIP_FULL)
    refs, pre, _, _ = orc.generate_segment(D, 1, 0)
    assert np.array_equal(pre, -refs.astype(np.float64))
    assert rel(pre, refs) == pytest.approx(2.0, rel=1e-15)
    for beta in (1.05, 1.10):
        D = desc(orc, tamper=orc.TAMPER_SCALE, tamper_param=beta)
        refs, pre, _, _ = orc.generate_segment(D, 1, 0)
        b = float(np.float32(beta))
        assert rel(pre, refs) == pytest.approx(abs(b - 1.0), rel=1e-12)


@pytest.mark.parametrize("p,d", [(0.01, 64), (0.01, 8192), (0.1, 1024), (1e-3, 1024), (0.5, 64)])
def test_channel_flip(orc, p, d):
    D = desc(orc, hidden=d, tokens=2, tamper=orc.TAMPER_SIGNFLIP_CHANNELS, tamper_param=p)
    _, _, flip = orc.config_tables(D)
    nf = max(1, int(math.floor(float(np.float32(p)) * d + 0.5)))
    assert flip[1].sum() == nf and flip[[0, 2, 3]].sum() == 0
    refs, pre, _, _ = orc.generate_segment(D, 1, 0)
    a = refs.astype(np.float64).reshape(2, d)
    mask = flip[1]
    assert np.array_equal(pre.reshape(2, d), np.where(mask, -a, a))
    assert rel(pre, refs) == pytest.approx(2 * math.sqrt((a[:, mask] ** 2).sum() / (a ** 2).sum()), rel=1e-12)


def test_malicious_stage_has_no_benign_noise(orc):
    D = desc(orc, tamper=orc.TAMPER_SCALE, tamper_param=1.05, benign_sigma=0.1)
    refs, pre, _, _ = orc.generate_segment(D, 1, 0)
    assert np.array_equal(pre, float(np.float32(1.05)) * refs.astype(np.float64))


def test_lognormal_stage_sigma(orc):
    """sigma_s = sigma exp(0.5 z_s): over many configurations log(sigma_s/sigma) ~ N(0, 0.25)."""
    logs = []
    for cid in range(400):
        D = desc(orc, n_shards=8, shard_sigma_lognormal=0.5, benign_sigma=1e-3, config_id=cid)
        _, sig, _ = orc.config_tables(D)
        logs += list(np.log(sig / float(np.float32(1e-3))))
    logs = np.array(logs)
    assert abs(logs.mean()) < 5 * 0.5 / math.sqrt(logs.size)
    assert logs.std() == pytest.approx(0.5, rel=0.05)
    D = desc(orc, n_shards=8)
    _, sig, _ = orc.config_tables(D)
    assert np.all(sig == float(np.float32(1e-3)))


def test_pipeline_matches_segments_and_labels(orc):
    D = desc(orc, malicious=(0, 3), n_outlier=2)
    acts, refs, labels = orc.generate_pipeline(D)
    assert labels.tolist() == [[1, 0, 0, 1]] * 3
    for s in range(4):
        for n in range(3):
            r, _, a, _ = orc.generate_segment(D, s, n)
            assert np.array_equal(refs[s, n], r) and np.array_equal(acts[s, n], a)


def test_bad_descriptions_rejected(orc):
    from oracle.oracle import OracleError
    for kw in [dict(malicious=(4,)), dict(malicious=(0, 1, 2, 3)), dict(malicious=(1, 1)),
               dict(n_outlier=65), dict(tamper=9), dict(tamper=1, tamper_param=0.0),
               dict(config_id=2**30)]:
        with pytest.raises(OracleError):
            orc.generate_segment(desc(orc, **kw), 0, 0)


def test_tiny_pipeline_detects(orc):
    """Full detector on the tiny pipeline: A-hat = 1 (Table 1, 'Full detector')."""
    import json, os
    paper = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_values.json")))
    D = orc.desc_from_dict(SI.TINY)
    acts, refs, labels = orc.generate_pipeline(D)
    sc = orc.drift_scores(acts, refs, 4, 16)
    res = orc.auroc(sc[0][None].astype(np.float32), labels[None])
    assert res["auroc"][0] == paper["full_detector_auroc"]["value"]
    # the malicious stage's mismatch tracks eps, the benign floor tracks sigma (Sec. 3.4)
    assert np.allclose(sc[0][:, 1], 0.05, rtol=0.02)
    assert sc[0][:, [0, 2, 3]].max() < 3e-3


def test_segment_ranges_equal_pipeline_slices(orc):
    """generate_segments / generate_stage return exactly the matching slice of
    the whole pipeline (the full-size GPU tests compare one stage at a time),
    and each segment's scalar as generate_segment gives it."""
    from oracle.oracle import OracleError
    for tamper, noise in [(SI.TAMPER_ADDITIVE, SI.NOISE_PAPER), (SI.TAMPER_SCALE, SI.NOISE_MULT)]:
        cfg = SI.shrink(SI.SEVEN_B, n_shards=3, hidden=24, n_canaries=5, tokens=3, malicious=(1,),
                        tamper=tamper, tamper_param=0.05 if tamper == SI.TAMPER_ADDITIVE else 1.1,
                        noise=noise)
        D = orc.desc_from_dict(cfg)
        acts, refs, _ = orc.generate_pipeline(D)
        for s in range(3):
            a, r, c = orc.generate_stage(D, s)
            assert np.array_equal(a, acts[s]) and np.array_equal(r, refs[s])
            for n in range(5):
                assert c[n] == orc.generate_segment(D, s, n)[3]
        a, r, c = orc.generate_segments(D, 4, 7)      # crosses the stage 0 / stage 1 boundary
        assert np.array_equal(a, acts.reshape(15, -1)[4:11])
        assert np.array_equal(r, refs.reshape(15, -1)[4:11])
        a, r, c = orc.generate_coefs(D)
        assert np.array_equal(a, acts) and np.array_equal(r, refs) and c.shape == (3, 5)
        with pytest.raises(OracleError):
            orc.generate_segments(D, 10, 6)
