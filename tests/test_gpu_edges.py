"""Edge cases and maximum sizes of the boundary on the GPU, against the oracle:
the largest stage count (1024) with almost every stage colluding, the
largest outlier count, a 65,536-wide hidden size with half the channels
flipped, single-element segments, a single segment of 2^32 + 8 elements, and
the degenerate ranking cases (no pair, one stage, all scores equal)."""
import numpy as np
import pytest

import seeded_inputs as SI
from tests._cmp import assert_live_close, assert_normals_close, half_ulp_distance

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cg():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_19490_gb300 as m
    m.build()
    return m


def compare(cg, orc, cfg):
    acts, refs, labels = cg.cg_generate_pipeline(cg.PipelineDesc.from_config(cfg))
    D = orc.desc_from_dict(cfg)
    _, _, o_labels = orc.generate_pipeline(D)
    o_acts, o_refs, o_coef = orc.generate_coefs(D)
    assert np.array_equal(labels.cpu().numpy(), o_labels)
    g_refs = refs.cpu().numpy()
    assert_normals_close(g_refs, o_refs, what="references")
    assert_live_close(acts.cpu().numpy().view(np.uint16), o_acts, g_refs, o_refs, o_coef)
    return acts, refs, labels


@pytest.mark.parametrize("cfg", [
    SI.shrink(SI.TINY, n_shards=1024, hidden=8, tokens=2, n_canaries=2, n_outlier=1,
              malicious=tuple(range(1023)), noise=SI.NOISE_PAPER),
    SI.shrink(SI.TINY, hidden=512, tokens=2, n_outlier=256),
    SI.shrink(SI.TINY, n_shards=2, hidden=65536, tokens=1, n_canaries=1, malicious=(1,),
              tamper=SI.TAMPER_SIGNFLIP_CHANNELS, tamper_param=0.5),
    SI.shrink(SI.TINY, hidden=1, tokens=1, n_canaries=3, n_outlier=0),
], ids=["1024_stages_1023_colluding", "256_outliers", "d65536_half_flipped", "one_element"])
def test_generator_extremes(cg, orc, cfg):
    compare(cg, orc, cfg)


def test_extreme_pipeline_ranks(cg, orc):
    """1024 stages, 1023 colluders: each canary has 1023 x 1 pairs."""
    import torch
    cfg = SI.shrink(SI.TINY, n_shards=1024, hidden=8, tokens=2, n_canaries=2, n_outlier=1,
                    malicious=tuple(range(1023)), noise=SI.NOISE_PAPER)
    acts, refs, labels = cg.cg_generate_pipeline(cg.PipelineDesc.from_config(cfg))
    sc = cg.cg_drift_scores(acts, refs, 1024, 2)
    res = cg.cg_auroc(sc[0][None].contiguous(), labels[None])
    o = orc.auroc(sc[0].cpu().numpy()[None], labels.cpu().numpy()[None])
    assert np.array_equal(res["u2"].cpu().numpy(), o["u2"])
    assert res["auroc"].item() == o["auroc"][0]


def test_degenerate_rankings(cg, orc):
    import torch
    scores = np.array([[[0.3, 0.3, 0.3, 0.3]], [[0.1, 0.2, 0.3, 0.4]], [[0.5, 0.5, 0.5, 0.5]]],
                      np.float32)
    labels = np.array([[[0, 0, 0, 0]], [[-1, -1, 1, -1]], [[1, 0, 0, 0]]], np.int8)
    g = cg.cg_auroc(torch.from_numpy(scores).cuda(), torch.from_numpy(labels).cuda())
    A = g["auroc"].cpu().numpy()
    assert np.isnan(A[0]) and np.isnan(A[1]) and A[2] == 0.5
    o = orc.auroc(scores, labels)
    assert np.array_equal(g["u2"].cpu().numpy(), o["u2"])
    one = cg.cg_auroc(torch.ones((2, 3, 1), device="cuda"),
                      torch.ones((2, 3, 1), dtype=torch.int8, device="cuda"))
    assert np.isnan(one["auroc"].cpu().numpy()).all()


def test_segment_beyond_2_32_elements(cg, orc):
    """One (stage, canary) segment of 2^32 + 8 elements (25.8 GB on the
    device), so element offsets inside a segment pass 32 bits.
    Sampled references and live values on both sides of element 2^32 match
    the oracle's Philox and Box-Muller one by one.  Then a planted
    construction with an exact closed form checks the drift scores of the
    streaming and the TMA kernels: a constant reference of 1, live values 1
    except 1.5 at elements 3 and 2^32 + 5 and 0.75 at 2^31 + 1."""
    import torch
    free, _ = torch.cuda.mem_get_info()
    if free < 32 * 2**30:
        pytest.skip("needs 32 GB of free device memory")
    L = 2**32 + 8
    sigma, seed = 1e-3, 11
    cfg = SI.shrink(SI.TINY, n_shards=1, malicious=(), n_canaries=1, hidden=8, tokens=L // 8,
                    n_outlier=0, noise=SI.NOISE_MULT, benign_sigma=sigma, seed=seed, config_id=0)
    acts, refs, _ = cg.cg_generate_pipeline(cg.PipelineDesc.from_config(cfg))
    a_flat, h_flat = refs.view(-1), acts.view(-1)
    for e in (0, 1, 4095, 2**31 + 3, 2**32 - 5, 2**32 - 1, 2**32, 2**32 + 3, L - 1):
        q, k = e // 4, e % 4
        z = orc.philox_normals(seed, 0, 0, 0, q, 1)[k]           # reference stream
        n = orc.philox_normals(seed, 0, 1, 0, q, 1)[k]           # benign-noise stream
        a_gpu = float(a_flat[e].item())
        assert abs(a_gpu - z) <= 2.0**-20 * max(abs(z), 2.0**-6), (e, a_gpu, z)
        h_bits = int(h_flat[e:e + 1].view(torch.int16).item()) & 0xFFFF
        o_bits = orc.half_from_double(np.float64(np.float32(z)) * (1.0 + np.float64(np.float32(sigma)) * n))
        assert half_ulp_distance(np.array([h_bits], np.uint16), np.array([o_bits], np.uint16))[0] <= 1, e
    # the benign floor of Eq. 2's relative form over the whole segment
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    s1 = cg.cg_drift_scores(acts, refs, 1, 1, algo=1, status=st).cpu().numpy()
    s2 = cg.cg_drift_scores(acts, refs, 1, 1, algo=2, status=st).cpu().numpy()
    assert cg.cg_read_status(st) == (0, 0)
    assert 0.9 * sigma < s1[0, 0, 0] < 1.2 * sigma
    assert abs(s1[0, 0, 0] - s2[0, 0, 0]) <= 2e-5 * s1[0, 0, 0]
    assert s1[1, 0, 0] == s2[1, 0, 0]
    # planted construction
    refs.fill_(1.0)
    acts.fill_(1.0)
    h_flat[3] = 1.5
    h_flat[2**32 + 5] = 1.5
    h_flat[2**31 + 1] = 0.75
    D = 0.25 + 0.25 + 0.0625
    E = (2.25 - 1.0) * 2 + (0.5625 - 1.0)
    A = float(L)
    H = A + E
    rel = np.sqrt(D / A)
    cosd = (D - E * E / (np.sqrt(H) + np.sqrt(A)) ** 2) / (2.0 * np.sqrt(H * A))
    for algo in (0, 1, 2):
        g = cg.cg_drift_scores(acts, refs, 1, 1, algo=algo, status=st).cpu().numpy()
        assert abs(g[0, 0, 0] - rel) <= 1e-5 * rel, (algo, g[0, 0, 0], rel)
        assert g[1, 0, 0] == 0.5, algo
        assert abs(g[2, 0, 0] - cosd) <= 1e-5 * max(cosd, rel * rel / 2) + 1e-12, (algo, g[2, 0, 0], cosd)
    assert cg.cg_read_status(st) == (0, 0)
    del acts, refs, a_flat, h_flat
    torch.cuda.empty_cache()
