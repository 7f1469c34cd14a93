"""Edge cases and maximum sizes of the boundary on the GPU, against the oracle:
the largest stage count (1024) with almost every stage colluding, the
largest outlier count, a 65,536-wide hidden size with half the channels
flipped, single-element segments, and the degenerate ranking cases (no pair,
one stage, all scores equal)."""
import numpy as np
import pytest

import seeded_inputs as SI
from tests._cmp import assert_normals_close, half_ulp_distance

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
    o_acts, o_refs, o_labels = orc.generate_pipeline(orc.desc_from_dict(cfg))
    assert np.array_equal(labels.cpu().numpy(), o_labels)
    assert_normals_close(refs.cpu().numpy(), o_refs, what="references")
    d = half_ulp_distance(acts.cpu().numpy().view(np.uint16), o_acts)
    assert d.max() <= 1
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
