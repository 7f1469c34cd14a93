"""End to end through the C ABI on the GPU: generate -> drift -> control
labels -> AUROC, checked against the detection outcomes the paper reports
(tests/golden/paper_values.json) and against the oracle: its own end-to-end
A-hat on the tiny pipeline, and on shrunk factorial configurations every
generated element, every drift score and the bit-exact ranking of the GPU's
own scores."""
import json
import os

import numpy as np
import pytest

import seeded_inputs as SI

pytestmark = pytest.mark.gpu
PAPER = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_values.json")))


@pytest.fixture(scope="module")
def cg():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_19490_gb300 as m
    m.build()
    return m


def gpu_path(cg, cfg, control_seeds=()):
    desc = cg.PipelineDesc.from_config(cfg)
    acts, refs, labels = cg.cg_generate_pipeline(desc)
    S, N = cfg["n_shards"], cfg["n_canaries"]
    scores = cg.cg_drift_scores(acts, refs, S, N)
    out = {}
    for k, name in enumerate(("rel_l2", "max_abs", "cos_dev")):
        out[name] = cg.cg_auroc(scores[k][None].contiguous(), labels[None])["auroc"].item()
    ctrl = []
    for seed in control_seeds:
        cl = cg.cg_make_control_labels(labels[None], seed=seed)
        ctrl.append(cg.cg_auroc(scores[0][None].contiguous(), cl)["auroc"].item())
    out["control"] = ctrl
    return out


def oracle_path(orc, cfg):
    acts, refs, labels = orc.generate_pipeline(orc.desc_from_dict(cfg))
    sc = orc.drift_scores(acts, refs, cfg["n_shards"], cfg["n_canaries"]).astype(np.float32)
    return {name: orc.auroc(sc[k][None], labels[None])["auroc"][0]
            for k, name in enumerate(("rel_l2", "max_abs", "cos_dev"))}


def test_tiny_full_detector(cg, orc):
    g = gpu_path(cg, SI.TINY)
    o = oracle_path(orc, SI.TINY)
    assert g["rel_l2"] == o["rel_l2"] == PAPER["full_detector_auroc"]["value"]


def test_paper_shape_detector_and_control(cg):
    cfg = SI.PAPER_SHAPE
    g = gpu_path(cg, cfg, control_seeds=range(100, 120))
    assert g["rel_l2"] == 1.0
    lo, hi = PAPER["control_acceptance"]["interval"]
    assert lo <= float(np.mean(g["control"])) <= hi


def test_cosine_blind_to_rescale(cg):
    """Cosine ablation on a pure rescale falls below chance (Sec. 5.2);
    relative-L2 still separates (Table 1)."""
    cfg = SI.shrink(SI.PAPER_SHAPE, tamper=SI.TAMPER_SCALE, tamper_param=1.10,
                    n_canaries=32)
    g = gpu_path(cg, cfg)
    assert g["rel_l2"] == 1.0
    assert g["cos_dev"] < 0.5 and PAPER["cosine_rescale_auroc"]["below_chance"]


@pytest.mark.parametrize("cid", [0, 13, 26, 53, 80, 107, 134, 190, 222, 271, 300, 323])
def test_factorial_configs_match_oracle(cg, orc, cid):
    """Shrunk factorial configurations end to end: the generator over every
    element, every drift score on the GPU's bytes, and u2 / gt / eq / A-hat of
    the GPU's own scores bit-exact against the oracle's ranking."""
    from tests._fullpath import check_against_oracle, run_gpu
    cfg = SI.shrink(SI.factorial_configs()[cid], n_canaries=12, tokens=8)
    check_against_oracle(orc, cfg, run_gpu(cg, cfg))
