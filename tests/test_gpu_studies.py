"""The paper's studies on the GPU path (Sec. 5.3-5.5), at full size.

Collusion (c = 1..4 evenly spaced), attacker position (five fractions) and
depth (k = 2..12) keep A-hat = 1.000; the frontier holds A-hat = 1.000 down
to eps = 0.002 at sigma_hw = 0.002 and gives way below it; the noise-floor
study holds while sigma_hw <= eps and fails once the floor is twice the
tamper.  The factorial's 324 configurations all separate with relative-L2.
Smaller copies of sampled configurations are checked end to end against the
oracle (generator, drift scores, bit-exact ranking of the GPU's scores)."""
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


def gpu_auroc(cg, cfg, stat=0):
    desc = cg.PipelineDesc.from_config(cfg)
    acts, refs, labels = cg.cg_generate_pipeline(desc)
    sc = cg.cg_drift_scores(acts, refs, cfg["n_shards"], cfg["n_canaries"])
    return cg.cg_auroc(sc[stat][None].contiguous(), labels[None])["auroc"].item()


@pytest.mark.parametrize("study", ["collusion", "position", "depth"])
def test_robustness_substudies(cg, study):
    """Sec. 5.3: A-hat = 1.000 for every depth, position and colluder count."""
    for cfg in SI.STUDIES[study]():
        assert gpu_auroc(cg, cfg) == PAPER["full_detector_auroc"]["value"], cfg


def test_frontier(cg):
    """Sec. 5.5: at the floor sigma_hw = 0.002, A-hat = 1.000 down to
    eps = 0.002 and gives way at eps = 0.001."""
    for cfg in SI.frontier_configs():
        A = gpu_auroc(cg, cfg)
        if cfg["tamper_param"] >= 0.002:
            assert A == 1.0, cfg["tamper_param"]
        else:
            assert A < 1.0


def test_paper_noise_floor(cg):
    """Sec. 5.4: detection survives sigma_hw up to eps = 0.05 and fails once
    the floor is twice the tamper; A-hat never rises with sigma_hw."""
    by_sigma = {}
    for cfg in SI.paper_snr_configs():
        by_sigma.setdefault(cfg["benign_sigma"], []).append(gpu_auroc(cg, cfg))
    sig = sorted(by_sigma)
    means = [np.mean(by_sigma[s]) for s in sig]
    assert all(a >= b for a, b in zip(means, means[1:]))
    assert all(m == 1.0 for s, m in zip(sig, means) if s <= 0.05)
    assert all(m < 1.0 for s, m in zip(sig, means) if s >= 0.1)


def test_raised_noise_floor_study(cg):
    """Heterogeneous per-stage noise (lognormal 0.5) against eps = 1e-2: A-hat
    falls as sigma / eps grows through 1."""
    A = [gpu_auroc(cg, cfg) for cfg in SI.snr_configs()]
    assert A[0] == 1.0 and A[-1] < 0.5
    assert all(a >= b - 1e-12 for a, b in zip(A, A[1:]))


def test_factorial_all_separate(cg):
    """All 324 factorial configurations separate with relative-L2 (Table 1,
    full detector)."""
    for cfg in SI.factorial_configs():
        assert gpu_auroc(cg, cfg) == 1.0, cfg["config_id"]


@pytest.mark.parametrize("study,idx", [("collusion", 9), ("position", 0), ("position", 12),
                                       ("frontier", 15), ("frontier", 18), ("depth", 0),
                                       ("paper_snr", 12), ("paper_snr", 15)])
def test_shrunk_study_configs_match_oracle(cg, orc, study, idx):
    """Shrunk study configurations end to end: every generated element, every
    drift score on the GPU's bytes, and u2 / gt / eq / A-hat of the GPU's own
    scores bit-exact against the oracle's ranking."""
    from tests._fullpath import check_against_oracle, run_gpu
    cfg = SI.shrink(SI.STUDIES[study]()[idx], n_canaries=16, tokens=8)
    check_against_oracle(orc, cfg, run_gpu(cg, cfg))


@pytest.mark.parametrize("study,idx", [("factorial", 323), ("factorial", 300), ("factorial", 270),
                                       ("snr", 6), ("snr", 0)])
def test_full_size_configs_sampled_against_oracle(cg, orc, study, idx):
    """The largest factorial configurations (16 x 8192 x 64 x 64) and the
    noise-floor steps (8 x 4096 x 128 x 128) at full size: sampled segments of
    the generator against the oracle, and neutral bytes planted into sampled
    segments scored in the same launch as the rest of the pipeline."""
    import torch
    from tests._cmp import assert_live_close, assert_normals_close, assert_scores_close
    cfg = SI.STUDIES[study]()[idx]
    S, N, L = cfg["n_shards"], cfg["n_canaries"], cfg["tokens"] * cfg["hidden"]
    acts, refs, labels = cg.cg_generate_pipeline(cg.PipelineDesc.from_config(cfg))
    D = orc.desc_from_dict(cfg)
    picks = [(0, 0), (cfg["malicious"][0], N - 1), (S // 2, N // 2)]
    for s, n in picks:
        o_r, _, o_a, o_c = orc.generate_segment(D, s, n)
        g_r = refs[s, n].cpu().numpy()
        assert_normals_close(g_r, o_r, what="references")
        assert_live_close(acts[s, n].cpu().numpy().view(np.uint16), o_a, g_r, o_r, o_c)
    planted = {}
    for i, (s, n) in enumerate([(1, 1), (S - 1, 0)]):
        pa, pr = SI.drift_arrays(1, 1, L, seed=900 + i)
        acts[s, n].copy_(torch.from_numpy(pa.view(np.float16).reshape(-1)))
        refs[s, n].copy_(torch.from_numpy(pr.reshape(-1)))
        planted[(s, n)] = (pa.reshape(-1), pr.reshape(-1))
    scores = cg.cg_drift_scores(acts, refs, S, N).cpu().numpy()
    for (s, n), (pa, pr) in planted.items():
        out, _ = orc.drift_segment(pa, pr)
        assert_scores_close(scores[:, n, s][:, None], out[:, None], what=f"segment {(s, n)}")
