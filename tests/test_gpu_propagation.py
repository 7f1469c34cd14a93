"""GPU parity of the propagating pipeline (Eq. 2's recursion with a
linearised block gain) against the oracle.

With gain <= 1 every rounding difference between the GPU's fp32 and the
oracle's fp64 arithmetic stays bounded, so the fp16 live values are compared
element by element.  The GPU rounds the inherited input
v = a + gain (h_prev - a_prev) to fp32 before the noise is added, so where
the live value nearly cancels to zero the difference is bounded by fp16 ulps
of the magnitudes entering the sum, not of the small result.  Each stage can
add one rounding disagreement of about one such ulp, and earlier ones are
carried with gain^k, so stage s is bounded by 1 + sum_{k<=s} gain^k ulps of
the largest magnitude along the chain, max over stages k <= s of
max(|h_k|, |a_k|) at that element.  With
gain > 1 such differences grow geometrically along the pipeline by
construction, so the mismatch scores (relative 1e-3) and the detection
outcome are compared instead."""
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


def base(**kw):
    c = SI.shrink(SI.PAPER_SHAPE, n_canaries=4, tokens=8, hidden=256)
    c.update(kw)
    return c


def test_gain_zero_equals_hop_local(cg):
    import torch
    c = base()
    desc = cg.PipelineDesc.from_config(c)
    a0, r0, l0 = cg.cg_generate_pipeline(desc)
    a1, r1, l1 = cg.cg_generate_propagating(desc, 0.0)
    assert torch.equal(a0, a1) and torch.equal(r0, r1) and torch.equal(l0, l1)


CASES = {
    "additive": base(),
    "mult_ragged": base(noise=SI.NOISE_MULT, hidden=100, tokens=3, n_outlier=2),
    "signflip": base(tamper=SI.TAMPER_SIGNFLIP_FULL),
    "channels": base(tamper=SI.TAMPER_SIGNFLIP_CHANNELS, tamper_param=0.05, malicious=(0, 6)),
    "scale": base(tamper=SI.TAMPER_SCALE, tamper_param=1.1),
}


@pytest.mark.parametrize("gain", [0.5, 1.0])
@pytest.mark.parametrize("name", sorted(CASES))
def test_propagating_matches_oracle(cg, orc, name, gain):
    c = CASES[name]
    g_acts, g_refs, _ = cg.cg_generate_propagating(cg.PipelineDesc.from_config(c), gain)
    o_acts, o_refs = orc.generate_propagating(orc.desc_from_dict(c), gain)
    assert_normals_close(g_refs.cpu().numpy(), o_refs, what="references")
    g = g_acts.cpu().numpy().astype(np.float64)
    o = o_acts.view(np.float16).astype(np.float64)
    scale = np.maximum.accumulate(np.maximum(np.abs(o), np.abs(o_refs.astype(np.float64))), axis=0)
    ulp = np.exp2(np.floor(np.log2(np.maximum(scale, 2.0 ** -14))) - 10)
    err = np.abs(g - o) / ulp
    d = half_ulp_distance(g_acts.cpu().numpy().view(np.uint16), o_acts)
    print(f"{name} gain {gain}: max scaled err {err.max():.2f}, raw ulp max {d.max()}, "
          f"differing {(d > 0).mean():.2e}")
    for stage in range(err.shape[0]):
        tol = 1.0 + sum(gain ** k for k in range(stage + 1))
        assert err[stage].max() <= tol, (stage, err[stage].max(), tol)
    assert (d > 0).mean() < 0.01


def test_amplifying_gain_scores_and_detection(cg, orc):
    import torch
    c = base(malicious=(3,), tamper_param=0.05)
    S, N = c["n_shards"], c["n_canaries"]
    for gain in (0.5, 1.5):
        g_acts, g_refs, labels = cg.cg_generate_propagating(cg.PipelineDesc.from_config(c), gain)
        g = cg.cg_drift_scores(g_acts, g_refs, S, N)
        A = cg.cg_auroc(g[0][None].contiguous(), labels[None])["auroc"].item()
        o_acts, o_refs = orc.generate_propagating(orc.desc_from_dict(c), gain)
        o = orc.drift_scores(o_acts, o_refs, S, N)
        assert np.allclose(g.cpu().numpy()[0], o[0], rtol=1e-3)
        o_lab = np.zeros((1, N, S), np.int8)
        o_lab[:, :, 3] = 1
        assert A == orc.auroc(o[0].astype(np.float32)[None], o_lab)["auroc"][0]
        assert (A == 1.0) == (gain < 1.0)


def test_propagation_study_position_invariance(cg):
    """With attenuating blocks (gain < 1) the tampering stage keeps the largest
    mismatch wherever it sits (A-hat = 1, the paper's position invariance);
    with amplifying blocks (gain > 1) downstream stages overtake it unless
    it is the last stage."""
    import seeded_inputs as SI
    for cfg in SI.propagation_configs():
        c = dict(cfg)
        gain = c.pop("gain")
        desc = cg.PipelineDesc.from_config(c)
        acts, refs, labels = cg.cg_generate_propagating(desc, gain)
        sc = cg.cg_drift_scores(acts, refs, c["n_shards"], c["n_canaries"])
        A = cg.cg_auroc(sc[0][None].contiguous(), labels[None])["auroc"].item()
        last = c["malicious"][0] == c["n_shards"] - 1
        if gain < 1.0 or last:
            assert A == 1.0, (gain, c["malicious"], A)
        elif gain > 1.0:
            assert A < 1.0, (gain, c["malicious"], A)
