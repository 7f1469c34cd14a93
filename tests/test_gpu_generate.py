"""GPU parity of the Philox layer and the pipeline generator against the oracle.

Philox words bit-exact; normals and references within the normal tolerance;
labels bit-exact; fp16 live values within the live-value bound of
tests/_cmp.py (one fp16 step away from cancellations).  Inputs are
descriptions only, so nothing the oracle sees comes from the CUDA path.
"""
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


@pytest.mark.parametrize("seed,c1,c2,c3,first,n", [
    (0, 0, 0, 0, 0, 4096),
    (0x123456789ABCDEF0, 4095, 4 * 7 + 2, 0, 2**32 - 100, 100),
    (2**64 - 1, (4 << 24) | 77, 4 * 323 + 3, 0, 12345, 777),
    (42, 1, 2, 3, 7, 1),
])
def test_philox_words_bit_exact(cg, orc, seed, c1, c2, c3, first, n):
    g = cg.cg_philox_words(seed, c1, c2, c3, first, n).cpu().numpy().view(np.uint32).ravel()
    o = orc.philox_words(seed, c1, c2, c3, first, n)
    assert np.array_equal(g, o)


def test_philox_normals(cg, orc):
    for seed, c1, c2 in [(0, 0, 0), (9, 511, 4 * 5 + 1), (2**63 + 5, 3, 4 * 2 + 2)]:
        g = cg.cg_philox_normals(seed, c1, c2, 0, 0, 1 << 16).cpu().numpy().ravel()
        o = orc.philox_normals(seed, c1, c2, 0, 0, 1 << 16)
        assert_normals_close(g, o)


def test_box_muller_exhaustive(cg, orc):
    """Each factor of the transform over every value of its 24-bit word
    index: the radius over all x0 >> 8 at angle 0, then the angle over all
    x1 >> 8 at the largest radius, a radius near 1 and radius 0.  The low 8
    bits of each word are set to show they are ignored."""
    import torch
    k = np.arange(1 << 24, dtype=np.uint32) << 8
    sweeps = [(k | 0xAB, np.zeros_like(k))]
    for k1 in (0, int(round(np.exp(-0.5) * 2**24)) - 1, 2**24 - 1):
        sweeps.append((np.full_like(k, (k1 << 8) | 0x5C), k | 0x3F))
    for i, (x0, x1) in enumerate(sweeps):
        w = np.stack([x0, x1], axis=1)
        g = cg.cg_box_muller_pairs(torch.from_numpy(w.view(np.int32)).cuda()).cpu().numpy()
        o = orc.box_muller_pairs(w)
        assert_normals_close(g, o, what=f"sweep {i}")
        if i == 0:
            # the radius alone: within 2.5 units of 2^-24 relative; exact 0 at u1 = 1
            r_g, r_o = g[:, 0].astype(np.float64), o[:, 0]
            assert np.all(g[:, 1] == 0.0)
            assert r_g[-1] == 0.0 and r_o[-1] == 0.0
            assert np.max(np.abs(r_g[:-1] - r_o[:-1]) / r_o[:-1]) <= 2.5 * 2.0**-24
        del g, o, w


CASES = {
    "tiny": SI.TINY,
    "7b_small": SI.shrink(SI.SEVEN_B, n_canaries=4, tokens=4, hidden=512),
    "70b_small": SI.shrink(SI.SEVENTY_B, n_canaries=3, tokens=2, hidden=8192),
    "paper_shape_small": SI.shrink(SI.PAPER_SHAPE, n_canaries=5, tokens=6),
    "snr_step": SI.shrink(SI.snr_configs()[5], n_canaries=3, tokens=4, hidden=1024),
    "signflip_full": SI.shrink(SI.TINY, tamper=SI.TAMPER_SIGNFLIP_FULL, malicious=(0, 3)),
    "scale": SI.shrink(SI.TINY, tamper=SI.TAMPER_SCALE, tamper_param=1.1),
    "scale_overflow": SI.shrink(SI.TINY, tamper=SI.TAMPER_SCALE, tamper_param=1.0e5),
    "scale_subnormal": SI.shrink(SI.TINY, tamper=SI.TAMPER_SCALE, tamper_param=1.0e-6),
    "collusion": SI.shrink(SI.TINY, n_shards=8, malicious=(1, 3, 5, 7), noise=SI.NOISE_PAPER),
    "ragged_d100": SI.shrink(SI.TINY, hidden=100, tokens=3, n_outlier=3),
    "ragged_L7": SI.shrink(SI.TINY, hidden=7, tokens=1, n_outlier=1,
                           tamper=SI.TAMPER_SIGNFLIP_CHANNELS, tamper_param=0.3),
    "d1": SI.shrink(SI.TINY, hidden=1, tokens=5, n_outlier=0, noise=SI.NOISE_PAPER),
    "clean": SI.shrink(SI.TINY, malicious=(), noise=SI.NOISE_PAPER),
}
CASES.update({f"factorial_{i}": SI.shrink(c, n_canaries=2, tokens=2)
              for i, c in enumerate(SI.factorial_configs()) if i in (0, 17, 40, 95, 161, 250, 323)})


def compare_pipeline(cg, orc, cfg, acts, refs, labels=None, segments=None):
    """acts/refs: device tensors [S][N][L]; compares the listed (s, n) segments
    (all when None) against the oracle's generator.  Returns the largest
    distance of a live value in fp16 steps."""
    D = orc.desc_from_dict(cfg)
    if segments is None:
        o_acts, o_refs, o_coef = orc.generate_coefs(D)
        g_acts = acts.cpu().numpy().view(np.uint16)
        g_refs = refs.cpu().numpy()
        if labels is not None:
            _, _, o_labels = orc.generate_pipeline(D)
            assert np.array_equal(labels.cpu().numpy(), o_labels)
        pairs = [(g_acts, g_refs, o_acts, o_refs, o_coef)]
    else:
        pairs = []
        for s, n in segments:
            o_r, _, o_a, o_c = orc.generate_segment(D, s, n)
            pairs.append((acts[s, n].cpu().numpy().view(np.uint16), refs[s, n].cpu().numpy(),
                          o_a, o_r, o_c))
    worst = 0
    for g_a, g_r, o_a, o_r, o_c in pairs:
        assert_normals_close(g_r, o_r, scale=1.0, what="references")
        worst = max(worst, assert_live_close(g_a, o_a, g_r, o_r, o_c))
        assert (half_ulp_distance(g_a, o_a) > 0).mean() < 1e-2
    return worst


@pytest.mark.parametrize("name", sorted(CASES))
def test_generator_matches_oracle(cg, orc, name):
    cfg = CASES[name]
    desc = cg.PipelineDesc.from_config(cfg)
    acts, refs, labels = cg.cg_generate_pipeline(desc)
    compare_pipeline(cg, orc, cfg, acts, refs, labels)


def test_generator_deterministic(cg):
    import torch
    desc = cg.PipelineDesc.from_config(CASES["7b_small"])
    a1, r1, _ = cg.cg_generate_pipeline(desc)
    a2, r2, _ = cg.cg_generate_pipeline(desc)
    assert torch.equal(a1, a2) and torch.equal(r1, r2)


@pytest.mark.parametrize("name,cfg,segments", [
    ("7b", SI.SEVEN_B, [(0, 0), (3, 17), (3, 63), (7, 40)]),
    ("70b", SI.SEVENTY_B, [(0, 0), (7, 0), (7, 255), (15, 128), (9, 77)]),
])
def test_generator_full_size_sampled(cg, orc, name, cfg, segments):
    """At the full workload sizes, sampled segments against the oracle."""
    import torch
    desc = cg.PipelineDesc.from_config(cfg)
    acts, refs, labels = cg.cg_generate_pipeline(desc)
    torch.cuda.synchronize()
    S = cfg["n_shards"]
    expect = np.zeros((cfg["n_canaries"], S), np.int8)
    expect[:, list(cfg["malicious"])] = 1
    assert np.array_equal(labels.cpu().numpy(), expect)
    compare_pipeline(cg, orc, cfg, acts, refs, segments=segments)
    del acts, refs
    torch.cuda.empty_cache()


def test_status_word_clean(cg):
    import torch
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    desc = cg.PipelineDesc.from_config(CASES["ragged_L7"])
    cg.cg_generate_pipeline(desc, status=st)
    assert cg.cg_read_status(st) == (0, 0)
