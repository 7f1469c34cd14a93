"""Out-of-bounds writes: every output and workspace buffer of every entry
point sits inside a larger device buffer with 4 KiB guard regions on both
sides, filled with a fixed byte pattern before the call.  After the call the
guards must hold the pattern byte for byte, the inputs must be unchanged and
the outputs must equal the oracle's.  Shapes are ragged on purpose: hidden
sizes 1, 7, 100 and 131; segment lengths 1, 9 and 16,385; 2, 33 and 1,024
stages; batch and canary counts that are not multiples of 8, 32 or 64; and
every kernel variant of the ranking (per-configuration lanes, one block per
configuration, per-canary lanes, and the wide-pipeline warps).

This stands in for a memory checker: the index arithmetic of each launch is
exercised on the shapes where an off-by-one would land in a guard."""
import numpy as np
import pytest

import seeded_inputs as SI
from tests._cmp import (assert_live_close, assert_normals_close, assert_scores_close,
                       half_ulp_distance)

pytestmark = pytest.mark.gpu
GUARD = 4096


@pytest.fixture(scope="module")
def cg():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_19490_gb300 as m
    m.build()
    return m


class Guarded:
    """A tensor of `shape` and `dtype` inside a byte buffer with GUARD bytes
    of pattern on both sides (the interior starts with the pattern too)."""

    def __init__(self, shape, dtype):
        import torch
        self.shape = tuple(int(x) for x in shape)
        esz = torch.empty((), dtype=dtype).element_size()
        self.nb = int(np.prod(self.shape)) * esz
        total = 2 * GUARD + self.nb
        k = torch.arange(total, device="cuda", dtype=torch.int64)
        self.pattern = ((k * 37 + 11) % 251).to(torch.uint8)
        self.base = self.pattern.clone()
        self.t = self.base[GUARD:GUARD + self.nb].view(dtype).view(self.shape)

    def check(self, what):
        import torch
        torch.cuda.synchronize()
        below = torch.equal(self.base[:GUARD], self.pattern[:GUARD])
        above = torch.equal(self.base[GUARD + self.nb:], self.pattern[GUARD + self.nb:])
        assert below, f"{what}: bytes written below the buffer"
        assert above, f"{what}: bytes written above the buffer"


def guarded_ws(nbytes):
    import torch
    return Guarded((nbytes,), torch.uint8)


# ----------------------------------------------------------------------------- generator

GEN_CASES = {
    "d1_T9_channels": SI._cfg(2, 1, 3, 9, [1], SI.NOISE_MULT, 1e-3, SI.TAMPER_SIGNFLIP_CHANNELS,
                              0.5, seed=21, n_outlier=1),
    "d7_T1_additive": SI._cfg(3, 7, 33, 1, [0, 2], SI.NOISE_PAPER, 2e-3, SI.TAMPER_ADDITIVE, 0.05,
                              seed=22, n_outlier=2, shard_sigma_lognormal=0.5),
    "d100_T9_scale": SI._cfg(2, 100, 5, 9, [0], SI.NOISE_PAPER, 1e-3, SI.TAMPER_SCALE, 1.05,
                             seed=23, n_outlier=3),
    "d7_S33_full": SI._cfg(33, 7, 3, 9, [5, 32], SI.NOISE_PAPER, 1e-3, SI.TAMPER_SIGNFLIP_FULL, 0.0,
                           seed=24),
    "d131_two_stat_chunks": SI._cfg(2, 131, 2, 501, [1], SI.NOISE_PAPER, 1e-3, SI.TAMPER_ADDITIVE,
                                    0.01, seed=25, n_outlier=1),
}


def compare_generated(g_acts, g_refs, o_acts, o_refs, o_coef):
    gr = g_refs.cpu().numpy()
    assert_normals_close(gr, o_refs, what="references")
    assert_live_close(g_acts.cpu().numpy().view(np.uint16), o_acts, gr, o_refs, o_coef)


@pytest.mark.parametrize("name", sorted(GEN_CASES))
def test_generator_writes_inside_its_buffers(cg, orc, name):
    import torch
    cfg = GEN_CASES[name]
    S, N, L = cfg["n_shards"], cfg["n_canaries"], cfg["tokens"] * cfg["hidden"]
    desc = cg.PipelineDesc.from_config(cfg)
    acts = Guarded((S, N, L), torch.float16)
    refs = Guarded((S, N, L), torch.float32)
    labels = Guarded((N, S), torch.int8)
    ws = guarded_ws(cg.cg_generate_workspace_size(desc))
    cg.cg_generate_pipeline(desc, acts.t, refs.t, labels.t, ws.t)
    for b, what in ((acts, "acts"), (refs, "refs"), (labels, "labels"), (ws, "workspace")):
        b.check(f"cg_generate_pipeline {name} {what}")
    D = orc.desc_from_dict(cfg)
    _, _, o_labels = orc.generate_pipeline(D)
    o_acts, o_refs, o_coef = orc.generate_coefs(D)
    compare_generated(acts.t, refs.t, o_acts, o_refs, o_coef)
    assert np.array_equal(labels.t.cpu().numpy(), o_labels)

    # the benign recompute (ceiling and noisy reference) into the same kind of buffers
    out = Guarded((S, N, L), torch.float32)
    ws2 = guarded_ws(cg.cg_generate_workspace_size(desc))
    cg.cg_generate_recompute(desc, 1, out.t, ws2.t)
    out.check(f"cg_generate_recompute {name} out")
    ws2.check(f"cg_generate_recompute {name} workspace")
    g = out.t.cpu().numpy()
    o = orc.generate_recompute(orc.desc_from_dict(cfg), 1)
    assert half_ulp_distance(g.astype(np.float16).view(np.uint16),
                             o.astype(np.float16).view(np.uint16)).max() <= 1


@pytest.mark.parametrize("name", ["d7_T1_additive", "d100_T9_scale", "d7_S33_full"])
def test_propagating_writes_inside_its_buffers(cg, orc, name):
    import torch
    cfg = GEN_CASES[name]
    S, N, L = cfg["n_shards"], cfg["n_canaries"], cfg["tokens"] * cfg["hidden"]
    desc = cg.PipelineDesc.from_config(cfg)
    acts = Guarded((S, N, L), torch.float16)
    refs = Guarded((S, N, L), torch.float32)
    labels = Guarded((N, S), torch.int8)
    ws = guarded_ws(cg.cg_generate_workspace_size(desc))
    gain = 0.5
    cg.cg_generate_propagating(desc, gain, acts.t, refs.t, labels.t, ws.t)
    for b, what in ((acts, "acts"), (refs, "refs"), (labels, "labels"), (ws, "workspace")):
        b.check(f"cg_generate_propagating {name} {what}")
    o_acts, o_refs = orc.generate_propagating(orc.desc_from_dict(cfg), gain)
    assert_normals_close(refs.t.cpu().numpy(), o_refs, what="references")
    # each stage inherits gain x the upstream rounding, so the bound grows
    # with depth: 1 + sum_k gain^k fp16 steps of the largest magnitude so far
    g = acts.t.cpu().numpy().astype(np.float64)
    o = o_acts.view(np.float16).astype(np.float64)
    scale = np.maximum.accumulate(np.maximum(np.abs(o), np.abs(o_refs.astype(np.float64))), axis=0)
    ulp = np.exp2(np.floor(np.log2(np.maximum(scale, 2.0 ** -14))) - 10)
    err = np.abs(g - o) / ulp
    for stage in range(S):
        assert err[stage].max() <= 1.0 + sum(gain ** k for k in range(stage + 1))


# ----------------------------------------------------------------------------- drift

DRIFT_SHAPES = [(2, 3, 1), (2, 3, 9), (33, 3, 16385), (2, 65, 16392), (3, 5, 8), (2, 3, 36864)]


@pytest.mark.parametrize("S,N,L", DRIFT_SHAPES)
def test_drift_writes_inside_scores_and_workspace(cg, orc, S, N, L):
    import torch
    acts_np, refs_np = SI.drift_arrays(S, N, L, seed=S * 1000 + N + L)
    acts = torch.from_numpy(acts_np.view(np.float16)).cuda()
    refs = torch.from_numpy(refs_np).cuda()
    a0, r0 = acts.clone(), refs.clone()
    o = orc.drift_scores(acts_np, refs_np, S, N)
    wsz = cg.cg_drift_workspace_size(S, N, L)
    algos = [("auto", None), ("stream", cg.DRIFT_STREAM)]
    if L % 8 == 0:
        algos += [("bulk", cg.DRIFT_BULK), ("bulk2", cg.DRIFT_BULK_2CTA)]
    for name, algo in algos:
        sc = Guarded((3, N, S), torch.float32)
        ws = guarded_ws(wsz)
        cg.cg_drift_scores(acts, refs, S, N, scores=sc.t, ws=ws.t, algo=algo)
        sc.check(f"drift {name} scores")
        ws.check(f"drift {name} workspace")
        assert_scores_close(sc.t.cpu().numpy(), o, what=f"drift {name}")
    # live activations in pinned host memory
    h_acts = torch.from_numpy(acts_np.view(np.float16)).pin_memory()
    sc = Guarded((3, N, S), torch.float32)
    ws = guarded_ws(wsz)
    cg.cg_drift_scores_host(h_acts, refs, S, N, scores=sc.t, ws=ws.t)
    sc.check("drift host scores")
    ws.check("drift host workspace")
    assert_scores_close(sc.t.cpu().numpy(), o, what="drift host")
    # the same problem as a batch of configurations: S = C x S' with C = 1
    # and, where S splits, C = 2 configurations of S / 2 stages
    for C in (1, 2) if S % 2 == 0 else (1,):
        sc = Guarded((3, C, N, S // C), torch.float32)
        ws = guarded_ws(cg.cg_drift_workspace_size(S, N, L))
        cg.cg_drift_scores_batch(acts, refs, C, S // C, N, scores=sc.t, ws=ws.t)
        sc.check(f"drift batch of {C} scores")
        ws.check(f"drift batch of {C} workspace")
        for c in range(C):
            oc = orc.drift_scores(acts_np[c * S // C:(c + 1) * S // C],
                                  refs_np[c * S // C:(c + 1) * S // C], S // C, N)
            assert_scores_close(sc.t.cpu().numpy()[:, c], oc, what=f"drift batch {C}, config {c}")
    # no workspace at all
    sc = Guarded((3, N, S), torch.float32)
    cg.cg_drift_scores_noalloc(acts, refs, S, N, sc.t)
    sc.check("drift no-alloc scores")
    assert_scores_close(sc.t.cpu().numpy(), o, what="drift no-alloc")
    assert torch.equal(acts, a0) and torch.equal(refs, r0), "inputs changed"


# ----------------------------------------------------------------------------- ranking

# (C, N, S, malicious, excluded, tie levels) -> the kernel each shape selects
RANK_SHAPES = [
    (1219, 5, 7, 2, 1, 4),        # a warp per configuration, rows narrower than 8
    (1217, 33, 16, 1, 0, None),   # a warp per configuration, 16-byte rows
    (13, 65, 2, 1, 0, 3),         # one block per configuration
    (2, 1025, 9, 3, 2, 5),        # a lane per canary, then one block per configuration
    (305, 3, 33, 4, 3, 6),        # wide pipelines, a warp per canary, many configurations
    (3, 65, 1024, 10, 5, None),   # wide pipelines, few configurations
]


@pytest.mark.parametrize("C,N,S,n_mal,excl,ties", RANK_SHAPES)
def test_ranking_writes_inside_its_outputs(cg, orc, C, N, S, n_mal, excl, ties):
    import torch
    sc_np, lb_np = SI.score_arrays(C, N, S, seed=C + N + S, n_malicious=n_mal, tie_levels=ties,
                                   excluded=excl)
    sc = torch.from_numpy(sc_np).cuda()
    lb = torch.from_numpy(lb_np).cuda()
    s0, l0 = sc.clone(), lb.clone()

    outs = {k: Guarded((C, N), torch.int64) for k in ("u2", "gt", "eq")}
    auroc = Guarded((C,), torch.float64)
    cg.cg_auroc(sc, lb, u2=outs["u2"].t, gt=outs["gt"].t, eq=outs["eq"].t, auroc=auroc.t)
    o = orc.auroc(sc_np, lb_np)
    for k, b in outs.items():
        b.check(f"cg_auroc {k}")
        assert np.array_equal(b.t.cpu().numpy(), o[k]), k
    auroc.check("cg_auroc auroc")
    assert np.array_equal(auroc.t.cpu().numpy().view(np.uint64), o["auroc"].view(np.uint64))

    ctrl = Guarded((C, N, S), torch.int8)
    cg.cg_make_control_labels(lb, seed=5, config_id0=3, ctrl=ctrl.t)
    ctrl.check("cg_make_control_labels")
    assert np.array_equal(ctrl.t.cpu().numpy(), orc.control_labels(lb_np, seed=5, config_id0=3))

    if N * S <= 16384:
        pooled = {k: Guarded((C,), torch.int64) for k in ("u2", "n_mal", "n_ben")}
        pa = Guarded((C,), torch.float64)
        cg.cg_auroc_pooled(sc, lb, u2=pooled["u2"].t, n_mal=pooled["n_mal"].t,
                           n_ben=pooled["n_ben"].t, auroc=pa.t)
        op = orc.auroc_pooled(sc_np, lb_np)
        for k, b in pooled.items():
            b.check(f"cg_auroc_pooled {k}")
            assert np.array_equal(b.t.cpu().numpy(), op[k]), k
        pa.check("cg_auroc_pooled auroc")
        assert np.array_equal(pa.t.cpu().numpy().view(np.uint64), op["auroc"].view(np.uint64))
    assert torch.equal(sc, s0) and torch.equal(lb, l0), "inputs changed"


@pytest.mark.parametrize("C,N,S", [(3, 65, 2), (1, 3, 1024), (1219, 5, 7)])
def test_random_scores_write_inside_their_output(cg, orc, C, N, S):
    import torch
    out = Guarded((C, N, S), torch.float32)
    cg.cg_random_scores(17, C, N, S, config_id0=9, out=out.t)
    out.check("cg_random_scores")
    assert np.array_equal(out.t.cpu().numpy(), orc.random_scores(17, C, N, S, config_id0=9))


def test_rng_views_write_inside_their_outputs(cg, orc):
    import torch
    w = Guarded((7, 4), torch.int32)
    cg.cg_philox_words(3, 1, 2, 0, 11, 7, out=w.t)
    w.check("cg_philox_words")
    assert np.array_equal(w.t.cpu().numpy().view(np.uint32).ravel(),
                          orc.philox_words(3, 1, 2, 0, 11, 7))
    z = Guarded((5, 4), torch.float32)
    cg.cg_philox_normals(3, 1, 2, 0, 11, 5, out=z.t)
    z.check("cg_philox_normals")
    assert_normals_close(z.t.cpu().numpy().ravel(), orc.philox_normals(3, 1, 2, 0, 11, 5))
    words = np.random.Generator(np.random.PCG64(4)).integers(0, 2**32, size=(9, 2), dtype=np.uint32)
    p = Guarded((9, 2), torch.float32)
    cg.cg_box_muller_pairs(torch.from_numpy(words.view(np.int32)).cuda(), out=p.t)
    p.check("cg_box_muller_pairs")
    assert_normals_close(p.t.cpu().numpy(), orc.box_muller_pairs(words))
