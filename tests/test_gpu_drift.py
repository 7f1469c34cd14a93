"""GPU parity of the drift reduction (Eq. 4, cosine ablation, max-abs) against
the fp64 oracle on the same bytes.  Inputs come from seeded_inputs (numpy),
never from the CUDA path.  Shapes span several work items (16384 elements
each), ragged tails and segment starts that are not 16-byte aligned."""
import numpy as np
import pytest

import seeded_inputs as SI
from tests._cmp import assert_scores_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cg():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_19490_gb300 as m
    m.build()
    return m


def run(cg, acts, refs, S, N, **kw):
    import torch
    d_acts = torch.from_numpy(acts.view(np.float16)).cuda()
    d_refs = torch.from_numpy(refs).cuda()
    return cg.cg_drift_scores(d_acts, d_refs, S, N, **kw)


@pytest.mark.parametrize("S,N,L", [
    (2, 3, 1), (2, 3, 7), (2, 3, 8), (3, 2, 9), (4, 4, 100), (2, 2, 16384), (2, 3, 16385),
    (3, 5, 40003), (1, 2, 65536 + 5), (5, 7, 4096), (4, 16, 8192),
])
def test_drift_matches_oracle(cg, orc, S, N, L):
    acts, refs = SI.drift_arrays(S, N, L, seed=S * 1000 + N * 10 + L)
    g = run(cg, acts, refs, S, N).cpu().numpy()
    o = orc.drift_scores(acts, refs, S, N)
    assert_scores_close(g, o, what=f"S={S} N={N} L={L}")


def test_drift_paper_regimes(cg, orc):
    """Benign floor, Gaussian tamper, sign flip, rescale: the regimes of Sec. 3.2."""
    S, N, L = 4, 6, 3000
    rels = np.array([1e-3, 5e-2, 2.0, 1e-4])[:, None, None] * np.ones((S, N, 1))
    acts, refs = SI.drift_arrays(S, N, L, seed=77, rel=rels)
    g = run(cg, acts, refs, S, N).cpu().numpy()
    assert_scores_close(g, orc.drift_scores(acts, refs, S, N))


def test_drift_oracle_generated_bytes(cg, orc):
    """The oracle's own synthetic pipeline bytes (tiny workload and a rescale)."""
    for cfg in (SI.TINY, SI.shrink(SI.TINY, tamper=SI.TAMPER_SCALE, tamper_param=1.05)):
        o_acts, o_refs, _ = orc.generate_pipeline(orc.desc_from_dict(cfg))
        S, N = cfg["n_shards"], cfg["n_canaries"]
        g = run(cg, o_acts, o_refs, S, N).cpu().numpy()
        assert_scores_close(g, orc.drift_scores(o_acts, o_refs, S, N))


def test_drift_stat_stride_and_sentinels(cg, orc):
    import torch
    S, N, L = 3, 4, 1000
    acts, refs = SI.drift_arrays(S, N, L, seed=3)
    C, c = 5, 2                                  # place this config at slot 2 of 5
    big = torch.full((3, C, N, S), -7.0, dtype=torch.float32, device="cuda")
    view = big.view(-1)[c * N * S:]
    run(cg, acts, refs, S, N, scores=view, stat_stride=C * N * S)
    out = big.cpu().numpy()
    o = orc.drift_scores(acts, refs, S, N)
    assert_scores_close(out[:, c], o)
    mask = np.ones(C, bool)
    mask[c] = False
    assert np.all(out[:, mask] == -7.0)


def test_drift_nan_and_edge_values(cg, orc):
    S, N, L = 2, 2, 33
    acts, refs = SI.drift_arrays(S, N, L, seed=9)
    a = acts.view(np.float16).copy()
    a[1, 1, 5] = np.nan
    g = run(cg, a.view(np.uint16), refs, S, N).cpu().numpy()
    o = orc.drift_scores(a.view(np.uint16), refs, S, N)
    assert_scores_close(g, o)
    assert np.isnan(g[0, 1, 1]) and np.isnan(g[2, 1, 1]) and np.isfinite(g[1, 1, 1])


def test_drift_deterministic(cg):
    S, N, L = 4, 8, 50000
    acts, refs = SI.drift_arrays(S, N, L, seed=1)
    g1 = run(cg, acts, refs, S, N).cpu().numpy()
    g2 = run(cg, acts, refs, S, N).cpu().numpy()
    assert np.array_equal(g1.view(np.uint32), g2.view(np.uint32))


def test_drift_full_size_planted_segments(cg, orc):
    """70B-like workload at full size in the benchmark's launch configuration:
    neutral host bytes are planted into sampled segments of the generated
    pipeline, and those segments' scores are compared with the oracle."""
    import torch
    cfg = SI.SEVENTY_B
    S, N, L = cfg["n_shards"], cfg["n_canaries"], cfg["tokens"] * cfg["hidden"]
    desc = cg.PipelineDesc.from_config(cfg)
    acts, refs, labels = cg.cg_generate_pipeline(desc)
    picks = [(0, 0), (7, 13), (15, 255), (3, 128)]
    planted = {}
    for i, (s, n) in enumerate(picks):
        pa, pr = SI.drift_arrays(1, 1, L, seed=500 + i)
        acts[s, n].copy_(torch.from_numpy(pa.view(np.float16).reshape(-1)))
        refs[s, n].copy_(torch.from_numpy(pr.reshape(-1)))
        planted[(s, n)] = (pa.reshape(-1), pr.reshape(-1))
    ws = torch.empty(cg.cg_drift_workspace_size(S, N, L), dtype=torch.uint8, device="cuda")
    scores = cg.cg_drift_scores(acts, refs, S, N, ws=ws).cpu().numpy()
    for (s, n), (pa, pr) in planted.items():
        out, _ = orc.drift_segment(pa, pr)
        assert_scores_close(scores[:, n, s][:, None], out[:, None], what=f"segment {(s, n)}")
    # properties of every generated segment: benign floor O(sigma) (Sec. 3.4),
    # channel-flip tamper far above it, and the full detector separates them
    mal = cfg["malicious"][0]
    keep = np.ones((N, S), bool)
    for s, n in picks:
        keep[n, s] = False
    rel = scores[0]
    benign = rel[:, [s for s in range(S) if s != mal]][keep[:, [s for s in range(S) if s != mal]]]
    assert np.all((benign > 0.3 * cfg["benign_sigma"]) & (benign < 3 * cfg["benign_sigma"]))
    assert np.all(rel[keep[:, mal], mal] > 0.1)
    del acts, refs
    torch.cuda.empty_cache()


def test_drift_host_live_activations(cg, orc):
    """Live activations read from pinned host memory give the same scores as
    from device memory (same kernel, same order) and match the oracle."""
    import torch
    S, N, L = 3, 5, 40003
    acts, refs = SI.drift_arrays(S, N, L, seed=21)
    h_acts = torch.from_numpy(acts.view(np.float16)).pin_memory()
    d_refs = torch.from_numpy(refs).cuda()
    g_host = cg.cg_drift_scores_host(h_acts, d_refs, S, N).cpu().numpy()
    g_dev = cg.cg_drift_scores(h_acts.cuda(), d_refs, S, N).cpu().numpy()
    assert np.array_equal(g_host.view(np.uint32), g_dev.view(np.uint32))
    assert_scores_close(g_host, orc.drift_scores(acts, refs, S, N))


def test_drift_host_rejects_pageable(cg):
    import ctypes
    L = cg.load()
    buf = (ctypes.c_uint16 * 64)()          # ordinary (pageable) host memory
    fake = ctypes.c_void_p(0x10000)
    st = L.cg_drift_scores_host(ctypes.cast(buf, ctypes.c_void_p), fake, 2, 2, 16, fake, 4, fake,
                                1 << 20, None, None)
    assert st == 1


@pytest.mark.parametrize("algo", [1, 2, 3])
@pytest.mark.parametrize("S,N,L", [(2, 3, 8), (4, 4, 104), (2, 2, 16384), (3, 5, 40000),
                                   (1, 2, 65536 + 8), (5, 7, 4096), (4, 16, 8192), (2, 3, 4096 * 3 + 8),
                                   (3, 4, 36864), (2, 3, 16392), (2, 2, 4 * 16384 + 8)])
def test_drift_kernels_match_oracle(cg, orc, algo, S, N, L):
    """The register-streaming kernel and both TMA bulk-copy pipelines against
    the oracle; the bulk pipelines' bounded waits never give up."""
    import torch
    acts, refs = SI.drift_arrays(S, N, L, seed=S * 31 + N * 7 + L + algo)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    g = run(cg, acts, refs, S, N, algo=algo, status=st).cpu().numpy()
    assert cg.cg_read_status(st) == (0, 0)
    assert_scores_close(g, orc.drift_scores(acts, refs, S, N), what=f"algo {algo}")


def test_drift_bulk_rejects_ragged(cg):
    import torch
    acts, refs = SI.drift_arrays(2, 2, 12, seed=1)
    with pytest.raises(cg.CgError) as e:
        run(cg, acts, refs, 2, 2, algo=cg.DRIFT_BULK)
    assert e.value.status == 7


@pytest.mark.parametrize("algo", [2, 3])
def test_drift_bulk_full_size_matches_stream(cg, algo):
    """70B-like workload: the bulk pipelines agree with the streaming kernel."""
    import torch
    from tests._cmp import REL_L2_RTOL
    cfg = SI.SEVENTY_B
    S, N = cfg["n_shards"], cfg["n_canaries"]
    acts, refs, _ = cg.cg_generate_pipeline(cg.PipelineDesc.from_config(cfg))
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    a = cg.cg_drift_scores(acts, refs, S, N, algo=1).cpu().numpy()
    b = cg.cg_drift_scores(acts, refs, S, N, algo=algo, status=st).cpu().numpy()
    assert cg.cg_read_status(st) == (0, 0)
    assert np.all(np.abs(a[0] - b[0]) <= 2 * REL_L2_RTOL * np.abs(a[0]))
    assert np.array_equal(a[1], b[1])
    del acts, refs
    torch.cuda.empty_cache()


@pytest.mark.parametrize("algo", [1, 2])
def test_drift_infinite_and_extreme_live_values(cg, orc, algo):
    """Live values an untrusted hop may send: +inf and -inf (rel_l2 and
    max_abs +inf, cos_dev NaN), the largest finite fp16 (65504) and fp16
    subnormals, against the oracle on the same bytes."""
    import torch
    S, N, L = 2, 4, 4096
    acts, refs = SI.drift_arrays(S, N, L, seed=31)
    h = acts.view(np.float16).copy()
    h[0, 1, 17] = np.inf                       # one +inf element
    h[0, 2, 5] = -np.inf                       # one -inf element
    h[0, 3, 100] = np.inf                      # +inf and -inf in one segment
    h[0, 3, 200] = -np.inf
    h[1, 0, :8] = np.float16(65504.0)          # the largest finite fp16
    h[1, 1, :] = np.float16(6.0e-8)            # subnormal fp16 everywhere
    h[1, 2, ::3] = np.float16(-1.0e-6)         # a mix of subnormals
    refs = refs.copy()
    refs[1, 3, 7] = np.nan                     # a NaN reference element
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    g = run(cg, h.view(np.uint16), refs, S, N, algo=algo, status=st).cpu().numpy()
    o = orc.drift_scores(h.view(np.uint16), refs, S, N)
    assert cg.cg_read_status(st) == (0, 0)
    assert_scores_close(g, o, what=f"algo {algo}")
    for n in (1, 2, 3):
        assert np.isinf(g[0, n, 0]) and np.isinf(g[1, n, 0]) and np.isnan(g[2, n, 0])
    assert np.isnan(g[0, 3, 1]) and np.isnan(g[2, 3, 1]) and np.isfinite(g[1, 3, 1])


@pytest.mark.parametrize("C,S,N,L", [(5, 3, 4, 36864), (3, 2, 5, 16385), (7, 4, 3, 8),
                                     (2, 12, 10, 4096 * 3 + 8), (4, 2, 3, 1)])
def test_drift_batch_matches_oracle(cg, orc, C, S, N, L):
    """cg_drift_scores_batch: C equal-shape configurations in one launch pair
    (the TMA pipeline when L is a multiple of 8, the streaming kernel
    otherwise), each configuration's [3][N][S] block against the oracle and
    against its own single-configuration call."""
    import torch
    acts, refs = SI.drift_arrays(C * S, N, L, seed=C * 100 + S * 10 + N + L)
    d_acts = torch.from_numpy(acts.view(np.float16)).cuda()
    d_refs = torch.from_numpy(refs).cuda()
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    g = cg.cg_drift_scores_batch(d_acts, d_refs, C, S, N, status=st).cpu().numpy()
    assert cg.cg_read_status(st) == (0, 0)
    assert g.shape == (3, C, N, S)
    for c in range(C):
        a, r = acts[c * S:(c + 1) * S], refs[c * S:(c + 1) * S]
        assert_scores_close(g[:, c], orc.drift_scores(a, r, S, N), what=f"batch config {c}")
        if L % 8 == 0:
            # the TMA pipeline's sums do not depend on where a segment sits,
            # so a batched configuration scores exactly as it does alone
            one = cg.cg_drift_scores(d_acts[c * S:(c + 1) * S].clone(),
                                     d_refs[c * S:(c + 1) * S].clone(), S, N)
            assert np.array_equal(g[:, c], one.cpu().numpy()), "batch and single call differ"


@pytest.mark.parametrize("algo", [1, 2])
def test_drift_magnitude_domain(cg, orc, algo):
    """The lower end of the fp32 sums' range (Eq. 4 on tiny activations).
    References of scale 1e-16 (squares normal) and 1e-20 (squares
    subnormal, live values fp16(a) = 0, so h - a = -a exactly and D = A
    term by term) match the oracle: rel_l2 = 1, cos_dev = 0, max_abs exact.
    At scale 1e-24 every square underflows fp32: the documented result is
    rel_l2 and cos_dev NaN (the oracle's fp64 gives 1), which the ranking
    then reports as CG_ERR_NAN_SCORE instead of ranking a wrong value."""
    import torch
    S, N, L = 2, 3, 8192
    rng = np.random.Generator(np.random.PCG64(5))
    base = rng.standard_normal((S, N, L)).astype(np.float64)
    scale = np.array([1e-16, 1e-20, 1e-24])[None, :, None]
    refs = (base * scale).astype(np.float32)
    acts = refs.astype(np.float16).view(np.uint16)            # fp16 rounds all of them to +-0
    assert not (acts & 0x7FFF).any()
    g = run(cg, acts, refs, S, N, algo=algo).cpu().numpy()
    o = orc.drift_scores(acts, refs, S, N)
    ok = [0, 1]                                               # canaries of scale 1e-16, 1e-20
    assert_scores_close(g[:, ok], o[:, ok], what="1e-16 and 1e-20")
    assert np.all(g[0, ok] == 1.0) and np.all(g[2, ok] == 0.0)
    assert np.all(np.isnan(g[0, 2])) and np.all(np.isnan(g[2, 2]))
    assert np.array_equal(g[1, 2], o[1, 2].astype(np.float32))   # max |a| is still exact
    assert np.all(o[0, 2] == 1.0)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    lab = torch.zeros((1, N, S), dtype=torch.int8, device="cuda")
    lab[:, :, 0] = 1
    cg.cg_auroc(torch.from_numpy(g[0]).cuda()[None].contiguous(), lab, status=st)
    assert cg.cg_read_status(st)[0] == 4                     # CG_ERR_NAN_SCORE
