"""cg_drift_scores_noalloc: the drift scores for callers that cannot allocate
device memory on their scoring path (a verifier embedded in an inference
server whose memory pool already owns nearly all of HBM and offers no
allocator, or a loop that cannot pay the synchronisation cudaMalloc may
cause).  It keeps its partial sums in a fixed device array inside the
library instead of a caller workspace.

The tests call the entry point through the C ABI (ctypes on the built
library) several times in a row, on different inputs, and check every
result against the fp64 oracle on the same bytes and against
cg_drift_scores, with the drift tolerances of the other tests.  One call
fills the array exactly: the 70B-like shape, 4,096 segments of 2^20
elements = CG_NOALLOC_MAX_WORK_ITEMS chunks, with seeded segments planted at
both ends so the first and the last scratch slots hold known sums.  The
file's name sorts last, so a run that stops at the first failure has already
run every other test; it also passes alone in a fresh process."""
import ctypes

import numpy as np
import pytest

import seeded_inputs as SI
from tests._cmp import COS_RTOL, REL_L2_RTOL, assert_scores_close

pytestmark = pytest.mark.gpu

MAX_WORK_ITEMS = 262144          # CG_NOALLOC_MAX_WORK_ITEMS in include/canary_guard.h
CHUNK = 16384                    # CG_NOALLOC_CHUNK_ELEMENTS


@pytest.fixture(scope="module")
def cg():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_19490_gb300 as m
    m.build()
    return m


def assert_same_scores(g, ref):
    rel_g, rel_r = g[0].astype(np.float64), ref[0].astype(np.float64)
    assert np.array_equal(np.isnan(rel_g), np.isnan(rel_r))
    fin = np.isfinite(rel_r)
    assert np.array_equal(rel_g[~fin], rel_r[~fin], equal_nan=True)
    assert np.all(np.abs(rel_g[fin] - rel_r[fin]) <= REL_L2_RTOL * np.abs(rel_r[fin]))
    assert np.array_equal(g[1], ref[1])
    m2 = np.where(fin, rel_r, 0.0) ** 2 / 2
    cos_g, cos_r = g[2].astype(np.float64), ref[2].astype(np.float64)
    assert np.all(np.abs(cos_g - cos_r) <= COS_RTOL * np.maximum(cos_r, m2) + 1e-12)


def call_noalloc(cg, acts, refs, S, N, seg_len):
    """One call through the C ABI into a NaN-filled output; returns host scores."""
    import torch
    L = cg.load()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    out = torch.full((3, N, S), float("nan"), dtype=torch.float32, device="cuda")
    st = L.cg_drift_scores_noalloc(ctypes.c_void_p(acts.data_ptr()),
                                   ctypes.c_void_p(refs.data_ptr()), S, N, seg_len,
                                   ctypes.c_void_p(out.data_ptr()), N * S, None, stream)
    assert st == 0, cg.cg_status_string(st)
    torch.cuda.synchronize()
    return out.cpu().numpy()


def test_noalloc_matches_oracle_and_workspace_entry_point_twice(cg, orc):
    import torch
    # two different problems back to back: the second must not see the first's scratch
    for S, N, seg_len, seed in [(3, 5, 40003, 11), (4, 16, 8192 * 4, 12)]:
        acts_np, refs_np = SI.drift_arrays(S, N, seg_len, seed=seed)
        acts = torch.from_numpy(acts_np.view(np.float16)).cuda()
        refs = torch.from_numpy(refs_np).cuda()
        got = call_noalloc(cg, acts, refs, S, N, seg_len)
        assert_scores_close(got, orc.drift_scores(acts_np, refs_np, S, N),
                            what=f"no-alloc {S}x{N}x{seg_len} vs oracle")
        assert_same_scores(got, cg.cg_drift_scores(acts, refs, S, N).cpu().numpy())


def test_noalloc_fills_the_whole_array(cg, orc):
    """The 70B-like pipeline (16 x 256 segments of 2^20 elements) is exactly
    CG_NOALLOC_MAX_WORK_ITEMS chunks.  Seeded segments are planted at the
    first and the last segment (the first and the last 64 scratch slots) and
    in between; every segment is scored by the oracle on the GPU's bytes,
    one stage at a time."""
    import torch
    cfg = SI.SEVENTY_B
    S, N, L = cfg["n_shards"], cfg["n_canaries"], cfg["tokens"] * cfg["hidden"]
    assert S * N * (L // CHUNK) == MAX_WORK_ITEMS
    acts, refs, _ = cg.cg_generate_pipeline(cg.PipelineDesc.from_config(cfg), want_labels=False)
    plant_at = [(0, 0), (S // 2, N // 3), (S - 1, N - 2), (S - 1, N - 1)]
    for i, (s, n) in enumerate(plant_at):
        pa, pr = SI.drift_arrays(1, 1, L, seed=700 + i)
        acts[s, n].copy_(torch.from_numpy(pa.view(np.float16).reshape(-1)))
        refs[s, n].copy_(torch.from_numpy(pr.reshape(-1)))
    got = call_noalloc(cg, acts, refs, S, N, L)
    for s in range(S):
        o = orc.drift_scores(acts[s].cpu().numpy().view(np.uint16), refs[s].cpu().numpy(), 1, N)
        assert_scores_close(got[:, :, s], o[:, :, 0], what=f"no-alloc at the cap, stage {s}")
    # a smaller call right after: it must not read the large call's leftovers
    acts_np, refs_np = SI.drift_arrays(2, 3, 3 * CHUNK + 5, seed=13)
    small = call_noalloc(cg, torch.from_numpy(acts_np.view(np.float16)).cuda(),
                         torch.from_numpy(refs_np).cuda(), 2, 3, 3 * CHUNK + 5)
    assert_scores_close(small, orc.drift_scores(acts_np, refs_np, 2, 3), what="after the cap")
    del acts, refs
    torch.cuda.empty_cache()


def test_noalloc_rejects_oversize_before_launch(cg):
    L = cg.load()
    fake = ctypes.c_void_p(0x10000)      # never touched: the size check comes first
    # 16 x 256 segments of 2^20 + 1 elements need 16 * 256 * 65 chunks > 262144
    st = L.cg_drift_scores_noalloc(fake, fake, 16, 256, (1 << 20) + 1, fake, 16 * 256, None, None)
    assert st == 7
    # one chunk over the cap: 262145 segments of one element
    st = L.cg_drift_scores_noalloc(fake, fake, 262145, 1, 1, fake, 262145, None, None)
    assert st == 7
