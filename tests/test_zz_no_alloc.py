"""cg_drift_scores_noalloc: the drift scores for callers that cannot allocate
device memory on their scoring path (a verifier embedded in an inference
server whose memory pool already owns nearly all of HBM and offers no
allocator, or a loop that cannot pay the synchronisation cudaMalloc may
cause).  It keeps its partial sums in a fixed device array inside the
library instead of a caller workspace.

The test calls the entry point through the C ABI (ctypes on the built
library) twice in a row, on different inputs, and checks each result against
cg_drift_scores with the drift tolerances of the other tests.  The file's
name sorts last, so a run that stops at the first failure has already run
every other test; it also passes alone in a fresh process."""
import ctypes

import numpy as np
import pytest

import seeded_inputs as SI
from tests._cmp import COS_RTOL, REL_L2_RTOL

pytestmark = pytest.mark.gpu


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


def test_noalloc_matches_workspace_entry_point_twice(cg):
    import torch
    L = cg.load()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    # two different problems back to back: the second must not see the first's scratch
    for S, N, seg_len, seed in [(3, 5, 40003, 11), (4, 16, 8192 * 4, 12)]:
        acts_np, refs_np = SI.drift_arrays(S, N, seg_len, seed=seed)
        acts = torch.from_numpy(acts_np.view(np.float16)).cuda()
        refs = torch.from_numpy(refs_np).cuda()
        expect = cg.cg_drift_scores(acts, refs, S, N).cpu().numpy()
        out = torch.full((3, N, S), float("nan"), dtype=torch.float32, device="cuda")
        st = L.cg_drift_scores_noalloc(ctypes.c_void_p(acts.data_ptr()),
                                       ctypes.c_void_p(refs.data_ptr()), S, N, seg_len,
                                       ctypes.c_void_p(out.data_ptr()), N * S, None, stream)
        assert st == 0, cg.cg_status_string(st)
        torch.cuda.synchronize()
        assert_same_scores(out.cpu().numpy(), expect)


def test_noalloc_rejects_oversize_before_launch(cg):
    L = cg.load()
    fake = ctypes.c_void_p(0x10000)      # never touched: the size check comes first
    # 16 x 256 segments of 2^20 + 1 elements need 16 * 256 * 65 chunks > 262144
    st = L.cg_drift_scores_noalloc(fake, fake, 16, 256, (1 << 20) + 1, fake, 16 * 256, None, None)
    assert st == 7
