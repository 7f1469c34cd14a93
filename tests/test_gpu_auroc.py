"""GPU parity of the ranking test: Mann-Whitney counts (bit-exact), A-hat
(bit-exact) and the scrambled-label control labels (bit-exact) against the
oracle on the same seeded inputs."""
import numpy as np
import pytest

import seeded_inputs as SI

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cg():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_19490_gb300 as m
    m.build()
    return m


def run(cg, scores, labels, status=None):
    import torch
    res = cg.cg_auroc(torch.from_numpy(scores).cuda(), torch.from_numpy(labels).cuda(),
                      status=status)
    return {k: (v.cpu().numpy() if v is not None else None) for k, v in res.items()}


@pytest.mark.parametrize("C,N,S,n_mal,excluded,ties", [
    (1, 1, 2, 1, 0, None), (5, 7, 4, 1, 0, None), (3, 64, 16, 1, 0, 3), (4, 9, 32, 3, 2, 5),
    (2, 5, 33, 2, 0, 4), (2, 3, 100, 7, 5, None), (1, 2, 1024, 10, 3, 6), (324, 64, 16, 1, 0, None),
    (6, 300, 8, 2, 1, 2), (2, 1500, 8, 2, 1, 3), (1, 4097, 16, 3, 2, None),
])
def test_auroc_matches_oracle(cg, orc, C, N, S, n_mal, excluded, ties):
    scores, labels = SI.score_arrays(C, N, S, seed=C + N + S, n_malicious=n_mal,
                                     tie_levels=ties, excluded=excluded)
    g = run(cg, scores, labels)
    o = orc.auroc(scores, labels)
    for k in ("u2", "gt", "eq"):
        assert np.array_equal(g[k], o[k]), k
    assert np.array_equal(g["auroc"].view(np.uint64), o["auroc"].view(np.uint64))


def test_auroc_nonuniform_pairs_bit_exact(cg, orc):
    scores, labels = SI.score_arrays(3, 40, 9, seed=4, n_malicious=2, tie_levels=5)
    labels[:, ::3, 8] = -1
    labels[1, 5, :] = 0
    labels[2, :, :] = 0           # no pair anywhere: A-hat is NaN
    g = run(cg, scores, labels)
    o = orc.auroc(scores, labels)
    assert np.array_equal(g["u2"], o["u2"])
    assert np.array_equal(g["auroc"][:2].view(np.uint64), o["auroc"][:2].view(np.uint64))
    assert np.isnan(g["auroc"][2]) and np.isnan(o["auroc"][2])


@pytest.mark.parametrize("C,N,S,n_mal,excluded,ties", [
    (2437, 37, 10, 2, 1, 4), (2440, 64, 32, 3, 2, None), (2500, 33, 4, 1, 0, 3),
    (2448, 70, 8, 2, 0, None), (2433, 64, 16, 1, 0, 2), (2436, 129, 16, 2, 1, None),
])
def test_auroc_batched_lanes_match_oracle(cg, orc, C, N, S, n_mal, excluded, ties):
    """Batches large enough for the warp-per-8-configurations kernel: partial
    last batch, canary counts that are not a multiple of 64, every SP,
    row-aligned and unaligned loads, ties, excluded stages, non-uniform pair
    counts and a configuration without any pair."""
    scores, labels = SI.score_arrays(C, N, S, seed=C + 3 * N + S, n_malicious=n_mal,
                                     tie_levels=ties, excluded=excluded)
    labels[5, ::3, :] = np.where(labels[5, ::3, :] == 0, -1, labels[5, ::3, :])   # fewer pairs
    labels[9, :, :] = 0                                                           # no pair
    g = run(cg, scores, labels)
    o = orc.auroc(scores, labels)
    for k in ("u2", "gt", "eq"):
        assert np.array_equal(g[k], o[k]), k
    fin = ~np.isnan(o["auroc"])
    assert not fin[9] and np.isnan(g["auroc"][9])
    assert np.array_equal(g["auroc"][fin].view(np.uint64), o["auroc"][fin].view(np.uint64))


@pytest.mark.parametrize("C,N,S,n_mal,excluded,ties", [
    (1216, 64, 16, 1, 0, None), (1300, 4, 4, 1, 0, 2), (1250, 36, 8, 2, 1, 3),
    (1230, 50, 32, 5, 3, None), (1290, 2, 8, 1, 0, None), (1217, 33, 16, 3, 2, 4),
    (3001, 64, 16, 2, 1, 5),
])
def test_auroc_many_small_configurations(cg, orc, C, N, S, n_mal, excluded, ties):
    """Batches of at least 8 configurations per SM with rows of exactly SP
    stages and at most 64 canaries (a warp per configuration, 16-byte row
    loads): every SP, a single canary pair, ties, excluded stages,
    non-uniform pair counts and a configuration without any pair."""
    scores, labels = SI.score_arrays(C, N, S, seed=C + 5 * N + S, n_malicious=n_mal,
                                     tie_levels=ties, excluded=excluded)
    labels[7, ::3, :] = np.where(labels[7, ::3, :] == 0, -1, labels[7, ::3, :])   # fewer pairs
    labels[11, :, :] = 0                                                          # no pair
    g = run(cg, scores, labels)
    o = orc.auroc(scores, labels)
    for k in ("u2", "gt", "eq"):
        assert np.array_equal(g[k], o[k]), k
    fin = ~np.isnan(o["auroc"])
    assert not fin[11] and np.isnan(g["auroc"][11])
    assert np.array_equal(g["auroc"][fin].view(np.uint64), o["auroc"][fin].view(np.uint64))


def test_auroc_stress_batch(cg, orc):
    """65,536 configurations x 64 canaries x 16 stages."""
    rng = np.random.Generator(np.random.PCG64(5))
    C, N, S = 65536, 64, 16
    scores = rng.random((C, N, S), dtype=np.float32)
    labels = np.zeros((C, N, S), np.int8)
    labels[np.arange(C), :, rng.integers(0, S, size=C)] = 1
    g = run(cg, scores, labels)
    o = orc.auroc(scores, labels)
    assert np.array_equal(g["u2"], o["u2"])
    assert np.array_equal(g["auroc"].view(np.uint64), o["auroc"].view(np.uint64))


def test_auroc_nan_flag(cg):
    import torch
    scores, labels = SI.score_arrays(2, 3, 4, seed=1)
    scores[1, 2, 0] = np.nan
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    run(cg, scores, labels, status=st)
    status, word = cg.cg_read_status(st)
    assert status == 4 and word & cg.DEVFLAG_NAN_SCORE


@pytest.mark.parametrize("C,N,S,n_mal", [(1, 50, 4, 1), (3, 64, 16, 2), (2, 7, 33, 5), (4, 9, 1000, 3)])
def test_control_labels_bit_exact(cg, orc, C, N, S, n_mal):
    import torch
    _, labels = SI.score_arrays(C, N, S, seed=S, n_malicious=n_mal, excluded=1)
    ctrl = cg.cg_make_control_labels(torch.from_numpy(labels).cuda(), seed=77, config_id0=9)
    assert np.array_equal(ctrl.cpu().numpy(), orc.control_labels(labels, seed=77, config_id0=9))


def test_control_no_benign_flag(cg):
    import torch
    labels = np.ones((1, 2, 3), np.int8)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    cg.cg_make_control_labels(torch.from_numpy(labels).cuda(), seed=1, status=st)
    status, word = cg.cg_read_status(st)
    assert status == 8 and word == cg.DEVFLAG_NO_BENIGN


@pytest.mark.parametrize("C,N,S,n_mal,excluded,ties", [
    (1, 1, 2, 1, 0, None), (5, 7, 4, 1, 0, None), (3, 64, 16, 1, 0, 3), (4, 9, 32, 3, 2, 5),
    (2, 256, 16, 1, 0, None), (2, 1000, 16, 2, 1, 7), (324, 64, 16, 1, 0, None), (1, 1, 1000, 10, 3, 6),
    (6, 50, 4, 3, 0, 3), (1, 1024, 16, 9, 0, 4), (1000, 32, 8, 5, 1, 3), (2, 16, 8, 2, 0, 1),
    # a warp per configuration (N S <= 1024) with a smaller side above 64 keys
    # (the shared-memory bitonic sort): 512 against 512, and a ragged 1023
    (50, 64, 16, 8, 0, None), (7, 33, 31, 13, 2, 9), (1300, 64, 16, 8, 0, 5),
])
def test_pooled_matches_oracle(cg, orc, C, N, S, n_mal, excluded, ties):
    import torch
    scores, labels = SI.score_arrays(C, N, S, seed=C * 7 + N + S, n_malicious=n_mal,
                                     tie_levels=ties, excluded=excluded)
    g = cg.cg_auroc_pooled(torch.from_numpy(scores).cuda(), torch.from_numpy(labels).cuda())
    o = orc.auroc_pooled(scores, labels)
    for k in ("u2", "n_mal", "n_ben"):
        assert np.array_equal(g[k].cpu().numpy(), o[k]), k
    assert np.array_equal(g["auroc"].cpu().numpy().view(np.uint64), o["auroc"].view(np.uint64))


def test_pooled_signed_zero_and_inf(cg, orc):
    import torch
    scores = np.array([[[0.0, -0.0, np.inf, -np.inf, 1.0, -1.0]]], np.float32)
    labels = np.array([[[1, 0, 1, 0, 0, 1]]], np.int8)
    g = cg.cg_auroc_pooled(torch.from_numpy(scores).cuda(), torch.from_numpy(labels).cuda())
    o = orc.auroc_pooled(scores, labels)
    assert g["u2"].item() == o["u2"][0]
    assert g["auroc"].item() == o["auroc"][0]


def test_pooled_nan_flag(cg, orc):
    import torch
    scores, labels = SI.score_arrays(2, 5, 4, seed=3)
    scores[1, 2, 1] = np.nan
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    g = cg.cg_auroc_pooled(torch.from_numpy(scores).cuda(), torch.from_numpy(labels).cuda(), status=st)
    o = orc.auroc_pooled(scores, labels, allow_nan=True)
    assert cg.cg_read_status(st)[0] == 4
    assert np.array_equal(g["u2"].cpu().numpy(), o["u2"])


@pytest.mark.parametrize("C,N,S", [(2, 5, 8), (1300, 8, 16), (1300, 65, 16), (2, 3, 40),
                                   (1300, 33, 4), (1300, 36, 8)],
                         ids=["block", "lane_config", "lane_config_N65", "wide", "lane_config_S4",
                              "lane_config_S8"])
def test_nan_on_excluded_stages_is_ignored(cg, orc, C, N, S):
    """A NaN score on a stage the labels exclude (-1) is not part of any pair:
    no NaN flag, and counts and A-hat equal the oracle's, on every kernel
    path (per-canary and pooled)."""
    import torch
    scores, labels = SI.score_arrays(C, N, S, seed=C + N + S, n_malicious=1, excluded=2)
    scores[labels == -1] = np.nan
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    g = run(cg, scores, labels, status=st)
    o = orc.auroc(scores, labels)
    assert cg.cg_read_status(st) == (0, 0)
    for k in ("u2", "gt", "eq"):
        assert np.array_equal(g[k], o[k]), k
    assert np.array_equal(g["auroc"].view(np.uint64), o["auroc"].view(np.uint64))
    gp = cg.cg_auroc_pooled(torch.from_numpy(scores).cuda(), torch.from_numpy(labels).cuda(),
                            status=st)
    op = orc.auroc_pooled(scores, labels)
    assert cg.cg_read_status(st) == (0, 0)
    assert np.array_equal(gp["u2"].cpu().numpy(), op["u2"])
    assert np.array_equal(gp["auroc"].cpu().numpy().view(np.uint64), op["auroc"].view(np.uint64))


@pytest.mark.parametrize("C,N,S", [(3, 40, 8), (1300, 8, 16), (1300, 70, 16), (2, 6, 40)],
                         ids=["block", "lane_config", "lane_config_N70", "wide"])
def test_auroc_infinities_and_signed_zero(cg, orc, C, N, S):
    """Scores of +inf (a drift score of an infinite activation), -inf, +0 and
    -0 (equal, a tie) among finite ones: counts and A-hat equal the oracle's
    on every per-canary path."""
    scores, labels = SI.score_arrays(C, N, S, seed=C * 3 + N + S, n_malicious=2, excluded=1,
                                     tie_levels=4)
    rng = np.random.Generator(np.random.PCG64(C + S))
    specials = np.array([np.inf, -np.inf, 0.0, -0.0], np.float32)
    pick = rng.random(scores.shape) < 0.2
    scores[pick] = specials[rng.integers(0, 4, size=int(pick.sum()))]
    g = run(cg, scores, labels)
    o = orc.auroc(scores, labels)
    for k in ("u2", "gt", "eq"):
        assert np.array_equal(g[k], o[k]), k
    assert np.array_equal(g["auroc"].view(np.uint64), o["auroc"].view(np.uint64))
