"""The verifier step captured in a CUDA graph: generation, drift scores,
control labels and both AUROCs recorded once through the public API and
replayed give the same bits as the eager calls (the library neither
allocates nor synchronises inside these calls)."""
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


@pytest.mark.parametrize("name", ["tiny", "7b_small", "paper_small"])
def test_step_graph_replay_matches_eager(cg, name):
    import torch
    cfg = {"tiny": SI.TINY,
           "7b_small": SI.shrink(SI.SEVEN_B, n_canaries=8, tokens=16),
           "paper_small": SI.shrink(SI.PAPER_SHAPE, n_canaries=12)}[name]
    S, N, L = cfg["n_shards"], cfg["n_canaries"], cfg["tokens"] * cfg["hidden"]
    desc = cg.PipelineDesc.from_config(cfg)
    dev = "cuda"
    acts = torch.empty((S, N, L), dtype=torch.float16, device=dev)
    refs = torch.empty((S, N, L), dtype=torch.float32, device=dev)
    labels = torch.empty((1, N, S), dtype=torch.int8, device=dev)
    ctrl = torch.empty_like(labels)
    gws = torch.empty(cg.cg_generate_workspace_size(desc), dtype=torch.uint8, device=dev)
    dws = torch.empty(cg.cg_drift_workspace_size(S, N, L), dtype=torch.uint8, device=dev)
    scores = torch.empty((3, N, S), dtype=torch.float32, device=dev)
    u2 = torch.empty((1, N), dtype=torch.int64, device=dev)
    auroc = torch.empty((2,), dtype=torch.float64, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)

    def step():
        cg.cg_generate_pipeline(desc, acts, refs, labels[0], gws, status=status)
        cg.cg_drift_scores(acts, refs, S, N, scores=scores, ws=dws, status=status)
        cg.cg_make_control_labels(labels, seed=11, ctrl=ctrl, status=status)
        cg.cg_auroc(scores[0][None], labels, u2=u2, auroc=auroc[0:1], want_counts=False,
                    status=status)
        cg.cg_auroc(scores[0][None], ctrl, u2=u2, auroc=auroc[1:2], want_counts=False,
                    status=status)

    step()                                   # eager (also warms every lazy setup)
    torch.cuda.synchronize()
    eager = [t.clone() for t in (acts, refs, labels, ctrl, scores, u2, auroc)]
    for t in (acts, refs, scores, auroc):
        t.zero_()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        step()
    for t in (acts, refs, scores, auroc):
        t.zero_()
    g.replay()
    torch.cuda.synchronize()
    for a, b in zip(eager, (acts, refs, labels, ctrl, scores, u2, auroc)):
        assert torch.equal(a.view(torch.uint8), b.view(torch.uint8))
    assert cg.cg_read_status(status) == (0, 0)
    assert np.isfinite(auroc.cpu().numpy()).all()


def test_generate_and_score_on_two_streams(cg):
    """One configuration scored on one stream while the next is generated on
    another (separate buffers and workspaces, event-ordered) gives the same
    bits as running both one after the other on a single stream."""
    import torch
    cfgs = [SI.shrink(SI.SEVEN_B, n_canaries=16, tokens=32),
            SI.shrink(SI.SEVEN_B, n_canaries=16, tokens=32, seed=9, tamper=SI.TAMPER_SCALE,
                      tamper_param=1.05)]
    S, N = cfgs[0]["n_shards"], cfgs[0]["n_canaries"]
    L = cfgs[0]["tokens"] * cfgs[0]["hidden"]

    def buffers():
        desc = cg.PipelineDesc.from_config(cfgs[0])
        return {"acts": torch.empty((S, N, L), dtype=torch.float16, device="cuda"),
                "refs": torch.empty((S, N, L), dtype=torch.float32, device="cuda"),
                "labels": torch.empty((1, N, S), dtype=torch.int8, device="cuda"),
                "gws": torch.empty(cg.cg_generate_workspace_size(desc), dtype=torch.uint8,
                                   device="cuda"),
                "dws": torch.empty(cg.cg_drift_workspace_size(S, N, L), dtype=torch.uint8,
                                   device="cuda"),
                "scores": torch.empty((3, N, S), dtype=torch.float32, device="cuda"),
                "auroc": torch.empty((1,), dtype=torch.float64, device="cuda")}

    def generate(b, cfg):
        cg.cg_generate_pipeline(cg.PipelineDesc.from_config(cfg), b["acts"], b["refs"],
                                b["labels"][0], b["gws"])

    def score(b):
        cg.cg_drift_scores(b["acts"], b["refs"], S, N, scores=b["scores"], ws=b["dws"])
        cg.cg_auroc(b["scores"][0][None], b["labels"], auroc=b["auroc"], want_counts=False)

    # reference: one stream, one after the other
    ref = [buffers(), buffers()]
    for b, cfg in zip(ref, cfgs):
        generate(b, cfg)
        score(b)
    torch.cuda.synchronize()
    # overlapped: config 1 generated on s_gen while config 0 is scored on s_score
    run = [buffers(), buffers()]
    s_gen, s_score = torch.cuda.Stream(), torch.cuda.Stream()
    done0, done1 = torch.cuda.Event(), torch.cuda.Event()
    s_gen.wait_stream(torch.cuda.current_stream())
    s_score.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s_gen):
        generate(run[0], cfgs[0])
        done0.record(s_gen)
        generate(run[1], cfgs[1])
        done1.record(s_gen)
    with torch.cuda.stream(s_score):
        s_score.wait_event(done0)
        score(run[0])
        s_score.wait_event(done1)
        score(run[1])
    torch.cuda.synchronize()
    for a, b in zip(ref, run):
        for k in ("acts", "refs", "labels", "scores", "auroc"):
            assert torch.equal(a[k].view(torch.uint8), b[k].view(torch.uint8)), k
