"""Whole-workload comparison of the CUDA path with the oracle, on the GPU's own bytes.

run_gpu() drives one configuration through the C ABI on the device: the
generator (Eq. 1-3), the drift scores of every (stage, canary) segment by each
drift kernel (Eq. 4 and the cosine mismatch), the scrambled-label control
(Sec. 4.5), the per-canary AUROC of every statistic and of the control
(Eq. 5-6) and the pooled Mann-Whitney AUROC of relative-L2.

check_against_oracle() then compares all of it with the oracle:
  - one stage at a time, the GPU's fp16 live values and fp32 references are
    copied to the host and compared with the oracle's generator over every
    element (the live-value bound and the normals tolerance of
    tests/_cmp.py);
  - every segment is scored by the oracle on those same GPU bytes, and all
    3 S N scores of each drift kernel are compared with assert_scores_close;
  - the GPU's own fp32 scores are ranked by the oracle, and u2, gt, eq and
    A-hat must equal the GPU's bit for bit, for the true labels of every
    statistic, the control labels (themselves bit-exact against the
    oracle's) and the pooled statistic.
No expected value comes from the CUDA path: the oracle recomputes each one
from the paper's definitions.
"""
import numpy as np

from tests._cmp import assert_live_close, assert_normals_close, assert_scores_close

STATS = ("rel_l2", "max_abs", "cos_dev")
CHUNK_ELEMENTS = 1 << 26          # host comparisons in slices of at most 64 Mi elements


def run_gpu(cg, cfg, ctrl_seed=77, algos=None):
    """Generate one configuration and run every step of the path on the GPU.
    Returns a dict of device tensors; algos lists extra drift kernels
    (cg.DRIFT_*) whose scores are kept beside the default call's."""
    import torch
    S, N = cfg["n_shards"], cfg["n_canaries"]
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    desc = cg.PipelineDesc.from_config(cfg)
    acts, refs, labels = cg.cg_generate_pipeline(desc, status=status)
    scores = {"default": cg.cg_drift_scores(acts, refs, S, N, status=status)}
    for algo in algos or ():
        scores[algo] = cg.cg_drift_scores(acts, refs, S, N, status=status, algo=algo)
    lab = labels[None]
    ctrl = cg.cg_make_control_labels(lab, seed=ctrl_seed, config_id0=cfg["config_id"],
                                     status=status)
    sc = scores["default"]
    ranks = {name: cg.cg_auroc(sc[k][None].contiguous(), lab, status=status)
             for k, name in enumerate(STATS)}
    ranks["control"] = cg.cg_auroc(sc[0][None].contiguous(), ctrl, status=status)
    pooled = (cg.cg_auroc_pooled(sc[0][None].contiguous(), lab, status=status)
              if S * N <= 16384 else None)
    st, word = cg.cg_read_status(status)
    assert st == 0, f"device status word {word}"
    return {"acts": acts, "refs": refs, "labels": labels, "scores": scores, "ctrl": ctrl,
            "ranks": ranks, "pooled": pooled, "ctrl_seed": ctrl_seed}


def _compare_stage_bytes(g_acts, g_refs, o_acts, o_refs, o_coef, what):
    N, L = g_acts.shape
    step = max(1, CHUNK_ELEMENTS // max(L, 1))
    worst, differing = 0, 0
    for n0 in range(0, N, step):
        sl = slice(n0, min(N, n0 + step))
        assert_normals_close(g_refs[sl], o_refs[sl], what=f"{what} references")
        worst = max(worst, assert_live_close(g_acts[sl], o_acts[sl], g_refs[sl], o_refs[sl],
                                             o_coef[sl], what=f"{what} live values"))
        differing += int(np.count_nonzero(g_acts[sl] != o_acts[sl]))
    # rounding decisions that differ are rare (fp32 against fp64 evaluation)
    assert differing <= 1e-2 * g_acts.size, f"{what}: {differing} live values differ"
    return worst


def _same_bits(a, b):
    a = np.ascontiguousarray(a, np.float64)
    b = np.ascontiguousarray(b, np.float64)
    return np.array_equal(a.view(np.uint64), b.view(np.uint64))


def check_against_oracle(orc, cfg, g, check_generator=True):
    """Compare the result of run_gpu with the oracle (see the module text)."""
    S, N = cfg["n_shards"], cfg["n_canaries"]
    D = orc.desc_from_dict(cfg)
    gsc = {k: v.cpu().numpy() for k, v in g["scores"].items()}
    for s in range(S):
        g_acts = g["acts"][s].cpu().numpy().view(np.uint16).reshape(N, -1)
        g_refs = g["refs"][s].cpu().numpy().reshape(N, -1)
        if check_generator:
            o_acts, o_refs, o_coef = orc.generate_stage(D, s)
            _compare_stage_bytes(g_acts, g_refs, o_acts, o_refs, o_coef, f"stage {s}")
            del o_acts, o_refs
        o_sc = orc.drift_scores(g_acts, g_refs, 1, N)[:, :, 0]         # [3][N]
        for name, sc in gsc.items():
            assert_scores_close(sc[:, :, s], o_sc, what=f"stage {s}, drift kernel {name}")

    # labels: 1 on the malicious stages (Sec. 3.2), and the oracle's control
    lab = np.zeros((1, N, S), dtype=np.int8)
    lab[:, :, list(cfg["malicious"])] = 1
    assert np.array_equal(g["labels"].cpu().numpy()[None], lab), "labels"
    o_ctrl = orc.control_labels(lab, seed=g["ctrl_seed"], config_id0=cfg["config_id"])
    assert np.array_equal(g["ctrl"].cpu().numpy(), o_ctrl), "control labels"

    sc = gsc["default"]
    cases = [(name, sc[k], lab) for k, name in enumerate(STATS)]
    cases.append(("control", sc[0], o_ctrl))
    out = {}
    for name, stat, labels in cases:
        o = orc.auroc(stat[None], labels)
        r = g["ranks"][name]
        for key in ("u2", "gt", "eq"):
            assert np.array_equal(r[key].cpu().numpy(), o[key]), f"{name}: {key}"
        a = r["auroc"].cpu().numpy()
        assert _same_bits(a, o["auroc"]), f"{name}: A-hat {a} vs oracle {o['auroc']}"
        out[name] = float(a[0])
    if g["pooled"] is not None:
        o = orc.auroc_pooled(sc[0][None], lab)
        for key in ("u2", "n_mal", "n_ben"):
            assert np.array_equal(g["pooled"][key].cpu().numpy(), o[key]), f"pooled {key}"
        assert _same_bits(g["pooled"]["auroc"].cpu().numpy(), o["auroc"]), "pooled A-hat"
        out["pooled"] = float(o["auroc"][0])
    return out
