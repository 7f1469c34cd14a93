"""GB300-native canary-trap hot path (arxiv 2607.19490): a thin ctypes binding
over ``libcanary_guard.so`` (declared in ``include/canary_guard.h``).

Functions keep the C names (``cg_generate_pipeline``, ``cg_drift_scores``,
``cg_auroc``, ...).  They only marshal torch CUDA tensors into device
pointers and the current stream; every step of the path runs in the
library's CUDA kernels.  There is no CPU fallback: without the built library
(``paper_2607_19490_gb300.build.build()``) or without a CUDA device every
call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

from .build import LIB_PATH, build  # noqa: F401

__all__ = [
    "CgError", "load", "cg_status_string", "cg_abi_version", "PipelineDesc",
    "cg_philox_words", "cg_philox_normals", "cg_box_muller_pairs", "cg_generate_workspace_size",
    "cg_generate_pipeline", "cg_drift_workspace_size", "cg_drift_scores",
    "cg_drift_scores_ex", "cg_drift_scores_batch", "cg_drift_scores_host",
    "cg_drift_scores_noalloc",
    "cg_make_control_labels", "cg_auroc", "cg_read_status", "cg_generate_recompute",
    "cg_random_scores", "cg_auroc_pooled", "cg_generate_propagating", "cg_selftest_bounded_wait",
    "NOISE_MULT", "NOISE_PAPER", "TAMPER_ADDITIVE", "TAMPER_SIGNFLIP_CHANNELS",
    "TAMPER_SIGNFLIP_FULL", "TAMPER_SCALE",
]

CG_OK = 0
STATUS_NAMES = {0: "CG_OK", 1: "CG_ERR_INVALID_ARG", 2: "CG_ERR_ALIGNMENT", 3: "CG_ERR_WORKSPACE",
                4: "CG_ERR_NAN_SCORE", 5: "CG_ERR_CUDA", 6: "CG_ERR_TIMEOUT",
                7: "CG_ERR_UNSUPPORTED", 8: "CG_ERR_NO_BENIGN"}
NOISE_MULT, NOISE_PAPER = 0, 1
TAMPER_ADDITIVE, TAMPER_SIGNFLIP_CHANNELS, TAMPER_SIGNFLIP_FULL, TAMPER_SCALE = 0, 1, 2, 3
DEVFLAG_NAN_SCORE, DEVFLAG_TIMEOUT, DEVFLAG_NO_BENIGN = 1, 2, 4
DRIFT_AUTO, DRIFT_STREAM, DRIFT_BULK, DRIFT_BULK_2CTA = 0, 1, 2, 3


class CgError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {STATUS_NAMES.get(status, status)}")


class PipelineDesc(ctypes.Structure):
    """Mirror of ``cg_pipeline_desc``."""
    _fields_ = [
        ("n_shards", ctypes.c_uint32), ("hidden", ctypes.c_uint32),
        ("n_canaries", ctypes.c_uint32), ("tokens", ctypes.c_uint32),
        ("malicious", ctypes.POINTER(ctypes.c_int32)), ("n_malicious", ctypes.c_uint32),
        ("noise", ctypes.c_int32), ("benign_sigma", ctypes.c_float),
        ("shard_sigma_lognormal", ctypes.c_float), ("n_outlier", ctypes.c_uint32),
        ("outlier_scale", ctypes.c_float), ("tamper", ctypes.c_int32),
        ("tamper_param", ctypes.c_float), ("seed", ctypes.c_uint64),
        ("config_id", ctypes.c_uint32),
    ]

    @classmethod
    def from_config(cls, cfg: dict) -> "PipelineDesc":
        mal = (ctypes.c_int32 * max(1, len(cfg["malicious"])))(*cfg["malicious"])
        d = cls(cfg["n_shards"], cfg["hidden"], cfg["n_canaries"], cfg["tokens"],
                ctypes.cast(mal, ctypes.POINTER(ctypes.c_int32)), len(cfg["malicious"]),
                cfg["noise"], cfg["benign_sigma"], cfg.get("shard_sigma_lognormal", 0.0),
                cfg.get("n_outlier", 0), cfg.get("outlier_scale", 20.0), cfg["tamper"],
                cfg["tamper_param"], cfg["seed"], cfg.get("config_id", 0))
        d._keep = mal
        return d

    @property
    def seg_len(self) -> int:
        return self.tokens * self.hidden


_lock = threading.Lock()
_lib = None


def load() -> ctypes.CDLL:
    """Load the built library (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                f"{LIB_PATH} is missing: build the CUDA library first "
                "(python -c 'import __graft_entry__ as g; g.build()'); there is no CPU fallback")
        L = ctypes.CDLL(LIB_PATH)
        P, u32, u64, i32, sz = ctypes.c_void_p, ctypes.c_uint32, ctypes.c_uint64, ctypes.c_int32, ctypes.c_size_t
        sigs = {
            "cg_status_string": ([ctypes.c_int], ctypes.c_char_p),
            "cg_abi_version": ([], ctypes.c_int),
            "cg_philox_words": ([u64, u32, u32, u32, u32, u32, P, P], ctypes.c_int),
            "cg_philox_normals": ([u64, u32, u32, u32, u32, u32, P, P], ctypes.c_int),
            "cg_box_muller_pairs": ([P, u64, P, P], ctypes.c_int),
            "cg_generate_workspace_size": ([ctypes.POINTER(PipelineDesc), ctypes.POINTER(sz)], ctypes.c_int),
            "cg_generate_pipeline": ([ctypes.POINTER(PipelineDesc), P, P, P, P, sz, P, P], ctypes.c_int),
            "cg_drift_workspace_size": ([u32, u32, u64, ctypes.POINTER(sz)], ctypes.c_int),
            "cg_generate_recompute": ([ctypes.POINTER(PipelineDesc), u32, P, P, sz, P, P], ctypes.c_int),
            "cg_generate_propagating": ([ctypes.POINTER(PipelineDesc), ctypes.c_float, P, P, P, P, sz, P, P], ctypes.c_int),
            "cg_random_scores": ([u64, u32, u32, u32, u32, P, P], ctypes.c_int),
            "cg_drift_scores": ([P, P, u32, u32, u64, P, u64, P, sz, P, P], ctypes.c_int),
            "cg_drift_scores_ex": ([P, P, u32, u32, u64, P, u64, P, sz, P, ctypes.c_int32, P], ctypes.c_int),
            "cg_drift_scores_batch": ([P, P, u32, u32, u32, u64, P, u64, P, sz, P, P], ctypes.c_int),
            "cg_drift_scores_host": ([P, P, u32, u32, u64, P, u64, P, sz, P, P], ctypes.c_int),
            "cg_drift_scores_noalloc": ([P, P, u32, u32, u64, P, u64, P, P], ctypes.c_int),
            "cg_make_control_labels": ([P, u32, u32, u32, u64, u32, P, P, P], ctypes.c_int),
            "cg_auroc": ([P, P, u32, u32, u32, P, P, P, P, P, P], ctypes.c_int),
            "cg_auroc_pooled": ([P, P, u32, u32, u32, P, P, P, P, P, P], ctypes.c_int),
            "cg_selftest_bounded_wait": ([u32, P, P], ctypes.c_int),
            "cg_read_status": ([P, P, ctypes.POINTER(i32)], ctypes.c_int),
        }
        for name, (args, res) in sigs.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = res
        _lib = L
        return _lib


# --------------------------------------------------------------------------- helpers

def _torch():
    import torch
    return torch


def _check(status: int, where: str):
    if status != CG_OK:
        raise CgError(status, where)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _cuda(t, name, dtypes):
    if t is None:
        return
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    # the library launches on the current device with the current stream
    if t.device.index != _torch().cuda.current_device():
        raise ValueError(f"{name} is on {t.device}, but the current device is "
                         f"cuda:{_torch().cuda.current_device()}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if t.dtype not in dtypes:
        raise ValueError(f"{name} has dtype {t.dtype}, expected one of {dtypes}")


def _stream(stream):
    torch = _torch()
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def cg_status_string(status: int) -> str:
    return load().cg_status_string(status).decode()


def cg_abi_version() -> int:
    return int(load().cg_abi_version())


# --------------------------------------------------------------------------- entry points

def cg_philox_words(seed, c1, c2, c3, first_block, n_blocks, out=None, stream=None):
    """Philox4x32-10 blocks as an int32 tensor [n_blocks, 4] (bit patterns of uint32)."""
    torch = _torch()
    if out is None:
        out = torch.empty((n_blocks, 4), dtype=torch.int32, device="cuda")
    _cuda(out, "out", (torch.int32,))
    if out.numel() < 4 * n_blocks:
        raise ValueError("out must hold 4 * n_blocks words")
    _check(load().cg_philox_words(seed, c1, c2, c3, first_block, n_blocks, _ptr(out),
                                  _stream(stream)), "cg_philox_words")
    return out


def cg_philox_normals(seed, c1, c2, c3, first_block, n_blocks, out=None, stream=None):
    torch = _torch()
    if out is None:
        out = torch.empty((n_blocks, 4), dtype=torch.float32, device="cuda")
    _cuda(out, "out", (torch.float32,))
    if out.numel() < 4 * n_blocks:
        raise ValueError("out must hold 4 * n_blocks floats")
    _check(load().cg_philox_normals(seed, c1, c2, c3, first_block, n_blocks, _ptr(out),
                                    _stream(stream)), "cg_philox_normals")
    return out


def cg_box_muller_pairs(words, out=None, stream=None):
    """Box-Muller of word pairs: words int32 [n, 2] (uint32 bit patterns) on
    the device -> float32 [n, 2] = (z0, z1) per pair."""
    torch = _torch()
    _cuda(words, "words", (torch.int32,))
    if words.numel() % 2 or words.numel() == 0:
        raise ValueError("words must hold a positive even number of words")
    n = words.numel() // 2
    if out is None:
        out = torch.empty((n, 2), dtype=torch.float32, device="cuda")
    _cuda(out, "out", (torch.float32,))
    if out.numel() < 2 * n:
        raise ValueError("out must hold 2 * n floats")
    _check(load().cg_box_muller_pairs(_ptr(words), n, _ptr(out), _stream(stream)),
           "cg_box_muller_pairs")
    return out


def cg_generate_workspace_size(desc: PipelineDesc) -> int:
    n = ctypes.c_size_t()
    _check(load().cg_generate_workspace_size(ctypes.byref(desc), ctypes.byref(n)),
           "cg_generate_workspace_size")
    return n.value


def cg_generate_pipeline(desc: PipelineDesc, acts=None, refs=None, labels=None, ws=None,
                         status=None, stream=None, want_labels=True):
    """Materialise one configuration; returns (acts fp16, refs fp32, labels int8 or None),
    acts/refs shaped [S][N][T*d], labels [N][S]."""
    torch = _torch()
    S, N, L = desc.n_shards, desc.n_canaries, desc.seg_len
    if acts is None:
        acts = torch.empty((S, N, L), dtype=torch.float16, device="cuda")
    if refs is None:
        refs = torch.empty((S, N, L), dtype=torch.float32, device="cuda")
    if labels is None and want_labels:
        labels = torch.empty((N, S), dtype=torch.int8, device="cuda")
    need = cg_generate_workspace_size(desc)
    if ws is None:
        ws = torch.empty(need, dtype=torch.uint8, device="cuda")
    _cuda(acts, "acts", (torch.float16,))
    _cuda(refs, "refs", (torch.float32,))
    _cuda(labels, "labels", (torch.int8,))
    _cuda(ws, "ws", (torch.uint8,))
    _cuda(status, "status", (torch.int32,))
    if acts.numel() != S * N * L or refs.numel() != S * N * L:
        raise ValueError("acts/refs must hold S*N*T*d elements")
    if labels is not None and labels.numel() != N * S:
        raise ValueError("labels must hold N*S elements")
    _check(load().cg_generate_pipeline(ctypes.byref(desc), _ptr(acts), _ptr(refs), _ptr(labels),
                                       _ptr(ws), ws.numel(), _ptr(status), _stream(stream)),
           "cg_generate_pipeline")
    return acts, refs, labels


def cg_generate_recompute(desc: PipelineDesc, replica, out=None, ws=None, status=None,
                          stream=None):
    """Independent benign recompute of every stage as fp32 [S][N][T*d] (the
    redundant-recompute ceiling's and the noisy reference's comparator)."""
    torch = _torch()
    S, N, L = desc.n_shards, desc.n_canaries, desc.seg_len
    if out is None:
        out = torch.empty((S, N, L), dtype=torch.float32, device="cuda")
    if ws is None:
        ws = torch.empty(cg_generate_workspace_size(desc), dtype=torch.uint8, device="cuda")
    _cuda(out, "out", (torch.float32,))
    _cuda(ws, "ws", (torch.uint8,))
    _cuda(status, "status", (torch.int32,))
    if out.numel() != S * N * L:
        raise ValueError("out must hold S*N*T*d elements")
    _check(load().cg_generate_recompute(ctypes.byref(desc), replica, _ptr(out), _ptr(ws),
                                        ws.numel(), _ptr(status), _stream(stream)),
           "cg_generate_recompute")
    return out


def cg_generate_propagating(desc: PipelineDesc, gain, acts=None, refs=None, labels=None, ws=None,
                            status=None, stream=None):
    """Pipeline whose stages inherit gain x the upstream deviation; returns
    (acts fp16, refs fp32, labels int8) like cg_generate_pipeline."""
    torch = _torch()
    S, N, L = desc.n_shards, desc.n_canaries, desc.seg_len
    acts = torch.empty((S, N, L), dtype=torch.float16, device="cuda") if acts is None else acts
    refs = torch.empty((S, N, L), dtype=torch.float32, device="cuda") if refs is None else refs
    labels = torch.empty((N, S), dtype=torch.int8, device="cuda") if labels is None else labels
    ws = (torch.empty(cg_generate_workspace_size(desc), dtype=torch.uint8, device="cuda")
          if ws is None else ws)
    _cuda(acts, "acts", (torch.float16,))
    _cuda(refs, "refs", (torch.float32,))
    _cuda(labels, "labels", (torch.int8,))
    _cuda(ws, "ws", (torch.uint8,))
    _cuda(status, "status", (torch.int32,))
    if acts.numel() != S * N * L or refs.numel() != S * N * L or labels.numel() != N * S:
        raise ValueError("acts/refs must hold S*N*T*d elements and labels N*S")
    _check(load().cg_generate_propagating(ctypes.byref(desc), float(gain), _ptr(acts), _ptr(refs),
                                          _ptr(labels), _ptr(ws), ws.numel(), _ptr(status),
                                          _stream(stream)), "cg_generate_propagating")
    return acts, refs, labels


def cg_random_scores(seed, n_configs, n_canaries, n_shards, config_id0=0, out=None, stream=None):
    """Random-baseline scores fp32 [C][N][S] ~ Uniform(0, 1)."""
    torch = _torch()
    if out is None:
        out = torch.empty((n_configs, n_canaries, n_shards), dtype=torch.float32, device="cuda")
    _cuda(out, "out", (torch.float32,))
    if out.numel() < n_configs * n_canaries * n_shards:
        raise ValueError("out too small")
    _check(load().cg_random_scores(seed, config_id0, n_configs, n_canaries, n_shards, _ptr(out),
                                   _stream(stream)), "cg_random_scores")
    return out


def cg_drift_workspace_size(n_shards, n_canaries, seg_len) -> int:
    n = ctypes.c_size_t()
    _check(load().cg_drift_workspace_size(n_shards, n_canaries, seg_len, ctypes.byref(n)),
           "cg_drift_workspace_size")
    return n.value


def cg_drift_scores(acts, refs, n_shards, n_canaries, scores=None, stat_stride=None, ws=None,
                    status=None, stream=None, algo=None):
    """Drift scores [3][N][S] (rel_l2, max_abs, cos_dev) of acts fp16 / refs fp32 [S][N][L].
    `algo` (DRIFT_*) selects the kernel through cg_drift_scores_ex; None calls cg_drift_scores."""
    torch = _torch()
    _cuda(acts, "acts", (torch.float16,))
    _cuda(refs, "refs", (torch.float32,))
    n_seg = n_shards * n_canaries
    if acts.numel() != refs.numel() or acts.numel() % n_seg:
        raise ValueError("acts and refs must both hold S*N*L elements")
    seg_len = acts.numel() // n_seg
    if scores is None:
        scores = torch.empty((3, n_canaries, n_shards), dtype=torch.float32, device=acts.device)
        stat_stride = n_seg
    if stat_stride is None:
        stat_stride = n_seg
    if ws is None:
        ws = torch.empty(cg_drift_workspace_size(n_shards, n_canaries, seg_len), dtype=torch.uint8,
                         device=acts.device)
    _cuda(scores, "scores", (torch.float32,))
    _cuda(ws, "ws", (torch.uint8,))
    _cuda(status, "status", (torch.int32,))
    if scores.numel() < 2 * stat_stride + n_seg:
        raise ValueError("scores must hold 2 * stat_stride + N * S floats")
    if ws.numel() < cg_drift_workspace_size(n_shards, n_canaries, seg_len):
        raise ValueError("workspace smaller than cg_drift_workspace_size")
    if algo is None:
        _check(load().cg_drift_scores(_ptr(acts), _ptr(refs), n_shards, n_canaries, seg_len,
                                      _ptr(scores), stat_stride, _ptr(ws), ws.numel(), _ptr(status),
                                      _stream(stream)), "cg_drift_scores")
    else:
        _check(load().cg_drift_scores_ex(_ptr(acts), _ptr(refs), n_shards, n_canaries, seg_len,
                                         _ptr(scores), stat_stride, _ptr(ws), ws.numel(),
                                         _ptr(status), int(algo), _stream(stream)),
               "cg_drift_scores_ex")
    return scores


def cg_drift_scores_batch(acts, refs, n_configs, n_shards, n_canaries, scores=None,
                          stat_stride=None, ws=None, status=None, stream=None):
    """Drift scores [3][C][N][S] of C equal-shape configurations, acts fp16 /
    refs fp32 [C][S][N][L], in one launch pair."""
    torch = _torch()
    _cuda(acts, "acts", (torch.float16,))
    _cuda(refs, "refs", (torch.float32,))
    n_seg = n_configs * n_shards * n_canaries
    if acts.numel() != refs.numel() or acts.numel() % n_seg:
        raise ValueError("acts and refs must both hold C*S*N*L elements")
    seg_len = acts.numel() // n_seg
    if scores is None:
        scores = torch.empty((3, n_configs, n_canaries, n_shards), dtype=torch.float32,
                             device=acts.device)
        stat_stride = n_seg
    if stat_stride is None:
        stat_stride = n_seg
    need = cg_drift_workspace_size(n_configs * n_shards, n_canaries, seg_len)
    if ws is None:
        ws = torch.empty(need, dtype=torch.uint8, device=acts.device)
    _cuda(scores, "scores", (torch.float32,))
    _cuda(ws, "ws", (torch.uint8,))
    _cuda(status, "status", (torch.int32,))
    if scores.numel() < 2 * stat_stride + n_seg:
        raise ValueError("scores must hold 2 * stat_stride + C * N * S floats")
    if ws.numel() < need:
        raise ValueError("workspace smaller than cg_drift_workspace_size(C * S, N, L)")
    _check(load().cg_drift_scores_batch(_ptr(acts), _ptr(refs), n_configs, n_shards, n_canaries,
                                        seg_len, _ptr(scores), stat_stride, _ptr(ws), ws.numel(),
                                        _ptr(status), _stream(stream)), "cg_drift_scores_batch")
    return scores


def cg_drift_scores_host(h_acts, refs, n_shards, n_canaries, scores=None, stat_stride=None,
                         ws=None, status=None, stream=None):
    """Drift scores with the live activations in pinned host memory (a CPU
    fp16 tensor with pin_memory=True); the kernel reads them directly over
    the host link and the fp32 references stay on the device."""
    torch = _torch()
    if h_acts.is_cuda or not h_acts.is_pinned():
        raise ValueError("h_acts must be a pinned CPU tensor")
    if not h_acts.is_contiguous() or h_acts.dtype != torch.float16:
        raise ValueError("h_acts must be contiguous float16")
    _cuda(refs, "refs", (torch.float32,))
    n_seg = n_shards * n_canaries
    if h_acts.numel() != refs.numel() or h_acts.numel() % n_seg:
        raise ValueError("h_acts and refs must both hold S*N*L elements")
    seg_len = h_acts.numel() // n_seg
    if scores is None:
        scores = torch.empty((3, n_canaries, n_shards), dtype=torch.float32, device=refs.device)
        stat_stride = n_seg
    if stat_stride is None:
        stat_stride = n_seg
    if ws is None:
        ws = torch.empty(cg_drift_workspace_size(n_shards, n_canaries, seg_len), dtype=torch.uint8,
                         device=refs.device)
    _cuda(scores, "scores", (torch.float32,))
    _cuda(ws, "ws", (torch.uint8,))
    _cuda(status, "status", (torch.int32,))
    if scores.numel() < 2 * stat_stride + n_seg:
        raise ValueError("scores must hold 2 * stat_stride + N * S floats")
    if ws.numel() < cg_drift_workspace_size(n_shards, n_canaries, seg_len):
        raise ValueError("workspace smaller than cg_drift_workspace_size")
    _check(load().cg_drift_scores_host(_ptr(h_acts), _ptr(refs), n_shards, n_canaries, seg_len,
                                       _ptr(scores), stat_stride, _ptr(ws), ws.numel(),
                                       _ptr(status), _stream(stream)), "cg_drift_scores_host")
    return scores


def cg_drift_scores_noalloc(acts, refs, n_shards, n_canaries, scores, stat_stride=None,
                            status=None, stream=None):
    """cg_drift_scores without a workspace, for callers that cannot allocate
    device memory while scoring (for example a verifier living inside an
    inference server whose memory pool owns nearly all of HBM).  The library
    keeps the partial sums in a fixed 4 MiB device array shared by every
    call, so calls must not overlap on the GPU; problems above
    CG_NOALLOC_MAX_WORK_ITEMS chunks of 16384 elements are rejected.  The
    caller passes the output buffer; nothing is allocated here."""
    torch = _torch()
    _cuda(acts, "acts", (torch.float16,))
    _cuda(refs, "refs", (torch.float32,))
    _cuda(scores, "scores", (torch.float32,))
    _cuda(status, "status", (torch.int32,))
    n_seg = n_shards * n_canaries
    if acts.numel() != refs.numel() or acts.numel() % n_seg:
        raise ValueError("acts and refs must both hold S*N*L elements")
    seg_len = acts.numel() // n_seg
    if stat_stride is None:
        stat_stride = n_seg
    if scores.numel() < 2 * stat_stride + n_seg:
        raise ValueError("scores must hold 2 * stat_stride + N * S floats")
    _check(load().cg_drift_scores_noalloc(_ptr(acts), _ptr(refs), n_shards, n_canaries, seg_len,
                                          _ptr(scores), stat_stride, _ptr(status),
                                          _stream(stream)), "cg_drift_scores_noalloc")
    return scores


def cg_make_control_labels(labels, seed, config_id0=0, ctrl=None, status=None, stream=None):
    """Scrambled-label control for labels int8 [C][N][S]."""
    torch = _torch()
    _cuda(labels, "labels", (torch.int8,))
    C, N, S = labels.shape
    if ctrl is None:
        ctrl = torch.empty_like(labels)
    _cuda(ctrl, "ctrl", (torch.int8,))
    _cuda(status, "status", (torch.int32,))
    _check(load().cg_make_control_labels(_ptr(labels), C, N, S, seed, config_id0, _ptr(ctrl),
                                         _ptr(status), _stream(stream)), "cg_make_control_labels")
    return ctrl


def cg_auroc(scores, labels, u2=None, gt=None, eq=None, auroc=None, status=None, stream=None,
             want_counts=True):
    """Mann-Whitney counts and AUROC of scores fp32 / labels int8 [C][N][S].

    Returns dict(u2, gt, eq, auroc) of device tensors (gt/eq None unless wanted)."""
    torch = _torch()
    _cuda(scores, "scores", (torch.float32,))
    _cuda(labels, "labels", (torch.int8,))
    if scores.shape != labels.shape or scores.dim() != 3:
        raise ValueError("scores and labels must both be [C][N][S]")
    C, N, S = scores.shape
    dev = scores.device
    if u2 is None:
        u2 = torch.empty((C, N), dtype=torch.int64, device=dev)
    if want_counts and gt is None:
        gt = torch.empty((C, N), dtype=torch.int64, device=dev)
    if want_counts and eq is None:
        eq = torch.empty((C, N), dtype=torch.int64, device=dev)
    if auroc is None:
        auroc = torch.empty((C,), dtype=torch.float64, device=dev)
    for t, n in ((u2, "u2"), (gt, "gt"), (eq, "eq")):
        _cuda(t, n, (torch.int64,))
    _cuda(auroc, "auroc", (torch.float64,))
    _cuda(status, "status", (torch.int32,))
    _check(load().cg_auroc(_ptr(scores), _ptr(labels), C, N, S, _ptr(u2), _ptr(gt), _ptr(eq),
                           _ptr(auroc), _ptr(status), _stream(stream)), "cg_auroc")
    return {"u2": u2, "gt": gt, "eq": eq, "auroc": auroc}


def cg_auroc_pooled(scores, labels, u2=None, n_mal=None, n_ben=None, auroc=None, status=None,
                    stream=None):
    """Pooled Mann-Whitney AUROC per configuration of scores/labels [C][N][S]."""
    torch = _torch()
    _cuda(scores, "scores", (torch.float32,))
    _cuda(labels, "labels", (torch.int8,))
    if scores.shape != labels.shape or scores.dim() != 3:
        raise ValueError("scores and labels must both be [C][N][S]")
    C, N, S = scores.shape
    dev = scores.device
    u2 = torch.empty((C,), dtype=torch.int64, device=dev) if u2 is None else u2
    n_mal = torch.empty((C,), dtype=torch.int64, device=dev) if n_mal is None else n_mal
    n_ben = torch.empty((C,), dtype=torch.int64, device=dev) if n_ben is None else n_ben
    auroc = torch.empty((C,), dtype=torch.float64, device=dev) if auroc is None else auroc
    for t, n in ((u2, "u2"), (n_mal, "n_mal"), (n_ben, "n_ben")):
        _cuda(t, n, (torch.int64,))
    _cuda(auroc, "auroc", (torch.float64,))
    _cuda(status, "status", (torch.int32,))
    _check(load().cg_auroc_pooled(_ptr(scores), _ptr(labels), C, N, S, _ptr(u2), _ptr(n_mal),
                                  _ptr(n_ben), _ptr(auroc), _ptr(status), _stream(stream)),
           "cg_auroc_pooled")
    return {"u2": u2, "n_mal": n_mal, "n_ben": n_ben, "auroc": auroc}


def cg_selftest_bounded_wait(limit_us, status, stream=None):
    """Run the bounded-wait diagnostic; returns nothing (read `status` afterwards)."""
    torch = _torch()
    _cuda(status, "status", (torch.int32,))
    _check(load().cg_selftest_bounded_wait(int(limit_us), _ptr(status), _stream(stream)),
           "cg_selftest_bounded_wait")


def cg_read_status(status, stream=None):
    """Synchronise and read a device status word: returns (cg_status, raw word)."""
    torch = _torch()
    _cuda(status, "status", (torch.int32,))
    word = ctypes.c_int32()
    st = load().cg_read_status(_ptr(status), _stream(stream), ctypes.byref(word))
    return st, word.value
