"""ctypes shim around the fp64 CPU oracle in ``cg_oracle.c``.

TEST INFRASTRUCTURE ONLY: the tests, the package's smoke check and the CPU
baseline leg of ``bench.py`` may import this module; the product library never
does, and this module imports nothing from the product package.

Every function here only marshals numpy arrays into the C oracle; all
arithmetic lives in ``cg_oracle.c`` (fp64, built with ``-ffp-contract=off``).
Parameters that the public API carries as binary32 (sigmas, scales, tamper
magnitudes) are rounded to float32 here before they are widened to double, so
the oracle sees exactly the value the API sees.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "cg_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "libcg_oracle.so")
_lock = threading.Lock()
_lib = None

OR_OK, OR_BAD_ARG, OR_NAN_SCORE, OR_NO_MEMORY = 0, 1, 2, 3
NOISE_MULT, NOISE_PAPER = 0, 1
TAMPER_ADDITIVE, TAMPER_SIGNFLIP_CHANNELS, TAMPER_SIGNFLIP_FULL, TAMPER_SCALE = 0, 1, 2, 3
STREAM_REF, STREAM_NOISE, STREAM_TAMPER, STREAM_AUX = 0, 1, 2, 3
AUX_OUTLIER, AUX_SHARD_SIGMA, AUX_FLIP, AUX_CONTROL, AUX_RANDOM = 1, 2, 3, 4, 5


def build(force: bool = False) -> str:
    """Compile the oracle into ``oracle/_build/libcg_oracle.so`` with gcc."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math",
           "-fopenmp", "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class _Desc(ctypes.Structure):
    _fields_ = [
        ("n_shards", ctypes.c_uint32), ("hidden", ctypes.c_uint32),
        ("n_canaries", ctypes.c_uint32), ("tokens", ctypes.c_uint32),
        ("malicious", ctypes.POINTER(ctypes.c_int32)),
        ("n_malicious", ctypes.c_uint32),
        ("noise", ctypes.c_int32),
        ("benign_sigma", ctypes.c_double),
        ("shard_sigma_lognormal", ctypes.c_double),
        ("n_outlier", ctypes.c_uint32),
        ("outlier_scale", ctypes.c_double),
        ("tamper", ctypes.c_int32),
        ("tamper_param", ctypes.c_double),
        ("seed", ctypes.c_uint64),
        ("config_id", ctypes.c_uint32),
    ]


def _p(a, ctype):
    return None if a is None else a.ctypes.data_as(ctypes.POINTER(ctype))


def lib():
    global _lib
    with _lock:
        if _lib is None:
            _lib = ctypes.CDLL(build())
            L = _lib
            u32, u64, i32, dbl = ctypes.c_uint32, ctypes.c_uint64, ctypes.c_int32, ctypes.c_double
            P = ctypes.POINTER
            L.or_philox4x32_10.argtypes = [P(u32), P(u32), P(u32)]
            L.or_philox_words.argtypes = [u64, u32, u32, u32, u32, u32, P(u32)]
            L.or_box_muller.argtypes = [u32, u32, P(dbl), P(dbl)]
            L.or_box_muller_pairs.argtypes = [P(u32), u64, P(dbl)]
            L.or_philox_normals.argtypes = [u64, u32, u32, u32, u32, u32, P(dbl)]
            L.or_aux_bounded.argtypes = [u64, u32, u32, u32, u32, u32, P(u32)]
            L.or_half_from_double.argtypes = [dbl]
            L.or_half_from_double.restype = ctypes.c_uint16
            L.or_half_to_double.argtypes = [ctypes.c_uint16]
            L.or_half_to_double.restype = dbl
            L.or_config_tables.argtypes = [P(_Desc), P(u32), P(dbl), P(ctypes.c_ubyte)]
            L.or_config_tables.restype = i32
            L.or_generate_segment.argtypes = [P(_Desc), u32, u32, P(ctypes.c_float), P(dbl),
                                              P(ctypes.c_uint16), P(dbl)]
            L.or_generate_segment.restype = i32
            L.or_generate_pipeline.argtypes = [P(_Desc), P(ctypes.c_uint16), P(ctypes.c_float),
                                               P(ctypes.c_int8), ctypes.c_int]
            L.or_generate_pipeline.restype = i32
            L.or_drift_segment.argtypes = [P(ctypes.c_uint16), P(ctypes.c_float), u64, P(dbl), P(dbl)]
            L.or_drift_scores.argtypes = [P(ctypes.c_uint16), P(ctypes.c_float), u32, u32, u64,
                                          P(dbl), u64, ctypes.c_int]
            L.or_auroc.argtypes = [P(ctypes.c_float), P(ctypes.c_int8), u32, u32, u32,
                                   P(ctypes.c_int64), P(ctypes.c_int64), P(ctypes.c_int64),
                                   P(ctypes.c_int64), P(dbl)]
            L.or_auroc.restype = i32
            L.or_control_labels.argtypes = [P(ctypes.c_int8), u32, u32, u32, u64, u32, P(ctypes.c_int8)]
            L.or_control_labels.restype = i32
            L.or_max_threads.restype = ctypes.c_int
            L.or_generate_recompute.argtypes = [P(_Desc), u32, P(ctypes.c_float), ctypes.c_int]
            L.or_generate_recompute.restype = i32
            L.or_random_scores.argtypes = [u64, u32, u32, u32, u32, P(ctypes.c_float)]
            L.or_auroc_pooled.argtypes = [P(ctypes.c_float), P(ctypes.c_int8), u32, u32, u32,
                                          P(ctypes.c_int64), P(ctypes.c_int64), P(ctypes.c_int64),
                                          P(dbl)]
            L.or_auroc_pooled.restype = i32
            L.or_generate_propagating.argtypes = [P(_Desc), dbl, P(ctypes.c_uint16), P(ctypes.c_float),
                                                  ctypes.c_int]
            L.or_generate_propagating.restype = i32
            L.or_generate_segments.argtypes = [P(_Desc), u64, u64, P(ctypes.c_uint16),
                                               P(ctypes.c_float), P(dbl), ctypes.c_int]
            L.or_generate_segments.restype = i32
        return _lib


class OracleError(RuntimeError):
    pass


def _check(status):
    if status != OR_OK:
        raise OracleError(f"oracle status {status}")


def max_threads() -> int:
    return int(lib().or_max_threads())


# --------------------------------------------------------------------------
# Philox and normals

def philox4x32_10(ctr, key):
    """One Philox4x32-10 block: ``ctr`` 4 words, ``key`` 2 words."""
    c = np.ascontiguousarray(ctr, dtype=np.uint32)
    k = np.ascontiguousarray(key, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib().or_philox4x32_10(_p(c, ctypes.c_uint32), _p(k, ctypes.c_uint32), _p(out, ctypes.c_uint32))
    return out


def philox_words(seed, c1, c2, c3, first_block, n_blocks):
    out = np.zeros(4 * n_blocks, dtype=np.uint32)
    lib().or_philox_words(seed, c1, c2, c3, first_block, n_blocks, _p(out, ctypes.c_uint32))
    return out


def box_muller(x0, x1):
    z0, z1 = ctypes.c_double(), ctypes.c_double()
    lib().or_box_muller(int(x0), int(x1), ctypes.byref(z0), ctypes.byref(z1))
    return z0.value, z1.value


def box_muller_pairs(words):
    """Box-Muller of word pairs: words uint32 [n, 2] -> float64 [n, 2]."""
    w = np.ascontiguousarray(words, dtype=np.uint32).reshape(-1, 2)
    out = np.zeros(w.shape, dtype=np.float64)
    lib().or_box_muller_pairs(_p(w, ctypes.c_uint32), w.shape[0], _p(out, ctypes.c_double))
    return out


def philox_normals(seed, c1, c2, c3, first_block, n_blocks):
    out = np.zeros(4 * n_blocks, dtype=np.float64)
    lib().or_philox_normals(seed, c1, c2, c3, first_block, n_blocks, _p(out, ctypes.c_double))
    return out


def aux_bounded(seed, purpose, sub, config_id, n, count):
    out = np.zeros(count, dtype=np.uint32)
    lib().or_aux_bounded(seed, purpose, sub, config_id, n, count, _p(out, ctypes.c_uint32))
    return out


def half_from_double(x: float) -> int:
    return int(lib().or_half_from_double(float(x)))


def half_to_double(h: int) -> float:
    return float(lib().or_half_to_double(int(h)))


# --------------------------------------------------------------------------
# Pipeline generation

def _f32(x) -> float:
    return float(np.float32(x))


def make_desc(n_shards, hidden, n_canaries, tokens, malicious=(), noise=NOISE_PAPER,
              benign_sigma=1e-3, shard_sigma_lognormal=0.0, n_outlier=0,
              outlier_scale=20.0, tamper=TAMPER_ADDITIVE, tamper_param=1e-2,
              seed=0, config_id=0):
    """Build the oracle's description; keeps the malicious array alive."""
    mal = np.ascontiguousarray(list(malicious), dtype=np.int32)
    d = _Desc(n_shards, hidden, n_canaries, tokens,
              mal.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)) if len(mal) else None,
              len(mal), noise, _f32(benign_sigma), _f32(shard_sigma_lognormal),
              n_outlier, _f32(outlier_scale), tamper, _f32(tamper_param), seed, config_id)
    d._keep = mal
    return d


def desc_from_dict(cfg: dict):
    return make_desc(**cfg)


def config_tables(desc):
    S, d = desc.n_shards, desc.hidden
    outl = np.zeros(max(desc.n_outlier, 1), dtype=np.uint32)
    sig = np.zeros(S, dtype=np.float64)
    flip = np.zeros((S, d), dtype=np.uint8)
    _check(lib().or_config_tables(ctypes.byref(desc), _p(outl, ctypes.c_uint32),
                                  _p(sig, ctypes.c_double), _p(flip, ctypes.c_ubyte)))
    return outl[:desc.n_outlier].copy(), sig, flip.astype(bool)


def generate_segment(desc, s, n):
    """(refs fp32, pre-rounding live fp64, acts as binary16 bits, coef)."""
    L = desc.tokens * desc.hidden
    refs = np.zeros(L, dtype=np.float32)
    pre = np.zeros(L, dtype=np.float64)
    acts = np.zeros(L, dtype=np.uint16)
    coef = ctypes.c_double()
    _check(lib().or_generate_segment(ctypes.byref(desc), s, n, _p(refs, ctypes.c_float),
                                     _p(pre, ctypes.c_double), _p(acts, ctypes.c_uint16),
                                     ctypes.byref(coef)))
    return refs, pre, acts, coef.value


def generate_pipeline(desc, n_threads=0):
    """acts (uint16 binary16 bits) and refs (float32), both [S][N][T*d]; labels [N][S]."""
    S, N, L = desc.n_shards, desc.n_canaries, desc.tokens * desc.hidden
    acts = np.zeros((S, N, L), dtype=np.uint16)
    refs = np.zeros((S, N, L), dtype=np.float32)
    labels = np.zeros((N, S), dtype=np.int8)
    _check(lib().or_generate_pipeline(ctypes.byref(desc), _p(acts, ctypes.c_uint16),
                                      _p(refs, ctypes.c_float), _p(labels, ctypes.c_int8),
                                      int(n_threads)))
    return acts, refs, labels


def generate_segments(desc, first, count, n_threads=0):
    """Segments first .. first + count - 1 (segment q = s * N + n): acts
    (uint16 binary16 bits) and refs (float32), both [count][T*d], equal to
    that slice of generate_pipeline, and each segment's scalar coef [count]
    (sigma_s mu under Eq. 2 noise, eps ||a|| / ||g|| under the Gaussian
    tamper, else 0; as generate_segment returns it)."""
    L = desc.tokens * desc.hidden
    acts = np.zeros((count, L), dtype=np.uint16)
    refs = np.zeros((count, L), dtype=np.float32)
    coef = np.zeros(count, dtype=np.float64)
    _check(lib().or_generate_segments(ctypes.byref(desc), first, count,
                                      _p(acts, ctypes.c_uint16), _p(refs, ctypes.c_float),
                                      _p(coef, ctypes.c_double), int(n_threads)))
    return acts, refs, coef


def generate_stage(desc, s, n_threads=0):
    """Every canary of stage s: acts uint16 and refs float32 [N][T*d], coef [N]."""
    N = desc.n_canaries
    return generate_segments(desc, s * N, N, n_threads)


def generate_coefs(desc, n_threads=0):
    """The whole pipeline as generate_segments gives it: acts, refs
    [S][N][T*d] and coef [S][N]."""
    S, N, L = desc.n_shards, desc.n_canaries, desc.tokens * desc.hidden
    acts, refs, coef = generate_segments(desc, 0, S * N, n_threads)
    return acts.reshape(S, N, L), refs.reshape(S, N, L), coef.reshape(S, N)


def generate_propagating(desc, gain, n_threads=0):
    """Pipeline whose stages inherit the upstream deviation with `gain`
    (binary32 value): acts uint16 and refs float32 [S][N][T*d]."""
    S, N, L = desc.n_shards, desc.n_canaries, desc.tokens * desc.hidden
    acts = np.zeros((S, N, L), dtype=np.uint16)
    refs = np.zeros((S, N, L), dtype=np.float32)
    _check(lib().or_generate_propagating(ctypes.byref(desc), _f32(gain), _p(acts, ctypes.c_uint16),
                                         _p(refs, ctypes.c_float), int(n_threads)))
    return acts, refs


def generate_recompute(desc, replica, n_threads=0):
    """Independent benign recompute of every stage: fp32 values of fp16
    outputs [S][N][T*d] (the ceiling's and the noisy reference's comparator)."""
    S, N, L = desc.n_shards, desc.n_canaries, desc.tokens * desc.hidden
    out = np.zeros((S, N, L), dtype=np.float32)
    _check(lib().or_generate_recompute(ctypes.byref(desc), replica, _p(out, ctypes.c_float),
                                       int(n_threads)))
    return out


def random_scores(seed, C, N, S, config_id0=0):
    """Random-baseline scores float32 [C][N][S], Uniform(0, 1)."""
    out = np.zeros((C, N, S), dtype=np.float32)
    lib().or_random_scores(seed, config_id0, C, N, S, _p(out, ctypes.c_float))
    return out


# --------------------------------------------------------------------------
# Drift, AUROC, control

def drift_segment(acts, refs):
    """[rel_l2, max_abs, cos_dev] and the sums [D, A, H, M] of one segment."""
    a = np.ascontiguousarray(acts, dtype=np.uint16).ravel()
    r = np.ascontiguousarray(refs, dtype=np.float32).ravel()
    assert a.size == r.size
    out = np.zeros(3, dtype=np.float64)
    sums = np.zeros(4, dtype=np.float64)
    lib().or_drift_segment(_p(a, ctypes.c_uint16), _p(r, ctypes.c_float), a.size,
                           _p(out, ctypes.c_double), _p(sums, ctypes.c_double))
    return out, sums


def drift_scores(acts, refs, n_shards, n_canaries, n_threads=0):
    """scores [3][N][S] (rel_l2, max_abs, cos_dev) in fp64 for acts/refs [S][N][L]."""
    a = np.ascontiguousarray(acts, dtype=np.uint16).ravel()
    r = np.ascontiguousarray(refs, dtype=np.float32).ravel()
    S, N = n_shards, n_canaries
    L = a.size // (S * N)
    assert a.size == r.size == S * N * L
    out = np.zeros((3, N, S), dtype=np.float64)
    lib().or_drift_scores(_p(a, ctypes.c_uint16), _p(r, ctypes.c_float), S, N, L,
                          _p(out, ctypes.c_double), N * S, int(n_threads))
    return out


def auroc(scores, labels):
    """scores float32 [C][N][S], labels int8 [C][N][S] -> dict of counts and A-hat [C]."""
    sc = np.ascontiguousarray(scores, dtype=np.float32)
    lb = np.ascontiguousarray(labels, dtype=np.int8)
    assert sc.shape == lb.shape and sc.ndim == 3
    C, N, S = sc.shape
    u2 = np.zeros((C, N), dtype=np.int64)
    gt = np.zeros((C, N), dtype=np.int64)
    eq = np.zeros((C, N), dtype=np.int64)
    pairs = np.zeros((C, N), dtype=np.int64)
    A = np.zeros(C, dtype=np.float64)
    st = lib().or_auroc(_p(sc, ctypes.c_float), _p(lb, ctypes.c_int8), C, N, S,
                        _p(u2, ctypes.c_int64), _p(gt, ctypes.c_int64), _p(eq, ctypes.c_int64),
                        _p(pairs, ctypes.c_int64), _p(A, ctypes.c_double))
    if st == OR_NAN_SCORE:
        raise OracleError("NaN score among labelled stages")
    _check(st)
    return {"u2": u2, "gt": gt, "eq": eq, "pairs": pairs, "auroc": A}


def auroc_pooled(scores, labels, allow_nan=False):
    """Pooled Mann-Whitney over all canaries of each configuration:
    dict(u2, n_mal, n_ben, auroc) per configuration."""
    sc = np.ascontiguousarray(scores, dtype=np.float32)
    lb = np.ascontiguousarray(labels, dtype=np.int8)
    C, N, S = sc.shape
    u2 = np.zeros(C, np.int64)
    nm = np.zeros(C, np.int64)
    nb = np.zeros(C, np.int64)
    A = np.zeros(C, np.float64)
    st = lib().or_auroc_pooled(_p(sc, ctypes.c_float), _p(lb, ctypes.c_int8), C, N, S,
                               _p(u2, ctypes.c_int64), _p(nm, ctypes.c_int64),
                               _p(nb, ctypes.c_int64), _p(A, ctypes.c_double))
    if st == OR_NAN_SCORE and not allow_nan:
        raise OracleError("NaN score among labelled stages")
    if st not in (OR_OK, OR_NAN_SCORE):
        _check(st)
    return {"u2": u2, "n_mal": nm, "n_ben": nb, "auroc": A}


def control_labels(labels, seed, config_id0=0):
    lb = np.ascontiguousarray(labels, dtype=np.int8)
    C, N, S = lb.shape
    out = np.zeros_like(lb)
    _check(lib().or_control_labels(_p(lb, ctypes.c_int8), C, N, S, seed, config_id0,
                                   _p(out, ctypes.c_int8)))
    return out
