"""Seeded synthetic inputs shared by the tests and the benchmark.

This module holds workload *descriptions* (shapes, seeds, noise and tamper
parameters) and numpy-drawn random test arrays.  It holds none of the
method's arithmetic: the pipeline generator, the drift statistics and the
AUROC are computed only by the CUDA library and, independently, by the
oracle.  Both sides receive the same description or the same arrays from
here.

Workloads follow the paper's problem statement (k stages of hidden size d,
n canaries of T tokens, a malicious set M, a benign noise level sigma_hw and
a tamper of magnitude eps; Sec. 3.1-3.3) at the shapes of five synthetic
pipelines: a tiny one, a 7B-like one (d = 4096), a 70B-like one (d = 8192),
a 324-configuration factorial sweep and a raised-noise-floor sweep, plus one
at the paper's own experiment shape (k = 12, d = 768, n = 100, T = 48;
Sec. 4.1-4.2).
"""
from __future__ import annotations

import itertools

import numpy as np

NOISE_MULT, NOISE_PAPER = 0, 1
TAMPER_ADDITIVE, TAMPER_SIGNFLIP_CHANNELS, TAMPER_SIGNFLIP_FULL, TAMPER_SCALE = 0, 1, 2, 3


def _cfg(n_shards, hidden, n_canaries, tokens, malicious, noise, benign_sigma,
         tamper, tamper_param, seed, config_id=0, n_outlier=0, outlier_scale=20.0,
         shard_sigma_lognormal=0.0):
    return dict(n_shards=n_shards, hidden=hidden, n_canaries=n_canaries, tokens=tokens,
                malicious=tuple(malicious), noise=noise, benign_sigma=benign_sigma,
                shard_sigma_lognormal=shard_sigma_lognormal, n_outlier=n_outlier,
                outlier_scale=outlier_scale, tamper=tamper, tamper_param=tamper_param,
                seed=seed, config_id=config_id)


# The tiny pipeline: 4 stages, stage 2 (1-based) malicious, d = 256,
# 16 canaries x 32 tokens, relative benign noise 1e-3, 2 outlier channels x20,
# Gaussian tamper with ||delta|| = 0.05 ||a||, seed 0.
TINY = _cfg(4, 256, 16, 32, [1], NOISE_MULT, 1e-3, TAMPER_ADDITIVE, 0.05, seed=0,
            n_outlier=2)

# 7B-like: 8 stages, d = 4096, 64 canaries x 128 tokens, benign noise 1e-3
# (Eq. 2 form), 4 outlier channels x20, one malicious stage (floor(k/2) in
# 1-based numbering -> 0-based 3) with Gaussian tamper 1e-2, seed 1.
SEVEN_B = _cfg(8, 4096, 64, 128, [3], NOISE_PAPER, 1e-3, TAMPER_ADDITIVE, 1e-2, seed=1,
               n_outlier=4)

# 70B-like: 16 stages, d = 8192, 256 canaries x 128 tokens (4.295e9 elements:
# 8.59 GB fp16 live + 17.18 GB fp32 references), benign noise 2e-3, the
# malicious stage (0-based 7) negates a random 1% of channels, seed 2.
SEVENTY_B = _cfg(16, 8192, 256, 128, [7], NOISE_PAPER, 2e-3, TAMPER_SIGNFLIP_CHANNELS,
                 0.01, seed=2)

# The paper's experiment shape: k = 12 blocks of d = 768, n = 100 canaries of
# 48 tokens, sigma_hw = 0.002, Gaussian tamper eps = 0.05 at i* = floor(k/2).
PAPER_SHAPE = _cfg(12, 768, 100, 48, [5], NOISE_PAPER, 2e-3, TAMPER_ADDITIVE, 0.05,
                   seed=5)

FACTORIAL_SHARDS = (4, 8, 16)
FACTORIAL_HIDDEN = (1024, 4096, 8192)
FACTORIAL_TYPES = (TAMPER_ADDITIVE, TAMPER_SIGNFLIP_CHANNELS, TAMPER_SCALE)
FACTORIAL_MAGNITUDES = (1e-3, 1e-2, 1e-1)
FACTORIAL_NOISE = (1e-4, 1e-3)
FACTORIAL_POSITIONS = ("first", "last")
FACTORIAL_SEED = 3
SCALE_FACTOR = 1.05


def factorial_configs(n_canaries=64, tokens=64):
    """All 3*3*3*3*2*2 = 324 configurations, row-major over (stages, hidden,
    tamper type, magnitude, benign noise, malicious position).  The magnitude
    is eps for the Gaussian tamper and the flipped-channel fraction for the
    channel sign flip; the rescale always uses the factor 1.05, its magnitude
    only changes the configuration id (and so its random draws)."""
    out = []
    axes = itertools.product(FACTORIAL_SHARDS, FACTORIAL_HIDDEN, FACTORIAL_TYPES,
                             FACTORIAL_MAGNITUDES, FACTORIAL_NOISE, FACTORIAL_POSITIONS)
    for cid, (S, d, kind, mag, sig, pos) in enumerate(axes):
        mal = [0] if pos == "first" else [S - 1]
        param = SCALE_FACTOR if kind == TAMPER_SCALE else mag
        out.append(_cfg(S, d, n_canaries, tokens, mal, NOISE_PAPER, sig, kind, param,
                        seed=FACTORIAL_SEED, config_id=cid))
    return out


SNR_SEED = 4


def snr_configs(n_canaries=128, tokens=128):
    """Raised noise floor: sigma_j = 10^(-4 + 0.5 j), j = 0..6, per-stage
    lognormal spread 0.5, fixed Gaussian tamper 1e-2, 8 stages, d = 4096."""
    out = []
    for j in range(7):
        sigma = 10.0 ** (-4.0 + 0.5 * j)
        out.append(_cfg(8, 4096, n_canaries, tokens, [3], NOISE_PAPER, sigma,
                        TAMPER_ADDITIVE, 1e-2, seed=SNR_SEED, config_id=j,
                        shard_sigma_lognormal=0.5))
    return out


WORKLOADS = {
    "tiny": TINY,
    "7b": SEVEN_B,
    "70b": SEVENTY_B,
    "paper_shape": PAPER_SHAPE,
}


def n_elements(cfg) -> int:
    return cfg["n_shards"] * cfg["n_canaries"] * cfg["tokens"] * cfg["hidden"]


def shrink(cfg, **over):
    """A copy of a workload with some fields replaced (smaller parity cases)."""
    c = dict(cfg)
    c.update(over)
    return c


# --------------------------------------------------------------------------
# Neutral random arrays for the drift and ranking parity tests.

def drift_arrays(S, N, L, seed, rel=None):
    """fp16 live (as uint16 bits) and fp32 references, both [S][N][L].

    References are standard normals with a few large channels; each live
    segment is the reference plus a Gaussian deviation whose relative size is
    drawn per segment from 1e-4 .. 1 (so the statistics span several decades),
    plus a few fixed special segments: an exact copy, a negated copy, a
    scaled copy, a zero reference and a zero live tensor.
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    refs = rng.standard_normal((S, N, L), dtype=np.float32)
    if L >= 16:
        big = rng.choice(L, size=max(1, L // 64), replace=False)
        refs[:, :, big] *= np.float32(20.0)
    if rel is None:
        rel = 10.0 ** rng.uniform(-4.0, 0.0, size=(S, N, 1))
    noise = rng.standard_normal((S, N, L)).astype(np.float64)
    live = refs.astype(np.float64) + rel * noise * np.sqrt(
        np.mean(refs.astype(np.float64) ** 2, axis=2, keepdims=True))
    specials = [lambda r: r, lambda r: -r, lambda r: 1.05 * r,
                lambda r: np.zeros_like(r)]
    flat = live.reshape(S * N, L)
    rflat = refs.reshape(S * N, L)
    for i, fn in enumerate(specials):
        if i < S * N:
            flat[i] = fn(rflat[i].astype(np.float64))
    if S * N > len(specials):
        rflat[len(specials)] = 0.0          # zero reference, nonzero live
    if S * N > len(specials) + 1:
        rflat[len(specials) + 1] = 0.0      # zero reference and zero live
        flat[len(specials) + 1] = 0.0
    acts = live.astype(np.float16).view(np.uint16)
    return np.ascontiguousarray(acts), np.ascontiguousarray(refs)


def score_arrays(C, N, S, seed, n_malicious=1, tie_levels=None, excluded=0):
    """Scores float32 [C][N][S] and labels int8 [C][N][S] (1/0/-1).

    With tie_levels set, scores are drawn from that many distinct values so
    that ties are frequent.  `excluded` stages per canary get label -1."""
    rng = np.random.Generator(np.random.PCG64(seed))
    if tie_levels:
        scores = rng.integers(0, tie_levels, size=(C, N, S)).astype(np.float32) * np.float32(0.25)
    else:
        scores = rng.random((C, N, S), dtype=np.float32)
    labels = np.zeros((C, N, S), dtype=np.int8)
    for c in range(C):
        for n in range(N):
            perm = rng.permutation(S)
            labels[c, n, perm[:n_malicious]] = 1
            labels[c, n, perm[n_malicious:n_malicious + excluded]] = -1
    return scores, labels


# --------------------------------------------------------------------------
# Substudies around the paper's anchor (Sec. 4.4: Gaussian tamper eps = 0.05,
# full mechanism, sigma_hw = 0.002, three seeds), at the paper's experiment
# shape (k = 12, d = 768, n = 100, T = 48).

SUBSTUDY_SEEDS = (5, 6, 7)


def anchor(**over):
    return shrink(PAPER_SHAPE, **over)


def collusion_positions(k, c):
    """c colluders spaced uniformly over k stages: 1-based floor(j k / (c+1)),
    j = 1..c, as 0-based ids (c = 1 gives floor(k/2), the main experiment's i*)."""
    return tuple((j * k) // (c + 1) - 1 for j in range(1, c + 1))


def collusion_configs(seeds=SUBSTUDY_SEEDS):
    return [anchor(malicious=collusion_positions(12, c), seed=sd, config_id=100 + 10 * c + i)
            for c in (1, 2, 3, 4) for i, sd in enumerate(seeds)]


POSITION_FRACTIONS = (0.0, 0.25, 0.5, 0.75, 1.0)


def position_configs(seeds=SUBSTUDY_SEEDS):
    """i* at five fractions f of the pipeline: 0-based floor(f (k-1) + 1/2)."""
    out = []
    for j, f in enumerate(POSITION_FRACTIONS):
        pos = int(f * 11 + 0.5)
        out += [anchor(malicious=(pos,), seed=sd, config_id=200 + 10 * j + i)
                for i, sd in enumerate(seeds)]
    return out


FRONTIER_EPS = (0.10, 0.05, 0.02, 0.01, 0.005, 0.002, 0.001)


def frontier_configs(seeds=SUBSTUDY_SEEDS):
    """eps from 0.10 down to 0.001 on a 1-2-5 grid at the fixed floor sigma_hw = 0.002."""
    return [anchor(tamper_param=e, seed=sd, config_id=300 + 10 * j + i)
            for j, e in enumerate(FRONTIER_EPS) for i, sd in enumerate(seeds)]


DEPTHS = (2, 4, 6, 8, 10, 12)


def depth_configs(seeds=SUBSTUDY_SEEDS):
    """k in {2, ..., 12} stages with i* = floor(k/2) (1-based)."""
    return [anchor(n_shards=k, malicious=(k // 2 - 1,), seed=sd, config_id=400 + 10 * j + i)
            for j, k in enumerate(DEPTHS) for i, sd in enumerate(seeds)]


PAPER_SNR_SIGMAS = (0.002, 0.005, 0.01, 0.02, 0.05, 0.1, 0.2)


def paper_snr_configs(seeds=SUBSTUDY_SEEDS):
    """The paper's own noise-floor substudy: sigma_hw from 0.002 to 0.2 against eps = 0.05."""
    return [anchor(benign_sigma=sg, seed=sd, config_id=500 + 10 * j + i)
            for j, sg in enumerate(PAPER_SNR_SIGMAS) for i, sd in enumerate(seeds)]


STUDIES = {
    "factorial": factorial_configs,
    "snr": snr_configs,
    "collusion": collusion_configs,
    "position": position_configs,
    "frontier": frontier_configs,
    "depth": depth_configs,
    "paper_snr": paper_snr_configs,
}


PROPAGATION_GAINS = (0.0, 0.5, 0.9, 1.0, 1.2)


def propagation_configs(seeds=SUBSTUDY_SEEDS):
    """Deviations that propagate along the pipeline (Eq. 2's recursion with a
    linearised block gain): gain x {first, middle, last} attacker position."""
    out = []
    for j, gain in enumerate(PROPAGATION_GAINS):
        for p, pos in enumerate((0, 5, 11)):
            out += [dict(anchor(malicious=(pos,), seed=sd, config_id=600 + 30 * j + 10 * p + i),
                         gain=gain) for i, sd in enumerate(seeds)]
    return out


STUDIES["propagation"] = propagation_configs
