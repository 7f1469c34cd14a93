#!/usr/bin/env python3
"""Benchmark of the canary-trap verifier hot path on GB300.

One step = one pass of the verifier over one synthetic pipeline already
resident in HBM: the drift reduction of every (stage, canary) segment
(relative-L2 of Eq. 4, max-abs, cosine mismatch), the scrambled-label
control labels (Sec. 4.5) and the Mann-Whitney AUROC (Eq. 5-6) of the true
and the control labels.  The pipeline itself (fp32 references and fp16 live
activations) is materialised on the device by the generator before the timed
region; its own throughput is reported under "generate".

Output: one JSON line (rank 0).  `value` = canary activation elements scored
per second over all ranks.  `roofline` is the drift kernel's algorithmic HBM
bytes (6 per element: 2 fp16 + 4 fp32, each read once) per launch over its
CUDA-event duration, against the measured copy bandwidth.  `e2e` repeats the
step with the inputs in pinned host memory, copied in every step, and the
scores and A-hat copied back.  `cpu_baseline` times the fp64 CPU oracle on a
bounded sample of the same workload.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload 70b|7b|paper_shape|tiny]
  python bench.py --impl reference ...   (times the CPU oracle as the reference arm)
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import seeded_inputs as SI  # noqa: E402

WORKLOAD_NAMES = {
    "70b": "70B-like pipeline: 16 stages x hidden 8192, 256 canaries x 128 tokens, fp16 live / fp32 "
           "references, benign noise 2e-3 (Eq. 2), stage 8 (1-based) flips the sign of 1% of channels, seed 2",
    "7b": "7B-like pipeline: 8 stages x hidden 4096, 64 canaries x 128 tokens, 4 outlier channels x20, "
          "benign noise 1e-3 (Eq. 2), Gaussian tamper 1e-2 on stage 4 (1-based), seed 1",
    "paper_shape": "paper-shape pipeline: 12 stages x hidden 768, 100 canaries x 48 tokens, sigma_hw 2e-3, "
                   "Gaussian tamper 0.05 on stage 6 (1-based), seed 5",
    "tiny": "tiny pipeline: 4 stages x hidden 256, 16 canaries x 32 tokens, seed 0",
}
WORKLOADS = {"70b": SI.SEVENTY_B, "7b": SI.SEVEN_B, "paper_shape": SI.PAPER_SHAPE, "tiny": SI.TINY}
METRIC = "canary activation elements scored/sec (HBM GB/s vs peak); AUROC configs/sec"
BYTES_PER_ELEMENT = 6          # 2 B fp16 live + 4 B fp32 reference, each read once
L2_BYTES = 129 * 2**20
NOMINAL_HBM_GBPS = 8000.0      # GB300 HBM3e, nominal


def parse_args(argv=None):
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=int(os.environ.get("WORLD_SIZE", "1")))
    p.add_argument("--steps", type=int, default=100)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--workload", default="70b", choices=sorted(WORKLOADS))
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--e2e-steps", type=int, default=25,
                   help="timed end-to-end steps (25 x ~40 ms: about a second)")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--cpu-seconds", type=float, default=10.0,
                   help="target duration of the timed CPU-oracle sample")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--drift-algo", default="auto", choices=["auto", "stream", "bulk", "bulk2"],
                   help="drift kernel (cg_drift_scores_ex); auto = cg_drift_scores")
    p.add_argument("--study", default=None, choices=sorted(SI.STUDIES),
                   help="run a whole study (generate + score + rank every configuration) and "
                        "report configurations/s instead of the default step")
    return p.parse_args(argv)


# ----------------------------------------------------------------------------- ranks

class Ranks:
    """One process per GPU (torchrun); timing = max over ranks."""

    def __init__(self):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None

    def init(self, backend):
        if self.world > 1:
            import torch.distributed as dist
            os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
            dist.init_process_group(backend=backend)
            self.pg = dist

    def barrier(self):
        if self.pg:
            self.pg.barrier()

    def max(self, x: float) -> float:
        if not self.pg:
            return x
        import torch
        dev = "cuda" if self.pg.get_backend() == "nccl" else "cpu"
        t = torch.tensor([x], dtype=torch.float64, device=dev)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def sum(self, x: float) -> float:
        if not self.pg:
            return x
        import torch
        dev = "cuda" if self.pg.get_backend() == "nccl" else "cpu"
        t = torch.tensor([x], dtype=torch.float64, device=dev)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.SUM)
        return float(t.item())

    def close(self):
        if self.pg:
            self.pg.destroy_process_group()


def rank_config(cfg: dict, rank: int) -> dict:
    """Weak scaling: rank r scores its own independent pipeline (config id + r)."""
    return SI.shrink(cfg, config_id=cfg["config_id"] + rank)


# ----------------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, FileNotFoundError):
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=2)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for name, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ----------------------------------------------------------------------------- peaks

def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


KERNEL_REGIONS = {
    # kernel -> (source file, first line of its region, text that ends the region)
    "drift_bulk_kernel": ("drift.cu", "// ----------------------------------------------------------------- TMA bulk pipeline",
                          "template <int NS>\nstatic cudaError_t launch_bulk"),
    "drift_partial_kernel": ("drift.cu", "constexpr int kUnroll = 4;",
                             "// Scores of one segment from its fp64 sums."),
}


def kernel_source_hash(kernel: str) -> str:
    """sha256 of the source region that defines `kernel` (its device code)."""
    fname, start, end = KERNEL_REGIONS[kernel]
    src = open(os.path.join(ROOT, "paper_2607_19490_gb300", "csrc", fname)).read()
    i = src.index(start)
    j = src.index(end, i)
    return hashlib.sha256(src[i:j].encode()).hexdigest()


def recorded_traffic(kernel: str, profile_name: str):
    """DRAM bytes per launch recorded by the committed ncu summary, when the
    kernel's source region still has the hash recorded there; else None."""
    path = os.path.join(ROOT, "profiles", profile_name)
    try:
        text = open(path).read()
    except OSError:
        return None
    m_t = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", text)
    m_h = re.search(r"kernel_source_sha256:\s*([0-9a-f]{64})", text)
    if not (m_t and m_h) or kernel_source_hash(kernel) != m_h.group(1):
        return None
    return float(m_t.group(1))


# ----------------------------------------------------------------------------- CPU oracle

def oracle_prepare(cfg, n_threads):
    """A bounded sample of the workload for the fp64 CPU oracle: every stage x
    the first few canaries (about 256 Mi elements at most), generated by the
    oracle's own generator (untimed)."""
    from oracle import oracle as O
    O.build()
    S, L = cfg["n_shards"], cfg["tokens"] * cfg["hidden"]
    n_can = max(1, min(cfg["n_canaries"], (256 * 2**20) // (S * L)))
    sub = SI.shrink(cfg, n_canaries=n_can)
    acts, refs, labels = O.generate_pipeline(O.desc_from_dict(sub), n_threads=n_threads)
    return {"acts": acts, "refs": refs, "labels": labels, "S": S, "n": n_can, "L": L}


def oracle_pass(sample, n_threads):
    """One pass of the oracle verifier over the sample: drift scores + AUROC."""
    from oracle import oracle as O
    sc = O.drift_scores(sample["acts"], sample["refs"], sample["S"], sample["n"],
                        n_threads=n_threads)
    O.auroc(sc[0].astype(np.float32)[None], sample["labels"][None])


def oracle_describe(sample, passes, seconds):
    S, n, L = sample["S"], sample["n"], sample["L"]
    e = S * n * L
    return (f"{S} stages x {n} canaries x {L} elements ({e} elements, "
            f"{e * BYTES_PER_ELEMENT / 1e9:.2f} GB) of the workload, generated by the oracle; "
            f"drift scores + AUROC in fp64, {passes} passes in {seconds:.1f} s")


def oracle_baseline(cfg, n_threads, seconds):
    """Time the oracle on the sample, repeating passes until `seconds` elapse
    on all `n_threads` cores; then one pass over a one-canary slice of the
    sample on a single core."""
    sample = oracle_prepare(cfg, n_threads)
    elems = sample["S"] * sample["n"] * sample["L"]
    passes, t0 = 0, time.perf_counter()
    while True:
        oracle_pass(sample, n_threads)
        passes += 1
        el = time.perf_counter() - t0
        if el >= seconds:
            break
    one = {"acts": np.ascontiguousarray(sample["acts"][:, :1]),
           "refs": np.ascontiguousarray(sample["refs"][:, :1]),
           "labels": np.ascontiguousarray(sample["labels"][:1]), "S": sample["S"], "n": 1,
           "L": sample["L"]}
    t1 = time.perf_counter()
    oracle_pass(one, 1)
    el1 = time.perf_counter() - t1
    return {"value": elems * passes / el, "unit": "elements/s", "cores": n_threads,
            "kind": "oracle", "sample": oracle_describe(sample, passes, el),
            "single_core": {"value": one["S"] * one["L"] / el1, "unit": "elements/s",
                            "sample": oracle_describe(one, 1, el1)},
            "auroc": oracle_auroc_baseline()}


def oracle_auroc_baseline(C=65536, N=64, S=16):
    """The oracle's brute-force Mann-Whitney counts and A-hat (single-threaded
    C) on the AUROC stress batch's shape: C configurations x N canaries x S
    stages of uniform scores, stage 0 malicious, drawn on the host."""
    from oracle import oracle as O
    rng = np.random.Generator(np.random.PCG64(7))
    scores = rng.random((C, N, S), dtype=np.float32)
    labels = np.zeros((C, N, S), dtype=np.int8)
    labels[:, :, 0] = 1
    t0 = time.perf_counter()
    O.auroc(scores, labels)
    el = time.perf_counter() - t0
    return {"value": C / el, "unit": "configs/s", "cores": 1, "kind": "oracle",
            "sample": f"the stress batch's shape: {C} configurations x {N} canaries x {S} stages, "
                      f"one pass in {el:.2f} s"}


def run_reference(args, ranks: Ranks):
    """The reference arm: the fp64 CPU oracle, one pass over the bounded
    sample per step, on all host cores."""
    if ranks.rank != 0:
        return
    cfg = WORKLOADS[args.workload]
    from oracle import oracle as O
    O.build()
    threads = O.max_threads()
    sample = oracle_prepare(cfg, threads)
    elems = sample["S"] * sample["n"] * sample["L"]
    for _ in range(args.warmup):
        oracle_pass(sample, threads)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        oracle_pass(sample, threads)
        times.append(time.perf_counter() - t0)
    value = elems / statistics.median(times)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "elements/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1000 * statistics.mean(times), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD_NAMES[args.workload],
                   "sample": oracle_describe(sample, args.steps, sum(times))},
        "cpu_baseline": {"value": value, "unit": "elements/s", "cores": threads,
                         "kind": "oracle", "sample": oracle_describe(sample, args.steps, sum(times))},
        "e2e": {"value": value, "unit": "elements/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------- GPU arm

def run_ours(args, ranks: Ranks):
    import torch
    import paper_2607_19490_gb300 as cg

    if not torch.cuda.is_available():
        raise RuntimeError("bench.py needs a CUDA device (no CPU fallback)")
    torch.cuda.set_device(ranks.local)
    cg.build()
    cfg = rank_config(WORKLOADS[args.workload], ranks.rank)
    S, N, T, d = cfg["n_shards"], cfg["n_canaries"], cfg["tokens"], cfg["hidden"]
    L = T * d
    E = S * N * L
    dev = torch.device("cuda", ranks.local)
    stream = torch.cuda.current_stream()

    # ---- resident inputs: materialised on the device by the generator
    desc = cg.PipelineDesc.from_config(cfg)
    acts = torch.empty((S, N, L), dtype=torch.float16, device=dev)
    refs = torch.empty((S, N, L), dtype=torch.float32, device=dev)
    labels = torch.empty((1, N, S), dtype=torch.int8, device=dev)
    gws = torch.empty(cg.cg_generate_workspace_size(desc), dtype=torch.uint8, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    gen_ms = []
    for i in range(2):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        cg.cg_generate_pipeline(desc, acts, refs, labels[0], gws, status=status)
        e1.record(stream)
        torch.cuda.synchronize()
        gen_ms.append(e0.elapsed_time(e1))
    del gws

    scores = torch.empty((3, 1, N, S), dtype=torch.float32, device=dev)
    dws = torch.empty(cg.cg_drift_workspace_size(S, N, L), dtype=torch.uint8, device=dev)
    ctrl = torch.empty((1, N, S), dtype=torch.int8, device=dev)
    outs = {k: torch.empty((1, N), dtype=torch.int64, device=dev) for k in ("u2", "gt", "eq")}
    outs_c = {k: torch.empty((1, N), dtype=torch.int64, device=dev) for k in ("u2", "gt", "eq")}
    auroc = torch.empty((2,), dtype=torch.float64, device=dev)
    # drift (pipeline kernel + finalize), control labels, and two AUROC calls
    # of one configuration
    launches_per_step = 2 + 1 + 2 * auroc_launches(N, S)

    algo = {"auto": None, "stream": cg.DRIFT_STREAM, "bulk": cg.DRIFT_BULK,
            "bulk2": cg.DRIFT_BULK_2CTA}[args.drift_algo]

    def step(i, ev=None):
        if ev is not None:
            ev[0].record(stream)
        cg.cg_drift_scores(acts, refs, S, N, scores=scores, stat_stride=N * S, ws=dws,
                           status=status, algo=algo)
        if ev is not None:
            ev[1].record(stream)
        cg.cg_make_control_labels(labels, seed=1000 + i, ctrl=ctrl, status=status)
        rel = scores[0]
        cg.cg_auroc(rel, labels, u2=outs["u2"], gt=outs["gt"], eq=outs["eq"], auroc=auroc[0:1],
                    status=status)
        cg.cg_auroc(rel, ctrl, u2=outs_c["u2"], gt=outs_c["gt"], eq=outs_c["eq"],
                    auroc=auroc[1:2], status=status)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    drift_events = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                    for _ in range(args.steps)]
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(ranks.local)
    clocks.start()
    time.sleep(0.3)
    ranks.barrier()
    torch.cuda.synchronize()
    t_start.record(stream)
    for i in range(args.steps):
        step(args.warmup + i, drift_events[i])
    t_end.record(stream)
    torch.cuda.synchronize()
    ranks.barrier()
    clk = clocks.stop()
    total_ms = ranks.max(t_start.elapsed_time(t_end))
    drift_ms = [a.elapsed_time(b) for a, b in drift_events]
    st, word = cg.cg_read_status(status)
    if st != 0:
        raise RuntimeError(f"device status {word} after the timed steps")
    auroc_true, auroc_ctrl = auroc.cpu().tolist()

    total_elems = ranks.sum(float(E)) * args.steps
    value = total_elems / (total_ms / 1e3)
    peak, peak_kind = measured_peaks()
    drift_avg_ms = statistics.mean(drift_ms)
    achieved = E * BYTES_PER_ELEMENT / (drift_avg_ms / 1e3) / 1e9
    # cg_drift_scores picks the TMA bulk pipeline for device-resident inputs
    # whose segments are a multiple of 8 elements
    drift_kernel = ("drift_partial_kernel" if args.drift_algo == "stream" or L % 8
                    else "drift_bulk_kernel")
    traffic = (recorded_traffic(drift_kernel, f"{drift_kernel}_{args.workload}.txt")
               if args.drift_algo in ("auto", "stream", "bulk") else None)

    # ---- AUROC batches (configs/s): the factorial batch and a stress batch
    auroc_rates = auroc_batches(cg, torch, dev, stream)

    # ---- end to end with host buffers
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(cg, torch, dev, stream, acts, refs, labels, S, N, L, args, ranks)
    del acts, refs
    torch.cuda.empty_cache()

    cpu = None
    if ranks.rank == 0 and ranks.world == 1 and not args.no_cpu_baseline:
        from oracle import oracle as O
        cpu = oracle_baseline(WORKLOADS[args.workload], O.max_threads(), args.cpu_seconds)

    if ranks.rank != 0:
        return
    gen_best = min(gen_ms)
    line = {
        "metric": METRIC,
        "value": value,
        "unit": "elements/s",
        "n_gpus": ranks.world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": total_ms / args.steps,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f32",
        "data": "synthetic",
        "config": {
            "workload": WORKLOAD_NAMES[args.workload], "n_shards": S, "hidden": d,
            "n_canaries": N, "tokens": T, "elements_per_step": E,
            "bytes_read_per_step": E * BYTES_PER_ELEMENT,
            "l2": f"inputs {E * BYTES_PER_ELEMENT / 1e9:.1f} GB per step, larger than the "
                  f"{L2_BYTES / 2**20:.0f} MB L2; no flush",
            "step": "drift scores (2 kernels) + control labels + AUROC true and control",
        },
        "roofline": {
            "kernel": drift_kernel + " (+ drift_finalize_kernel inside the same events)",
            "bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
            "frac": achieved / peak, "peak_kind": f"{peak_kind} copy bandwidth",
            # the measured peak is a read+write copy; this kernel only reads, so
            # its fraction can pass 1.  Beside it, the fraction of the nominal
            # HBM3e bandwidth the workload targets (about 8 TB/s)
            "nominal_peak": NOMINAL_HBM_GBPS, "frac_of_nominal": achieved / NOMINAL_HBM_GBPS,
            "traffic": traffic,
            "algorithmic_bytes_per_launch": E * BYTES_PER_ELEMENT,
            "launch_ms_mean": drift_avg_ms, "launch_ms_min": min(drift_ms),
        },
        "auroc": {"true_labels": auroc_true, "control": auroc_ctrl, **auroc_rates},
        "generate": {
            "ms": gen_best, "elements_per_s": E / (gen_best / 1e3),
            "write_GBps": E * BYTES_PER_ELEMENT / (gen_best / 1e3) / 1e9,
        },
        "e2e": e2e,
        "cpu_baseline": cpu,
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clk,
    }
    print(json.dumps(line), flush=True)


def auroc_batches(cg, torch, dev, stream):
    out = {}
    g = torch.Generator(device=dev)
    g.manual_seed(7)
    for name, C, N, S in (("factorial_batch", 324, 64, 16), ("stress_batch", 65536, 64, 16)):
        scores = torch.rand((C, N, S), generator=g, device=dev, dtype=torch.float32)
        labels = torch.zeros((C, N, S), dtype=torch.int8, device=dev)
        labels[:, :, 0] = 1
        res = {k: torch.empty((C, N), dtype=torch.int64, device=dev) for k in ("u2",)}
        au = torch.empty((C,), dtype=torch.float64, device=dev)
        for _ in range(3):
            cg.cg_auroc(scores, labels, u2=res["u2"], auroc=au, want_counts=False)
        reps = 20
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            cg.cg_auroc(scores, labels, u2=res["u2"], auroc=au, want_counts=False)
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / reps
        out[f"{name}_configs_per_s"] = C / (ms / 1e3)
        out[f"{name}_ms"] = ms
        if name == "stress_batch":
            # algorithmic bytes: every score (4 B) and label (1 B) read once,
            # u2 (8 B per canary) and A-hat (8 B per configuration) written
            read = C * N * S * 5
            written = C * N * 8 + C * 8
            peak, _ = measured_peaks()
            out["stress_batch_read_GBps"] = read / (ms / 1e3) / 1e9
            out["stress_batch_GBps"] = (read + written) / (ms / 1e3) / 1e9
            out["stress_batch_frac"] = (read + written) / (ms / 1e3) / 1e9 / peak
        if name == "factorial_batch":
            # the same call replayed from a CUDA graph: the kernels' own time,
            # without the host's per-call cost
            try:
                gr = torch.cuda.CUDAGraph()
                with torch.cuda.graph(gr):
                    cg.cg_auroc(scores, labels, u2=res["u2"], auroc=au, want_counts=False)
                gr.replay()
                torch.cuda.synchronize()
                e0.record(stream)
                for _ in range(reps):
                    gr.replay()
                e1.record(stream)
                torch.cuda.synchronize()
                gms = e0.elapsed_time(e1) / reps
                out[f"{name}_graph_configs_per_s"] = C / (gms / 1e3)
                out[f"{name}_graph_ms"] = gms
            except Exception as exc:       # capture unsupported here: the eager figure stands
                out[f"{name}_graph_error"] = f"{type(exc).__name__}: {exc}"[:200]
        if name == "stress_batch":
            # the pooled Mann-Whitney statistic: per configuration the smaller
            # side's keys sorted, the larger side's bound-searched in them
            pu = {k: torch.empty((C,), dtype=torch.int64, device=dev) for k in ("u2", "nm", "nb")}
            pa = torch.empty((C,), dtype=torch.float64, device=dev)
            for _ in range(3):
                cg.cg_auroc_pooled(scores, labels, u2=pu["u2"], n_mal=pu["nm"], n_ben=pu["nb"],
                                   auroc=pa)
            e0.record(stream)
            for _ in range(reps):
                cg.cg_auroc_pooled(scores, labels, u2=pu["u2"], n_mal=pu["nm"], n_ben=pu["nb"],
                                   auroc=pa)
            e1.record(stream)
            torch.cuda.synchronize()
            pms = e0.elapsed_time(e1) / reps
            out["pooled_stress_batch_configs_per_s"] = C / (pms / 1e3)
            out["pooled_stress_batch_ms"] = pms
            out["pooled_stress_batch_read_GBps"] = C * N * S * 5 / (pms / 1e3) / 1e9
            # the random baseline's scores (Sec. 4.5) of the same shape: one
            # Philox block per four scores, 4 B written per score
            rs = torch.empty_like(scores)
            for _ in range(3):
                cg.cg_random_scores(11, C, N, S, out=rs)
            e0.record(stream)
            for _ in range(reps):
                cg.cg_random_scores(11, C, N, S, out=rs)
            e1.record(stream)
            torch.cuda.synchronize()
            rms = e0.elapsed_time(e1) / reps
            out["random_scores_stress_batch_ms"] = rms
            out["random_scores_stress_batch_write_GBps"] = C * N * S * 4 / (rms / 1e3) / 1e9
            del rs
        del scores, labels
    return out


def run_e2e(cg, torch, dev, stream, acts, refs, labels, S, N, L, args, ranks):
    """End to end through the public API with host buffers.

    Every step, the live fp16 activations (the step's input, returned by the
    untrusted pipeline) are read from pinned host memory by
    cg_drift_scores_host -- the kernel streams them over the host link in its
    single pass -- against the fp32 references resident in HBM (the
    verifier's stored references, Sec. 3.3); then the control labels and both
    AUROCs run and the scores and A-hat are copied back to pinned host memory.
    A second figure streams the references from host memory as well."""
    h_acts = torch.empty(acts.shape, dtype=acts.dtype, pin_memory=True)
    h_acts.copy_(acts)
    h_scores = torch.empty((3, N, S), dtype=torch.float32, pin_memory=True)
    h_auroc = torch.empty((2,), dtype=torch.float64, pin_memory=True)
    scores = torch.empty((3, N, S), dtype=torch.float32, device=dev)
    dws = torch.empty(cg.cg_drift_workspace_size(S, N, L), dtype=torch.uint8, device=dev)
    ctrl = torch.empty_like(labels)
    auroc = torch.empty((2,), dtype=torch.float64, device=dev)

    def step(i):
        cg.cg_drift_scores_host(h_acts, refs, S, N, scores=scores, ws=dws)
        cg.cg_make_control_labels(labels, seed=5000 + i, ctrl=ctrl)
        cg.cg_auroc(scores[0][None], labels, auroc=auroc[0:1], want_counts=False)
        cg.cg_auroc(scores[0][None], ctrl, auroc=auroc[1:2], want_counts=False)
        h_scores.copy_(scores, non_blocking=True)
        h_auroc.copy_(auroc, non_blocking=True)

    def timed(fn, steps):
        fn(0)
        torch.cuda.synchronize()
        ranks.barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(steps):
            fn(i + 1)
        e1.record(stream)
        torch.cuda.synchronize()
        return ranks.max(e0.elapsed_time(e1)) / steps

    elems = ranks.sum(float(S * N * L))
    d2h = h_scores.numel() * 4 + h_auroc.numel() * 8
    ms = timed(step, args.e2e_steps)
    if not np.isfinite(h_auroc.numpy()).all():
        raise RuntimeError("e2e produced a non-finite A-hat")
    h2d = acts.numel() * acts.element_size()
    out = {"value": elems / (ms / 1e3), "unit": "elements/s", "h2d_bytes_per_step": h2d,
           "d2h_bytes_per_step": d2h, "ms_per_step": ms, "steps": args.e2e_steps,
           "link_GBps": h2d / (ms / 1e3) / 1e9,
           "inputs": "live fp16 activations read from pinned host memory every step by "
                     "cg_drift_scores_host; fp32 references resident in HBM"}

    # the same step with an explicit copy-engine transfer of the live
    # activations (cudaMemcpyAsync into device memory) before the drift pass
    def step_copy(i):
        acts.copy_(h_acts, non_blocking=True)
        cg.cg_drift_scores(acts, refs, S, N, scores=scores, ws=dws)
        cg.cg_make_control_labels(labels, seed=5000 + i, ctrl=ctrl)
        cg.cg_auroc(scores[0][None], labels, auroc=auroc[0:1], want_counts=False)
        cg.cg_auroc(scores[0][None], ctrl, auroc=auroc[1:2], want_counts=False)
        h_scores.copy_(scores, non_blocking=True)
        h_auroc.copy_(auroc, non_blocking=True)

    variant_steps = max(1, min(args.e2e_steps, 10))
    ms_copy = timed(step_copy, variant_steps)
    out["memcpy_variant"] = {"value": elems / (ms_copy / 1e3), "unit": "elements/s",
                             "h2d_bytes_per_step": h2d, "ms_per_step": ms_copy,
                             "steps": variant_steps,
                             "link_GBps": h2d / (ms_copy / 1e3) / 1e9,
                             "inputs": "live activations copied with cudaMemcpyAsync, then the "
                                       "device-resident drift pass"}

    h_refs = torch.empty(refs.shape, dtype=refs.dtype, pin_memory=True)
    h_refs.copy_(refs)

    def step_all(i):
        refs.copy_(h_refs, non_blocking=True)
        step(i)

    ms2 = timed(step_all, variant_steps)
    h2d2 = h2d + refs.numel() * refs.element_size()
    out["all_inputs_streamed"] = {"value": elems / (ms2 / 1e3), "unit": "elements/s",
                                  "h2d_bytes_per_step": h2d2, "ms_per_step": ms2,
                                  "steps": variant_steps,
                                  "link_GBps": h2d2 / (ms2 / 1e3) / 1e9}
    del h_acts, h_refs
    return out


# ----------------------------------------------------------------------------- studies

STUDY_METRIC = "AUROC configs/sec (whole study: generate, score and rank every configuration)"


STUDY_BATCH_ELEMENTS = 1 << 29      # elements per drift launch in a study (3.2 GB at 6 B each)


def study_batches(configs):
    """Consecutive runs of configurations with one shape (stages, canaries,
    segment length) and at most STUDY_BATCH_ELEMENTS elements in all (a
    larger configuration stands alone).  A run is generated into one buffer
    and scored by one cg_drift_scores_batch launch pair."""
    out, key_of_run = [], None
    for i, c in enumerate(configs):
        key = (c["n_shards"], c["n_canaries"], c["tokens"] * c["hidden"])
        if (out and key == key_of_run
                and (len(out[-1]) + 1) * SI.n_elements(c) <= STUDY_BATCH_ELEMENTS):
            out[-1].append(i)
        else:
            out.append([i])
            key_of_run = key
    return out


def id_runs(configs, idx):
    """Split a batch into runs of consecutive config ids: (first position,
    end position) pairs; one control-label call serves each run."""
    runs, j = [], 0
    while j < len(idx):
        k = j + 1
        while k < len(idx) and configs[idx[k]]["config_id"] == configs[idx[k - 1]]["config_id"] + 1:
            k += 1
        runs.append((j, k))
        j = k
    return runs


def study_pass(cg, torch, configs, batches, bufs, res, drift_events=None, overlap=True):
    """Every configuration of a study on the device, one batch of equal-shape
    configurations at a time: generate each into the batch's buffer, one
    batched drift launch pair, control labels, per-canary AUROC of rel_l2 /
    max_abs / cos_dev and of the control, pooled AUROC of rel_l2, each over
    the whole batch.  res[k, c] = A-hat k of configuration c.

    overlap: batch b + 1 is generated on one stream while batch b is scored
    on another, in alternating pipeline buffers (the generator is bound by
    integer/FP32 issue, the scoring by HBM, and the generator leaves room on
    every SM for a drift block).  The passes fork from and join back into the
    current stream, so a CUDA graph capture of a pass holds both streams."""
    main = torch.cuda.current_stream()
    if overlap:
        s_gen, s_score = bufs["s_gen"], bufs["s_score"]
        s_gen.wait_stream(main)
        s_score.wait_stream(main)
    else:
        s_gen = s_score = main
    for k, idx in enumerate(batches):
        c0, B = idx[0], len(idx)
        cfg0 = configs[c0]
        S, N, L = cfg0["n_shards"], cfg0["n_canaries"], cfg0["tokens"] * cfg0["hidden"]
        E = S * N * L
        b = k % 2 if overlap else 0
        acts = bufs["acts"][b][:B * E].view(B, S, N, L)
        refs = bufs["refs"][b][:B * E].view(B, S, N, L)
        labels = bufs["labels"][b][:B * N * S].view(B, N, S)
        ctrl = bufs["ctrl"][:B * N * S].view(B, N, S)
        with torch.cuda.stream(s_gen):
            if overlap and k >= 2:
                s_gen.wait_event(bufs["scored"][b])      # buffer b is free once batch k - 2 is scored
            for j, i in enumerate(idx):
                cfg = configs[i]
                desc = cg.PipelineDesc.from_config(cfg)
                if cfg.get("gain", 0.0):
                    cg.cg_generate_propagating(desc, cfg["gain"], acts[j], refs[j], labels[j],
                                               bufs["gws"], status=bufs["status"])
                else:
                    cg.cg_generate_pipeline(desc, acts[j], refs[j], labels[j], bufs["gws"],
                                            status=bufs["status"])
            if overlap:
                bufs["generated"][b].record(s_gen)
        with torch.cuda.stream(s_score):
            if overlap:
                s_score.wait_event(bufs["generated"][b])
            scores = bufs["scores"][:3 * B * N * S].view(3, B, N, S)
            if drift_events is not None:
                drift_events[k][0].record(s_score)
            cg.cg_drift_scores_batch(acts, refs, B, S, N, scores=scores, ws=bufs["dws"],
                                     status=bufs["status"])
            if drift_events is not None:
                drift_events[k][1].record(s_score)
            for j0, j1 in id_runs(configs, idx):
                cg.cg_make_control_labels(labels[j0:j1], seed=7000,
                                          config_id0=configs[idx[j0]]["config_id"],
                                          ctrl=ctrl[j0:j1], status=bufs["status"])
            u2 = bufs["u2"][:B * N].view(B, N)
            for st in range(3):
                cg.cg_auroc(scores[st], labels, u2=u2, auroc=res[st, c0:c0 + B],
                            want_counts=False, status=bufs["status"])
            cg.cg_auroc(scores[0], ctrl, u2=u2, auroc=res[3, c0:c0 + B], want_counts=False,
                        status=bufs["status"])
            cg.cg_auroc_pooled(scores[0], labels, u2=bufs["pu2"][:B], n_mal=bufs["pnm"][:B],
                               n_ben=bufs["pnb"][:B], auroc=res[4, c0:c0 + B],
                               status=bufs["status"])
            if overlap:
                bufs["scored"][b].record(s_score)
    if overlap:
        main.wait_stream(s_gen)
        main.wait_stream(s_score)


def run_study(args, ranks: Ranks):
    import torch
    import paper_2607_19490_gb300 as cg

    torch.cuda.set_device(ranks.local)
    cg.build()
    configs = [rank_config(c, ranks.rank) for c in SI.STUDIES[args.study]()]
    batches = study_batches(configs)
    dev = torch.device("cuda", ranks.local)
    stream = torch.cuda.current_stream()

    def per_batch(fn):
        return max(fn(configs[idx[0]], len(idx)) for idx in batches)

    maxE = per_batch(lambda c, B: B * SI.n_elements(c))
    maxNS = per_batch(lambda c, B: B * c["n_canaries"] * c["n_shards"])
    maxN = per_batch(lambda c, B: B * c["n_canaries"])
    maxB = max(len(idx) for idx in batches)
    gws = max(cg.cg_generate_workspace_size(cg.PipelineDesc.from_config(c)) for c in configs)
    dws = per_batch(lambda c, B: cg.cg_drift_workspace_size(B * c["n_shards"], c["n_canaries"],
                                                            c["tokens"] * c["hidden"]))
    bufs = {
        # two pipeline buffers: one being generated while the other is scored
        "acts": [torch.empty(maxE, dtype=torch.float16, device=dev) for _ in range(2)],
        "refs": [torch.empty(maxE, dtype=torch.float32, device=dev) for _ in range(2)],
        "labels": [torch.empty(maxNS, dtype=torch.int8, device=dev) for _ in range(2)],
        "s_gen": torch.cuda.Stream(device=dev),
        "s_score": torch.cuda.Stream(device=dev),
        "generated": [torch.cuda.Event() for _ in range(2)],
        "scored": [torch.cuda.Event() for _ in range(2)],
        "ctrl": torch.empty(maxNS, dtype=torch.int8, device=dev),
        "scores": torch.empty(3 * maxNS, dtype=torch.float32, device=dev),
        "u2": torch.empty(maxN, dtype=torch.int64, device=dev),
        "pu2": torch.empty(maxB, dtype=torch.int64, device=dev),
        "pnm": torch.empty(maxB, dtype=torch.int64, device=dev),
        "pnb": torch.empty(maxB, dtype=torch.int64, device=dev),
        "gws": torch.empty(gws, dtype=torch.uint8, device=dev),
        "dws": torch.empty(dws, dtype=torch.uint8, device=dev),
        "status": torch.zeros(1, dtype=torch.int32, device=dev),
    }
    res = torch.empty((5, len(configs)), dtype=torch.float64, device=dev)
    for _ in range(max(1, args.warmup)):
        study_pass(cg, torch, configs, batches, bufs, res)
    torch.cuda.synchronize()
    clocks = ClockSampler(ranks.local)
    clocks.start()
    ranks.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = max(1, args.steps)
    e0.record(stream)
    for _ in range(reps):
        study_pass(cg, torch, configs, batches, bufs, res)
    e1.record(stream)
    torch.cuda.synchronize()
    ms_eager = ranks.max(e0.elapsed_time(e1)) / reps
    # the same pass captured once as a CUDA graph and replayed: every kernel
    # of every configuration still runs, without the host's per-launch cost
    graph, graph_error = None, None
    try:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            study_pass(cg, torch, configs, batches, bufs, res)
        eager_res = res.clone()
        res.fill_(-1.0)
        g.replay()
        torch.cuda.synchronize()
        if not torch.equal(res.view(torch.int64), eager_res.view(torch.int64)):
            raise RuntimeError("the replayed graph's A-hat values differ from the eager pass")
        graph = g
    except Exception as exc:           # capture unsupported here: the eager figure stands
        graph_error = f"{type(exc).__name__}: {exc}"[:200]
        torch.cuda.synchronize()
    ms = ms_eager
    if graph is not None:
        ranks.barrier()
        e0.record(stream)
        for _ in range(reps):
            graph.replay()
        e1.record(stream)
        torch.cuda.synchronize()
        ms = ranks.max(e0.elapsed_time(e1)) / reps
    ranks.barrier()
    clk = clocks.stop()
    st, word = cg.cg_read_status(bufs["status"])
    if st != 0:
        raise RuntimeError(f"device status {word} during the study")
    # one more pass with events around every drift call: the drift reduction's
    # own bandwidth on these pipelines (6 algorithmic bytes per element)
    # (one stream, nothing overlapping it); its A-hat values must equal the
    # overlapped passes' bit for bit
    dev_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in batches]
    overlapped_res = res.clone()
    study_pass(cg, torch, configs, batches, bufs, res, drift_events=dev_ev, overlap=False)
    torch.cuda.synchronize()
    if not torch.equal(res.view(torch.int64), overlapped_res.view(torch.int64)):
        raise RuntimeError("the overlapped passes' A-hat values differ from the one-stream pass")
    drift_ms = sum(a.elapsed_time(b) for a, b in dev_ev)
    drift_bytes = float(sum(SI.n_elements(c) for c in configs)) * BYTES_PER_ELEMENT
    peak, peak_kind = measured_peaks()
    A = res.cpu().numpy().T
    total_cfg = ranks.sum(float(len(configs)))
    elems = ranks.sum(float(sum(SI.n_elements(c) for c in configs)))

    cpu = None
    if ranks.rank == 0 and ranks.world == 1 and not args.no_cpu_baseline:
        cpu = study_oracle_baseline(configs, args.cpu_seconds)
    if ranks.rank != 0:
        return
    names = ["rel_l2", "max_abs", "cos_dev", "control", "pooled_rel_l2"]
    summary = {n: {"min": float(np.nanmin(A[:, k])), "mean": float(np.nanmean(A[:, k])),
                   "max": float(np.nanmax(A[:, k])), "n_equal_1": int((A[:, k] == 1.0).sum())}
               for k, n in enumerate(names)}
    line = {
        "metric": STUDY_METRIC, "value": total_cfg / (ms / 1e3), "unit": "configs/s",
        "n_gpus": ranks.world, "steps": reps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic",
        "config": {"workload": f"study '{args.study}': {len(configs)} configurations",
                   "elements_per_pass": elems,
                   "batches": len(batches),
                   "step": "per batch of equal-shape configurations (at most 2^29 elements): "
                           "generate each (2 to 4 kernels), one batched drift (2), control labels "
                           "(one call per run of consecutive config ids), 3 + 1 per-canary AUROC "
                           "and 1 pooled AUROC over the batch; batch b + 1 is generated on a "
                           "second stream while b is scored (two pipeline buffers)"},
        "elements_per_s": elems / (ms / 1e3),
        "execution": "CUDA graph of one whole pass, replayed" if graph is not None else "eager",
        "eager": {"value": total_cfg / (ms_eager / 1e3), "unit": "configs/s",
                  "ms_per_step": ms_eager, "graph_error": graph_error},
        "drift": {"ms_per_pass": drift_ms, "GBps": drift_bytes / (drift_ms / 1e3) / 1e9,
                  "frac": drift_bytes / (drift_ms / 1e3) / 1e9 / peak,
                  "peak_GBps": peak, "peak_kind": f"{peak_kind} copy bandwidth",
                  "elements_per_s": drift_bytes / BYTES_PER_ELEMENT / (drift_ms / 1e3)},
        "auroc_summary": summary,
        "per_config_auroc": {n: [round(float(x), 6) for x in A[:, k]] for k, n in enumerate(names)},
        "cpu_baseline": cpu,
        "gpu_launches": study_launches(configs, batches,
                                       torch.cuda.get_device_properties(dev).multi_processor_count)
                        * reps,
        "clocks": clk,
    }
    print(json.dumps(line), flush=True)


def auroc_launches(N, S, C=1, sm_count=152) -> int:
    """Launches of one cg_auroc call on C configurations: one block per
    configuration ranks and combines it (S <= 32, N <= 1024), or a warp per
    configuration (S <= 32, C >= 8 per SM; S > 32, C >= 2 per SM); else
    canary-parallel counts and a per-configuration combine."""
    if S <= 32:
        return 1 if (N <= 1024 or C >= 8 * sm_count) else 2
    return 1 if C >= 2 * sm_count else 2


def generator_launches(cfg) -> int:
    """Generator kernels of one configuration: 2 when every stage's live values
    follow element by element, else 4; 2 + 3 per stage when propagating."""
    if cfg.get("gain", 0.0):
        return 2 + 3 * cfg["n_shards"]
    n_mal = len(cfg["malicious"])
    needs_stats = ((n_mal < cfg["n_shards"] and cfg["noise"] == SI.NOISE_PAPER) or
                   (n_mal > 0 and cfg["tamper"] == SI.TAMPER_ADDITIVE))
    return 4 if needs_stats else 2


def study_launches(configs, batches, sm_count=152) -> int:
    """Kernel launches of one study pass: per batch, every configuration's
    generator, the batched drift (2), one control-label call per run of
    consecutive ids, three per-canary AUROC calls and the control's, and
    the pooled AUROC (1)."""
    total = 0
    for idx in batches:
        c, B = configs[idx[0]], len(idx)
        total += sum(generator_launches(configs[i]) for i in idx)
        total += 2 + len(id_runs(configs, idx)) + 1
        total += 4 * auroc_launches(c["n_canaries"], c["n_shards"], B, sm_count)
    return total


def study_oracle_baseline(cfgs, seconds):
    """The fp64 oracle on a bounded sample of the study: its configurations in
    order, each with its canaries cut to at most 8, until `seconds` pass."""
    from oracle import oracle as O
    O.build()
    threads = O.max_threads()
    done, t0 = 0, time.perf_counter()
    for cfg in cfgs:
        sub = SI.shrink(cfg, n_canaries=min(8, cfg["n_canaries"]))
        gain = sub.pop("gain", 0.0)
        D = O.desc_from_dict(sub)
        acts, refs, labels = O.generate_pipeline(D, n_threads=threads)
        if gain:
            acts, refs = O.generate_propagating(D, gain, n_threads=threads)
        sc = O.drift_scores(acts, refs, sub["n_shards"], sub["n_canaries"], n_threads=threads)
        for k in range(3):
            O.auroc(sc[k].astype(np.float32)[None], labels[None])
        O.auroc_pooled(sc[0].astype(np.float32)[None], labels[None])
        done += 1
        if time.perf_counter() - t0 >= seconds:
            break
    el = time.perf_counter() - t0
    first = cfgs[0] if cfgs else {"n_canaries": 1}
    frac = min(8, first["n_canaries"]) / first["n_canaries"]
    return {"value": done * frac / el, "unit": "cfgs/s", "cores": threads, "kind": "oracle",
            "sample": f"first {done} configurations with at most 8 canaries each (generate + "
                      f"drift + AUROC in fp64), scaled to full canary counts by {frac:.3f}, "
                      f"{el:.1f} s"}


def main(argv=None):
    args = parse_args(argv)
    ranks = Ranks()
    if args.impl == "reference":
        if ranks.world > 1 and ranks.rank != 0:
            return 0
        run_reference(args, ranks)
        return 0
    ranks.init("nccl")
    try:
        if args.study:
            run_study(args, ranks)
            return 0
        run_ours(args, ranks)
    finally:
        ranks.close()
    return 0


if __name__ == "__main__":
    sys.exit(main())
