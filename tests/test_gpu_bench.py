"""bench.py on the GPU: a short run on the tiny workload prints one JSON line
with every key of the contract (roofline, cpu_baseline, e2e, clocks,
gpu_launches), and a short study run prints its line."""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def bench_line(*args):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], cwd=ROOT,
                         capture_output=True, text=True, timeout=600)
    assert out.returncode == 0, out.stderr[-3000:]
    lines = [l for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, out.stdout[-2000:]
    return json.loads(lines[0])


def test_bench_line_contract():
    d = bench_line("--workload", "tiny", "--steps", "5", "--warmup", "3", "--cpu-seconds", "1")
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
              "roofline", "cpu_baseline", "e2e", "gpu_launches", "clocks"):
        assert k in d, k
    assert d["value"] > 0 and d["steps"] == 5 and d["warmup"] == 3 and d["n_gpus"] == 1
    r = d["roofline"]
    for k in ("bound", "achieved", "peak", "unit", "frac", "traffic"):
        assert k in r, k
    assert r["bound"] == "hbm" and abs(r["frac"] - r["achieved"] / r["peak"]) < 1e-9
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] > 0 and cb["sample"]
    e = d["e2e"]
    assert e["value"] > 0 and e["h2d_bytes_per_step"] > 0 and e["d2h_bytes_per_step"] > 0
    assert d["gpu_launches"] == 5 * 5          # drift 2, control 1, two one-launch AUROC calls
    assert {"sm_mhz", "sm_max_mhz", "reasons"} <= set(d["clocks"])


def test_bench_study_line():
    d = bench_line("--study", "collusion", "--steps", "2", "--warmup", "1", "--no-cpu-baseline")
    assert d["unit"] == "configs/s" and d["value"] > 0
    assert d["execution"].startswith("CUDA graph") and d["eager"]["graph_error"] is None
    assert d["auroc_summary"]["rel_l2"]["min"] == 1.0
