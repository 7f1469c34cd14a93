"""The boundary from plain C: tests/c_abi_client.c is compiled with gcc
against include/canary_guard.h and the built library (no Python, no torch
in the client) and run; it generates, scores and ranks the tiny pipeline,
then scores a batch of two configurations and the no-workspace variant and
compares them with the single call."""
import os
import shutil
import subprocess

import pytest

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_c_client_runs(tmp_path):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_19490_gb300.build import build
    lib = build()
    cuda = os.path.dirname(os.path.dirname(shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"))
    exe = str(tmp_path / "c_abi_client")
    subprocess.run(["gcc", "-O2", "-std=c11", os.path.join(ROOT, "tests", "c_abi_client.c"),
                    "-I", os.path.join(ROOT, "include"), "-I", os.path.join(cuda, "include"),
                    lib, "-L", os.path.join(cuda, "lib64"), "-lcudart", "-lm",
                    f"-Wl,-rpath,{os.path.dirname(lib)}", f"-Wl,-rpath,{os.path.join(cuda, 'lib64')}",
                    "-o", exe], check=True)
    out = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert out.returncode == 0, out.stderr
    fields = out.stdout.split()
    assert fields[0] == "A_hat" and float(fields[1]) == 1.0          # Table 1, full detector
    assert 0.0 <= float(fields[3]) <= 1.0 and fields[5] == "0"
    assert fields[6:10] == ["batch_equal", "1", "noalloc_close", "1"]
