"""A second library pin of the oracle's Philox4x32-10: cuRAND's device API.

curand_init(seed, subsequence, offset) starts the generator at key
(seed lo, seed hi) and counter (offset / 4 as a 64-bit number over words 0
and 1, subsequence lo, subsequence hi), so its first words pin the oracle's
Philox for counter word 3 != 0, the word the independent benign recompute
uses, and for word 1 >= 2^24, the auxiliary streams' (purpose << 24) | sub
(cuRAND's host generator reaches neither).  The program runs on the GPU;
the comparison is with the oracle only (not with this repository's CUDA)."""
import os
import shutil
import subprocess

import numpy as np
import pytest

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_oracle_philox_matches_curand_device(orc, tmp_path):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    exe = str(tmp_path / "curand_words")
    subprocess.run([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O2", "-o", exe,
                    os.path.join(ROOT, "tests", "curand_device_words.cu")], check=True)
    out = subprocess.run([exe], capture_output=True, text=True, timeout=120, check=True).stdout
    n_c3 = n_c1 = 0
    for line in out.strip().splitlines():
        f = [int(x) for x in line.split()]
        seed, sub, off, words = f[0], f[1], f[2], f[3:]
        c2, c3 = sub & 0xFFFFFFFF, sub >> 32
        block = off // 4                      # 64-bit block index over counter words 0 and 1
        first, c1 = block & 0xFFFFFFFF, block >> 32
        got = orc.philox_words(seed, c1, c2, c3, first, 2)
        assert list(got) == words, (seed, sub, off)
        n_c3 += c3 != 0
        n_c1 += c1 >= (1 << 24)
    assert n_c3 >= 3 and n_c1 >= 3
