"""Host threads calling the library at once (GPU).

The library keeps two pieces of host state, the per-device attribute and
occupancy caches, each behind a mutex; every other argument travels with the
call, and ctypes releases the interpreter lock while a call runs.  A fresh
process (so the caches start empty and the first calls race) runs four
threads, each generating, scoring, drawing control labels and ranking five
configurations on its own stream, then repeats the same work on one thread;
tests/_threads_child.py asserts the two agree bit for bit."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def built():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_19490_gb300 as m
    m.build()
    return m


def test_concurrent_host_threads_match_sequential(built):
    child = os.path.join(ROOT, "tests", "_threads_child.py")
    r = subprocess.run([sys.executable, child], capture_output=True, text=True, timeout=600,
                       cwd=ROOT)
    assert r.returncode == 0 and "threads ok" in r.stdout, (r.stdout[-2000:], r.stderr[-2000:])
