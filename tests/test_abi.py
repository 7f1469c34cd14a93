"""Host-only checks of the C ABI (no GPU needed, no kernel launched).

The library builds, loads and exports every function include/canary_guard.h
declares; the size queries and the host-side argument validation answer
without touching a device (a rejected call launches nothing)."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "canary_guard.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2607_19490_gb300.build import build
    build()
    import paper_2607_19490_gb300 as cg
    return cg


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(cg_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("cg_generate_pipeline", "cg_drift_scores", "cg_auroc"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", lib.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT\s+(\w+)$", out, flags=re.M))
    missing = [n for n in declared_functions() if n not in exported]
    assert not missing, missing
    L = lib.load()
    for n in declared_functions():
        assert getattr(L, n) is not None


def test_status_strings_and_version(lib):
    for code, name in lib.STATUS_NAMES.items():
        assert lib.cg_status_string(code).startswith(name)
    assert lib.cg_abi_version() == 1


def test_drift_workspace_size(lib):
    n = lib.cg_drift_workspace_size(16, 256, 128 * 8192)
    chunks = (128 * 8192 + 16383) // 16384
    assert n >= 256 + 16 * 16 * 256 * chunks and n % 256 == 0
    with pytest.raises(lib.CgError):
        lib.cg_drift_workspace_size(0, 1, 1)


def test_generate_workspace_and_validation(lib):
    import seeded_inputs as SI
    d = lib.PipelineDesc.from_config(SI.SEVENTY_B)
    assert lib.cg_generate_workspace_size(d) > 0
    for bad in (dict(malicious=(16,)), dict(malicious=(1, 1)), dict(config_id=2**30),
                dict(tamper=7), dict(noise=3), dict(n_outlier=300),
                dict(tamper=1, tamper_param=1.5), dict(benign_sigma=-1.0),
                dict(n_shards=2000)):
        cfg = SI.shrink(SI.TINY, **bad)
        with pytest.raises(lib.CgError) as e:
            lib.cg_generate_workspace_size(lib.PipelineDesc.from_config(cfg))
        assert e.value.status in (1, 7)


def test_rejected_calls_launch_nothing(lib):
    L = lib.load()
    P = ctypes.c_void_p
    fake = P(0x10000)           # never dereferenced: validation fails first
    odd = P(0x10002)
    # NULL inputs
    assert L.cg_drift_scores(None, fake, 4, 4, 64, fake, 16, fake, 1 << 20, None, None) == 1
    # misaligned live activations
    assert L.cg_drift_scores(odd, fake, 4, 4, 64, fake, 16, fake, 1 << 20, None, None) == 2
    # workspace too small
    assert L.cg_drift_scores(fake, fake, 4, 4, 64, fake, 16, fake, 8, None, None) == 3
    # stat_stride below N*S
    assert L.cg_drift_scores(fake, fake, 4, 4, 64, fake, 15, fake, 1 << 20, None, None) == 1
    # ranking: S too large, missing outputs
    assert L.cg_auroc(fake, fake, 1, 1, 5000, fake, None, None, fake, None, None) == 7
    assert L.cg_auroc(fake, fake, 1, 1, 4, None, None, None, fake, None, None) == 1
    assert L.cg_make_control_labels(fake, 1, 1, 4, 0, 2**30, fake, None, None) == 1
    assert L.cg_philox_words(0, 0, 0, 0, 0, 0, fake, None) == 1
    assert L.cg_philox_words(0, 0, 0, 0, 0, 4, odd, None) == 2
    assert L.cg_read_status(None, None, None) == 1
