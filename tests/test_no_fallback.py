"""The product path has no CPU fallback and never reaches the oracle (host
only, no kernel launched).

- A missing CUDA library makes the first call fail with an error that says
  so, rather than computing anything on the host.
- Host (CPU) tensors are refused before any launch.
- Nothing in the package or the C ABI imports, links or names the oracle.
"""
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2607_19490_gb300")


def test_missing_library_fails_loudly(monkeypatch):
    import paper_2607_19490_gb300 as cg
    monkeypatch.setattr(cg, "LIB_PATH", os.path.join(ROOT, "no_such_dir", "libcanary_guard.so"))
    monkeypatch.setattr(cg, "_lib", None)
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        cg.load()
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        cg.cg_drift_workspace_size(4, 4, 64)


def test_host_tensors_are_refused():
    torch = pytest.importorskip("torch")
    import paper_2607_19490_gb300 as cg
    acts = torch.zeros((2, 3, 64), dtype=torch.float16)
    refs = torch.zeros((2, 3, 64), dtype=torch.float32)
    with pytest.raises(ValueError, match="CUDA tensor"):
        cg.cg_drift_scores(acts, refs, 2, 3)
    scores = torch.zeros((1, 3, 2), dtype=torch.float32)
    labels = torch.zeros((1, 3, 2), dtype=torch.int8)
    with pytest.raises(ValueError, match="CUDA tensor"):
        cg.cg_auroc(scores, labels)


def _sources():
    for d, _, files in os.walk(PKG):
        if "_build" in d or "__pycache__" in d:
            continue
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h", ".c", ".cpp")):
                yield os.path.join(d, f)
    for f in os.listdir(os.path.join(ROOT, "include")):
        yield os.path.join(ROOT, "include", f)


def test_package_never_reaches_the_oracle():
    pat = re.compile(r"^\s*(from\s+oracle\b|import\s+oracle\b|#\s*include\s*[<\"][^>\"]*oracle)|"
                     r"libcg_oracle|cg_oracle\.[ch]\b", re.M)
    hits = []
    for p in _sources():
        text = open(p, encoding="utf-8", errors="replace").read()
        for m in pat.finditer(text):
            hits.append(f"{os.path.relpath(p, ROOT)}: {m.group(0).strip()}")
    assert not hits, hits
