"""Shared pytest setup: repository root on sys.path and the `gpu` marker."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a); runs the CUDA path")


@pytest.fixture(scope="session")
def orc():
    """The fp64 CPU oracle (built on first use)."""
    from oracle import oracle as O
    O.build()
    return O
