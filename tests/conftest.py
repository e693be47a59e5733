"""Shared pytest set-up: the gpu marker, import paths and the library build."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a); runs the kernels")


@pytest.fixture(scope="session")
def lib():
    """The built C-ABI library (built in-tree on first use)."""
    from paper_2608_08684_gb300 import build as _build
    _build.build_library()
    from paper_2608_08684_gb300 import ripple
    return ripple
