import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built libsdq.so")


def gpu_available():
    try:
        import torch
        return torch.cuda.is_available()
    except Exception:
        return False


@pytest.fixture(scope="session")
def golden():
    import json
    with open(os.path.join(ROOT, "tests", "golden", "worked_rows.json")) as f:
        return json.load(f)


def _lib_stale(lib_path, csrc):
    if not os.path.exists(lib_path):
        return True
    t = os.path.getmtime(lib_path)
    for f in os.listdir(csrc):
        if os.path.getmtime(os.path.join(csrc, f)) > t:
            return True
    return False


@pytest.fixture(scope="session")
def sdq():
    """The binding with libsdq.so built (built here if missing or stale)."""
    import paper_2510_03275_gb300 as P
    from paper_2510_03275_gb300 import build as B
    if _lib_stale(B.LIB, B.CSRC):
        B.build()
    P.lib()
    return P
