"""Shared test configuration: the ``gpu`` marker and the golden-fixture reader."""
import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

GOLDEN = os.path.join(ROOT, "tests", "golden")


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (runs the CUDA path through the C ABI)")


def golden_kv(name):
    """Parse ``key = v1 v2 ...`` lines of a golden fixture (comments start with '#')."""
    out = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if "=" in line:
                k, v = line.split("=", 1)
                out[k.strip()] = v.split()
    return out


def golden_lines(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return [l.rstrip("\n") for l in f if l.strip() and not l.lstrip().startswith("#")]


@pytest.fixture(scope="session")
def lib():
    """The packed-convolution C library (built on demand; loads without a GPU)."""
    from paper_2003_06513_gb300 import _lib
    return _lib.load(build_if_missing=True)


def cuda_ok():
    try:
        import torch
        return torch.cuda.is_available()
    except Exception:
        return False
