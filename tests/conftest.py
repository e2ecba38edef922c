import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the compiled library")


@pytest.fixture(scope="session")
def oracle():
    import oracle as o
    o.build()
    return o


@pytest.fixture(scope="session")
def gpu():
    """cuda:0 with libmpq.so built and loaded (the CUDA path; no fallback)."""
    import torch
    from paper_2002_09049_gb300 import _build, binding
    assert torch.cuda.is_available(), "gpu tests need a CUDA device"
    _build.build()
    binding.load()
    return torch.device("cuda:0")
