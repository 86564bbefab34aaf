import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300) and runs the CUDA kernels")


@pytest.fixture(scope="session")
def cuda_lib():
    """Builds (if needed) and loads libmemplan.so; GPU tests fail loudly without CUDA."""
    import torch

    assert torch.cuda.is_available(), "GPU test run without a CUDA device"
    from paper_2203_00448_gb300 import build
    from paper_2203_00448_gb300 import _lib

    build.build()
    return _lib.load()
