import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built libomq")
    config.addinivalue_line("markers", "full: runs the full workload sizes (minutes of oracle time on the host)")


@pytest.fixture(scope="session")
def cuda_lib():
    """The C-ABI library on cuda:0; fails loudly when the GPU or the build is missing."""
    import torch
    if not torch.cuda.is_available():
        pytest.fail("gpu test selected but no CUDA device is visible")
    from paper_2308_13137_gb300 import _lib
    return _lib.lib()
