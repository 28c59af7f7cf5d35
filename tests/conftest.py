import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line(
        "markers", "gpu: needs a CUDA GPU (sm_103a); parity tests of the CUDA path")


@pytest.fixture(scope="session")
def cuda_device():
    """The GPU for parity tests. Fails (does not skip) when the native library
    is missing on a machine that has a GPU."""
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2010_07565_gb300 import binding
    binding.lib()  # raises if libbigcn.so has not been built
    return torch.device("cuda", 0)
