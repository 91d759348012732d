import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: long-running CPU test")


@pytest.fixture(scope="session")
def oscars_lib():
    """The built C-ABI library (built here if it is missing or stale)."""
    from paper_2102_08550_gb300 import _build
    _build.build()
    import paper_2102_08550_gb300 as P
    return P.lib()


@pytest.fixture(scope="session")
def cuda_device():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2102_08550_gb300 import _build
    _build.build()
    return torch.device("cuda:0")
