import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)
TESTS = os.path.dirname(os.path.abspath(__file__))
if TESTS not in sys.path:
    sys.path.insert(0, TESTS)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (runs on the GB300 box)")
    config.addinivalue_line("markers", "slow: long-running full-size case")


@pytest.fixture(scope="session")
def cuda_available():
    import torch
    return torch.cuda.is_available()


@pytest.fixture(scope="session")
def vie(cuda_available):
    """The CUDA binding, loaded where a CUDA device is present; GPU tests fail loudly without it."""
    if not cuda_available:
        pytest.skip("no CUDA device")
    import paper_2608_27460_gb300 as vie_mod
    vie_mod.load()
    return vie_mod
