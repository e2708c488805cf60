"""pytest configuration: the `gpu` marker and shared fixtures."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")


@pytest.fixture(scope="session")
def cuda():
    """The CUDA device; skips only when the machine has no GPU at all."""
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device on this machine")
    return torch.device("cuda:0")


@pytest.fixture(scope="session")
def lrc(cuda):
    """The GPU library binding.  On a GPU machine a missing or broken library
    is an error, never a skip."""
    import paper_2607_12969_gb300 as lrc_mod
    lrc_mod.load()
    return lrc_mod
