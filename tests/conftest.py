import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300) and the built library")


def pytest_collection_modifyitems(config, items):
    # fail loudly rather than skip: a GPU test that cannot find a GPU is an error,
    # but only when GPU tests were asked for (-m gpu)
    pass


@pytest.fixture(scope="session")
def gpu_lib():
    """The C-ABI library, built for this machine; GPU tests only."""
    import torch
    if not torch.cuda.is_available():
        pytest.fail("GPU test selected but no CUDA device is visible")
    from paper_2206_00470_gb300 import adapm
    adapm.load()
    return adapm
