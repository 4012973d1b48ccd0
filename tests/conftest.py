import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")


import pytest


@pytest.fixture(scope="session")
def dslib():
    """The built CUDA library and its binding (GPU tests only)."""
    import torch
    if not torch.cuda.is_available():
        pytest.fail("GPU test collected without a CUDA device")
    from paper_1905_13298_gb300 import build
    build.build_library()
    import paper_1905_13298_gb300 as ds
    ds.lib()
    return ds
