import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")


@pytest.fixture(scope="session")
def orc():
    import oracle
    return oracle.default()


@pytest.fixture(scope="session")
def cuda_lib_path():
    """Build (nvcc cross-compiles without a GPU) and return the library path."""
    from paper_2606_02955_gb300 import build as fbuild
    return fbuild.build_library()


@pytest.fixture(scope="session")
def fd():
    """The Python binding over the CUDA library (GPU tests only)."""
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_02955_gb300 import build as fbuild
    fbuild.build_library()
    import paper_2606_02955_gb300 as fd
    return fd
