import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")


@pytest.fixture(scope="session")
def oracle_mod():
    import oracle
    oracle.build()
    return oracle


@pytest.fixture(scope="session")
def mmbev_lib():
    """The CUDA library, built in-tree; GPU tests fail loudly if it is absent."""
    import paper_2608_15437_gb300 as mmbev
    mmbev.build()
    mmbev.load()
    return mmbev


@pytest.fixture(scope="session")
def cuda_dev(mmbev_lib):
    import torch
    if not torch.cuda.is_available():
        pytest.fail("GPU test collected without a CUDA device")
    return torch.device("cuda:0")
