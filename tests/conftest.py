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
def oracle_mod():
    from oracle import oracle
    oracle._lib()
    return oracle


def pytest_collection_modifyitems(config, items):
    """GPU tests need CUDA and the built library; on a machine without a GPU
    they are skipped (select them with -m gpu on a GB300)."""
    try:
        import torch
        has_cuda = torch.cuda.is_available()
    except Exception:  # pragma: no cover
        has_cuda = False
    if has_cuda:
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for item in items:
        if "gpu" in item.keywords:
            item.add_marker(skip)


@pytest.fixture(scope="session")
def libcsr():
    """Build (if stale) and load the C-ABI library."""
    from paper_2605_07325_gb300 import build
    build.build()
    from paper_2605_07325_gb300 import csr
    return csr
