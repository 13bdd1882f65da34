import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: large oracle comparisons")


@pytest.fixture(scope="session")
def lib():
    """The CUDA library through its C ABI; fails loudly if it is not built."""
    from paper_2609_01068_gb300 import outlets
    return outlets.load()
