import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: large CPU-side case")


@pytest.fixture(scope="session")
def polyq_lib():
    """The C-ABI library, built in-tree on first use."""
    from paper_2607_14618_gb300 import build as _build
    _build.build_library()
    from paper_2607_14618_gb300 import polyq
    return polyq
