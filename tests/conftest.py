import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: full-size workloads (minutes of host work)")


@pytest.fixture(scope="session")
def lib():
    """The built C-ABI library (builds it in-tree when missing)."""
    from paper_2605_31457_gb300 import build as _build
    _build.ensure_built()
    from paper_2605_31457_gb300 import vp
    return vp
