import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: longer oracle runs")


@pytest.fixture(scope="session")
def svl_lib():
    """The CUDA library, built in-tree on first use."""
    from paper_2607_20357_gb300.build import build_library
    from paper_2607_20357_gb300 import svl
    build_library()
    return svl.lib()
