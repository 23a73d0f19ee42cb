import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA device (a GB300) and the built CUDA library")
    config.addinivalue_line("markers", "slow: long-running case")


@pytest.fixture(scope="session")
def ea_lib():
    """The in-tree CUDA library (built here with nvcc if needed); loading needs no GPU."""
    from paper_2205_14473_gb300 import build as B
    import paper_2205_14473_gb300 as ea

    B.build()
    return ea.lib()
