import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")


@pytest.fixture(scope="session")
def vlib():
    """The VarRate binding with its CUDA library built in-tree (built here if missing)."""
    from paper_2607_15498_gb300 import build, varrate
    if not os.path.exists(varrate.LIB_PATH):
        build.build()
    varrate.lib()
    return varrate
