import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line(
        "markers", "gpu: needs a GB300 (sm_103a) and the built CUDA library")


@pytest.fixture(scope="session")
def built_library():
    """Path of libsolo_readout.so, compiling it first when it is missing."""
    from paper_2609_35440_gb300 import build
    return build.ensure_built()
