import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (runs the CUDA path through the C ABI)")
    # the library is compiled in-tree; make sure the tests load a current build
    from paper_2609_24150_gb300 import build as _build
    _build.build_if_stale()


@pytest.fixture(scope="session")
def root_dir():
    return ROOT
