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


_BAND_LOG = []


@pytest.fixture(autouse=True)
def _band_accounting(request):
    """Counts what the widened tie and threshold bands set aside in each test (tests/parity.py)."""
    try:
        from tests import parity
    except Exception:  # the library is not importable (e.g. collection on a box without it)
        yield
        return
    parity.band_reset()
    yield
    b = dict(parity.BAND)
    if b["tie_elems"] or b["rescued"] or b["thr_windows"]:
        _BAND_LOG.append((request.node.nodeid, b, parity.band_shares()))


def pytest_terminal_summary(terminalreporter):
    if not _BAND_LOG:
        return
    terminalreporter.write_sep("-", "widened bands: what they set aside")
    for nodeid, b, sh in _BAND_LOG:
        terminalreporter.write_line(
            f"{nodeid}: tie-band elements {b['tie_elems']}/{b['elems']} ({sh['tie']:.2e}), "
            f"rescued {b['rescued']} ({sh['rescued']:.2e}), threshold-band windows "
            f"{b['thr_windows']}/{b['windows']} ({sh['thr']:.2e})")
