import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")


@pytest.fixture(scope="session")
def repo_root():
    return ROOT


@pytest.fixture(scope="session")
def jet():
    """The ctypes binding, building libjet.so first when it is missing or stale."""
    from paper_2609_33874_gb300 import build as _build
    _build.build()
    from paper_2609_33874_gb300 import jet as _jet
    return _jet
