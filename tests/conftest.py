import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (runs through libkvxfer.so)")


def pytest_sessionstart(session):
    """Build the CUDA library and the C oracle in tree if they are missing or stale
    (no-ops otherwise), so the binding's import never meets a stale build."""
    from paper_2609_15021_gb300 import _build
    _build.build()
    import oracle
    oracle.build()


@pytest.fixture(scope="session")
def orc():
    import oracle
    return oracle.c_oracle()
