import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300) and the built library")

import pytest  # noqa: E402


@pytest.fixture(scope="session")
def zlib():
    """The C-ABI library, built in-tree first if it is missing."""
    from paper_2509_01190_gb300 import build, zsaa
    if not os.path.exists(zsaa.LIB_PATH):
        build.build()
    return zsaa
