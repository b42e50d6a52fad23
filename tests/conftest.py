import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")


@pytest.fixture(scope="session")
def padlib():
    """libpad.so, built for sm_103a if it is missing or stale."""
    from paper_2607_02963_gb300 import build, binding
    build.build()
    return binding.lib()
