import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a); runs the CUDA path")
    config.addinivalue_line("markers", "slow: full-size workloads (GPU box only)")


@pytest.fixture(scope="session", autouse=True)
def _host_libs():
    """The generator and the oracle are plain C; build them if they are missing (seconds)."""
    from oracle import build as ob
    from synth import build as sb
    sb.build()
    ob.build()
    yield
