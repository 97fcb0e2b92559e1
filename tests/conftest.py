import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a GB300 (sm_103a) and the built CUDA library")


@pytest.fixture(scope="session", autouse=True)
def _cpu_libraries():
    """The generator and the oracle are plain C; compile them once per session if needed."""
    import oracle
    import synth
    synth.build()
    oracle.build()
