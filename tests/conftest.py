import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built CUDA library")
    config.addinivalue_line("markers", "slow: long-running (full-size shards)")


@pytest.fixture(scope="session", autouse=True)
def _build_host_libs():
    """Compile the host-side C helpers (input generator, oracle) once."""
    import oracle
    import synth
    synth.build()
    oracle.build()
    # the oracle parallelises over independent output rows only: results do
    # not depend on the thread count
    oracle.set_threads(os.cpu_count() or 1)
    yield
