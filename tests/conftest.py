import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: full-size case (minutes)")


@pytest.fixture(scope="session")
def orc():
    import oracle
    oracle.build()
    return oracle


@pytest.fixture(scope="session")
def oracle_index():
    """Workload indexes built by the oracle (mixture vectors, Lloyd training,
    float32 encoding; oracle.pq_index), cached per workload for the session."""
    from oracle import pq_index
    cache = {}

    def get(w):
        if w not in cache:
            cache[w] = pq_index.OracleIndex(w)
        return cache[w]

    yield get
    for oi in cache.values():
        oi.close()


@pytest.fixture(scope="session")
def golden_dir():
    return os.path.join(ROOT, "tests", "golden")
