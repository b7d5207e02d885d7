import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

GOLDEN = os.path.join(ROOT, "tests", "golden")


def pytest_configure(config):
    config.addinivalue_line(
        "markers", "gpu: needs a CUDA GPU and the compiled sm_103a library")
    config.addinivalue_line(
        "markers", "slow: full-size case, minutes rather than seconds")


@pytest.fixture(scope="session")
def oracle():
    import oracle as O
    O.lib()
    return O


@pytest.fixture(scope="session")
def golden():
    import json
    with open(os.path.join(GOLDEN, "worked_example.json")) as f:
        return json.load(f)


@pytest.fixture(scope="session")
def stream_golden():
    import json
    with open(os.path.join(GOLDEN, "stream_example.json")) as f:
        return json.load(f)
