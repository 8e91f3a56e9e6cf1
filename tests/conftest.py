import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (runs the CUDA library on cuda:0)")


def read_golden(name):
    """Sections of a tests/golden fixture: {title: list of rows of numbers}."""
    out, cur = {}, None
    with open(os.path.join(ROOT, "tests", "golden", name)) as f:
        for line in f:
            line = line.strip()
            if line.startswith("# section"):
                cur = line[len("# section"):].strip()
                out[cur] = []
            elif line and not line.startswith("#") and cur is not None:
                out[cur].append([float(t) for t in line.split()])
    return out


@pytest.fixture(scope="session")
def orc():
    import oracle
    oracle.build()
    return oracle
