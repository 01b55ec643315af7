import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

GOLDEN = os.path.join(ROOT, "tests", "golden")


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300) and the built CUDA library")
    config.addinivalue_line("markers", "slow: full-size workload; minutes of oracle time")


def parse_value(v):
    """Golden values are numbers or exact fractions / powers written as strings."""
    from fractions import Fraction
    if isinstance(v, str):
        if v.startswith("2^"):
            return 2.0 ** int(v[2:])
        return float(Fraction(v))
    return float(v)


@pytest.fixture(scope="session")
def golden():
    import json

    def load(name):
        with open(os.path.join(GOLDEN, name)) as f:
            return json.load(f)
    return load
