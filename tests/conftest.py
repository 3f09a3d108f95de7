import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a GB300 (sm_103a) and the built librfq.so")


def read_golden(name):
    """Parse a tests/golden fixture: '# ...' comment lines, then 'key: values'."""
    out = {}
    with open(os.path.join(ROOT, "tests", "golden", name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, val = line.split(":", 1)
            out[key.strip()] = val.split()
    return out


@pytest.fixture(scope="session")
def orc():
    import oracle
    oracle.build()
    return oracle


@pytest.fixture(autouse=True)
def _canary_guards(request, monkeypatch):
    """GPU tests: every quantized matrix the test allocates through
    rfq.empty_qtensor carries canary bytes past its codes and its scales,
    checked once the test has run (tests/gpu_util.py)."""
    if request.node.get_closest_marker("gpu") is None:
        yield
        return
    import gpu_util
    from paper_2608_26581_gb300 import rfq
    monkeypatch.setattr(rfq, "empty_qtensor", gpu_util.guarded_qtensor)
    gpu_util._guarded.clear()
    yield
    gpu_util.check_guards()
