import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)
HERE = os.path.dirname(os.path.abspath(__file__))
if HERE not in sys.path:
    sys.path.insert(0, HERE)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built CUDA library")


@pytest.fixture(scope="session")
def oracle_mod():
    import oracle
    oracle.build()
    return oracle


@pytest.fixture(autouse=True)
def _name_parity_records(request):
    import parity
    parity._CURRENT_TEST[0] = request.node.nodeid
    yield


def pytest_terminal_summary(terminalreporter):
    """Per test, the largest per-tensor error (the bound that is asserted) and
    the largest elementwise relative error of the oracle comparisons."""
    import parity
    if not parity.RECORD:
        return
    worst = {}
    for test, name, e, ew in parity.RECORD:
        w = worst.setdefault(test, [0.0, "", 0.0, ""])
        if e >= w[0]:
            w[0], w[1] = e, name
        if ew >= w[2]:
            w[2], w[3] = ew, name
    terminalreporter.section("oracle comparisons: largest errors per test")
    for test, (e, n, ew, nw) in worst.items():
        terminalreporter.write_line(f"{test}: per-tensor {e:.2e} ({n}); elementwise {ew:.2e} ({nw})")
