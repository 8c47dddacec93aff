import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA device (sm_103a) and the built library")


def pytest_runtest_setup(item):
    import parity_util
    parity_util.CURRENT_TEST[0] = item.nodeid


def pytest_terminal_summary(terminalreporter):
    """Largest elementwise and normwise error of every parity check, per test."""
    import parity_util
    if parity_util.NOTES:
        terminalreporter.section("tables measured in this session")
        for line in parity_util.NOTES:
            terminalreporter.write_line(line)
    if not parity_util.REPORT:
        return
    terminalreporter.section("parity errors (max over outputs: elementwise / normwise, bound)")
    worst = {}
    for test, tol, errs in parity_util.REPORT:
        if not errs:
            continue
        e = max(v[0] for v in errs.values())
        n = max(v[1] for v in errs.values())
        pe, pn, _ = worst.get(test, (0.0, 0.0, tol))
        worst[test] = (max(pe, e), max(pn, n), tol)
    for test, (e, n, tol) in worst.items():
        terminalreporter.write_line(f"{e:.2e} / {n:.2e}  <= {tol:.0e}  {test}")


@pytest.fixture(scope="session")
def lib():
    """The built C-ABI library (ctypes handle); builds it if missing."""
    from paper_1905_00689_gb300 import _binding
    return _binding.load()


@pytest.fixture(scope="session")
def cuda_device():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return torch.device("cuda:0")
