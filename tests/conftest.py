import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300) and the built libpgc.so")
    config.addinivalue_line("markers", "slow: long-running")


_HEADROOM: list[str] = []


@pytest.fixture(scope="session")
def headroom():
    """Lines "case: worst observed error against its tolerance", printed after
    the run, so the margin of every floating-point parity check is on record."""
    return _HEADROOM


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    if _HEADROOM:
        terminalreporter.section("parity headroom: worst observed error / tolerance")
        for line in _HEADROOM:
            terminalreporter.write_line(line)


@pytest.fixture(scope="session")
def root_dir():
    return ROOT


@pytest.fixture(scope="session")
def libpgc():
    """The built library (built here if missing; nvcc cross-compiles without a GPU)."""
    from paper_2607_20739_gb300 import build as B
    B.build()
    from paper_2607_20739_gb300 import binding
    return binding


@pytest.fixture(scope="session")
def cuda(libpgc):
    import torch
    if not torch.cuda.is_available():
        pytest.fail("GPU test collected on a machine without CUDA")
    torch.cuda.init()
    return torch
