import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: long-running CPU test")


@pytest.fixture(scope="session")
def rng():
    return np.random.Generator(np.random.PCG64(12345))


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """Lists every block a GPU parity test excused at a documented near-tie."""
    try:
        from _parity import EXCUSED
    except ImportError:
        return
    terminalreporter.write_line(f"parity: {len(EXCUSED)} block(s) excused at a near-tie")
    for line in EXCUSED:
        terminalreporter.write_line("  " + line)
