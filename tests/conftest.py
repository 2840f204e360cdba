import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built libeti")
    config.addinivalue_line("markers", "slow: long-running check")


@pytest.fixture(scope="session")
def oracle_lib():
    import oracle
    oracle.build()
    return oracle


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """One line with the parity counts of the session (near-ties accepted by
    the stated rules, worst errors), so that a run's log keeps them."""
    parity = sys.modules.get("parity")
    if parity is not None and any(parity.TALLY.values()):
        terminalreporter.write_line(parity.tally_line())
