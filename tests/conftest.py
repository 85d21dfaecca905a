import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA device and the built libcospec.so")
    config.addinivalue_line("markers", "slow: full-size workload (minutes)")


GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


@pytest.fixture(scope="session")
def golden_dir():
    return GOLDEN


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """Near-tie counts of the parity tests (sequences whose discrete outputs
    hinge on a top-1/top-2 margin or a policy probability within 1e-3)."""
    from tests.parity_util import TIE_REPORT
    if not TIE_REPORT:
        return
    terminalreporter.write_sep("-", "near ties excluded from bit-exact checks")
    for r in TIE_REPORT:
        terminalreporter.write_line(
            f"{r['workload']}: {r['tie_affected_sequences']}/{r['sequences']} sequences, "
            f"{r['tie_positions']} positions ({r['test']})")
    path = os.environ.get("COSPEC_PARITY_REPORT")
    if path:
        import json
        with open(path, "w") as fh:
            json.dump(TIE_REPORT, fh, indent=1)
