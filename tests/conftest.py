import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built libpps.so")
    config.addinivalue_line("markers", "slow: long-running statistical check")
    # PPS_PHILOX_ROUNDS=7: the binding loads libpps_r7.so (the Philox4x32-7 keyed source), and the
    # oracle's keyed source takes the same round count
    rounds = os.environ.get("PPS_PHILOX_ROUNDS")
    if rounds:
        import oracle
        oracle.set_philox_rounds(int(rounds))


def pytest_terminal_summary(terminalreporter):
    """Print the full-size parity report (flip counts, accept lengths vs the oracle and the closed
    form) that tests/parity.py collects, so that a -q run still shows it."""
    mod = sys.modules.get("parity")
    rows = getattr(mod, "REPORT", None) if mod is not None else None
    if not rows:
        return
    terminalreporter.section("full-size parity report")
    for r in rows:
        terminalreporter.write_line("  ".join(f"{k}={v}" for k, v in r.items()))
