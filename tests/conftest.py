import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built libpps.so")
    config.addinivalue_line("markers", "slow: long-running statistical check")


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
