"""The cheaper keyed source: libpps_r7.so (Philox4x32-7, built from the same sources with
PPS_PHILOX_ROUNDS=7) against the oracle at 7 rounds.  The parity, truncation, tree,
non-identical-proposal, LM-head, detector, acceptance and word-statistics suites run again in a
child process with PPS_PHILOX_ROUNDS=7, which makes the binding load libpps_r7.so and the
oracle's keyed source take 7 rounds (tests/conftest.py).  The full-size suite stays on the default build (the
bench line's `philox7` compares every row of the bench step at 7 rounds)."""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.gpu
def test_seven_round_build_reports_its_rounds():
    from paper_2609_21858_gb300 import pps
    import ctypes
    L = ctypes.CDLL(pps.library_path(7))
    L.pps_philox_rounds.restype = ctypes.c_int
    assert L.pps_philox_rounds() == 7
    assert pps.philox_rounds() == int(os.environ.get("PPS_PHILOX_ROUNDS", "10"))


@pytest.mark.gpu
def test_parity_suites_with_the_seven_round_keyed_source():
    if os.environ.get("PPS_PHILOX_ROUNDS"):
        pytest.skip("already the child run")
    env = dict(os.environ, PPS_PHILOX_ROUNDS="7")
    cmd = [sys.executable, "-m", "pytest", "-x", "-q", "-m", "gpu", "-p", "no:cacheprovider",
           "tests/test_gpu_parity.py", "tests/test_gpu_trunc.py", "tests/test_gpu_tree.py",
           "tests/test_gpu_hetero.py", "tests/test_gpu_lmhead.py", "tests/test_gpu_detect.py",
           "tests/test_gpu_accept.py", "tests/test_gpu_words_stats.py"]
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=1800)
    tail = (r.stdout[-4000:] + "\n" + r.stderr[-2000:])
    print(tail)
    assert r.returncode == 0, tail
    assert " passed" in r.stdout
