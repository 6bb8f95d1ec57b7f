"""Shared pytest set-up: the ``gpu`` marker, the repo-root import path and
the parity report printed at the end of the session."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """Near-tie counts and worst element-wise errors of every GPU-oracle
    comparison (relative to max(|ref_i|, row rms); val relative to |x|)."""
    from tests import parity
    lines = parity.summary_lines()
    if not lines:
        return
    terminalreporter.write_sep("=", "parity report: near-ties (counted, exempt) and worst errors")
    for line in lines:
        terminalreporter.write_line(line)
