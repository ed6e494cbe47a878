"""Test configuration: the ``gpu`` marker and import paths.

Tests marked ``gpu`` need a CUDA device and the compiled library; everything
else runs on a CPU-only machine.
"""

import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
TESTS = os.path.dirname(os.path.abspath(__file__))
for p in (ROOT, TESTS):
    if p not in sys.path:
        sys.path.insert(0, p)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU and the compiled MPM library")


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """Print the parity records of the full-size workload tests, if any ran."""
    parity = sys.modules.get("parity")
    lines = getattr(parity, "SUMMARY_LINES", None) if parity else None
    if lines:
        terminalreporter.section("MPM parity on the full workloads")
        for line in lines:
            terminalreporter.write_line(line)
