import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (run on the GB300 box)")
    config.addinivalue_line("markers", "slow: long-running CPU test")


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """Print the parity reports the tests recorded: tokens compared with the
    oracle, tokens excused by the routing gap rule, and the output errors."""
    try:
        from pmpe_testlib import PARITY_REPORT
    except Exception:
        return
    if not PARITY_REPORT:
        return
    terminalreporter.write_line("parity against the oracle (tokens excused by the gap rule z_(k) - z_(k+1) < 1e-4):")
    for r in PARITY_REPORT:
        terminalreporter.write_line(
            f"  {r['name']}: {r['tokens']} tokens, {r['excused']} excused "
            f"({r.get('excused_selection_differs', 0)} with another valid selection), "
            f"max_abs_rel {r['max_abs_rel']:.3g}, mean_rel {r['mean_rel']:.3g}, "
            f"excused max_abs_rel {r.get('excused_max_abs_rel', 0.0):.3g}")
