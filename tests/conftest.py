import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")


def pytest_terminal_summary(terminalreporter):
    """Error figures of the parity tests: per element normalised by max(rms, |ref|)
    of its output (the bar), the whole-tensor max|diff| / rms(ref) (the literal
    reading), and the aggregate rms(diff) / rms(ref)."""
    try:
        import gpu_helpers
    except Exception:
        return
    rows = gpu_helpers.REPORT
    if not rows:
        return
    tr = terminalreporter
    tr.write_sep("-", "parity error figures (per-element bar | literal max/rms | aggregate)")
    for case, name, rel, lit, rms in rows:
        tr.write_line("%-22s %-14s %.5f | %.5f | %.6f" % (case, name, rel, lit, rms))
