import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: long-running CPU test")


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """bf16 token agreement per parity test (tests/parity.py AGREEMENT): raw
    agreement over all slots, and over the decidable slots (noise farther
    than the logit-error bound from every CDF boundary)."""
    try:
        from parity import AGREEMENT
    except ImportError:
        return
    if not AGREEMENT:
        return
    tr = terminalreporter
    tr.write_sep("-", "bf16 token agreement vs the oracle")
    for name, (n, m, bad, dec, dm) in sorted(AGREEMENT.items()):
        raw = 100.0 * (n - m) / max(1, n)
        drate = 100.0 * (dec - dm) / max(1, dec)
        tr.write_line(f"{name}: {n - m}/{n} slots agree ({raw:.2f}%), {m - bad} of {m} "
                      f"mismatches explained; decidable {dec - dm}/{dec} ({drate:.2f}%)")
