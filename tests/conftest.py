import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built libmone.so")
    config.addinivalue_line("markers", "slow: long-running CPU test")


def pytest_terminal_summary(terminalreporter):
    """Worst observed error under each (check, quantity, bound) of the parity tests run."""
    try:
        from harness import MARGINS
    except Exception:
        return
    if not MARGINS:
        return
    worst = {}
    for check, key, value, bound in MARGINS:
        k = (check, key, bound)
        worst[k] = max(worst.get(k, 0.0), value)
    terminalreporter.write_sep("-", "parity margins (worst observed error / bound)")
    for (check, key, bound), value in sorted(worst.items()):
        terminalreporter.write_line(f"{check:<28} {key:<10} {value:.3e} / {bound:.0e}  ({value / bound:.3f})")
