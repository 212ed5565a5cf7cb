import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built extension")
    config.addinivalue_line("markers", "slow: long-running CPU test")


def pytest_terminal_summary(terminalreporter):
    """Measured errors of every GPU parity check, so that the bars' margins are visible."""
    try:
        from helpers import PARITY_LOG
    except ImportError:
        return
    if not PARITY_LOG:
        return
    tr = terminalreporter
    tr.section("decode parity: measured errors against the fp64 oracle")
    tr.write_line(f"{'case':60s} {'bf16 max':>10s} {'bf16 mean':>10s} {'fp32 max':>10s}  widened bar")
    for where, mx, mean, m32, widened in PARITY_LOG:
        tr.write_line(f"{where[:60]:60s} {mx:10.3e} {mean:10.3e} {m32:10.3e}  {'yes' if widened else 'no'}")
    tr.write_line(f"bars: bf16 max-abs 5e-3, bf16 mean-abs 5e-4 (each widened only to the bf16 half-ulp), "
                  f"fp32 1e-4 * max(1, |y|); cases needing the widened bar: {sum(1 for r in PARITY_LOG if r[4])}")


@pytest.fixture(scope="session")
def oracle_lib():
    import oracle
    return oracle.lib()
