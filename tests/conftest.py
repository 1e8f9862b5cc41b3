import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: a full-size workload (minutes)")


@pytest.fixture(scope="session")
def oracle():
    from oracle import oracle as O
    O.build()
    return O


def pytest_terminal_summary(terminalreporter):
    """Mask parity counts of every layer a GPU test checked (near-tie rows are
    the fp64 rows within the fp32 error bound; the GPU must differ from the
    oracle's fp32 decision on none)."""
    mod = sys.modules.get("parity_util")
    stats = getattr(mod, "MASK_STATS", None) if mod else None
    if not stats:
        return
    tr = terminalreporter
    tr.write_sep("-", "block-mask parity (rows: query blocks x heads x batch)")
    tr.write_line(f"{'layer':48s} {'rows':>8s} {'near-tie':>9s} {'%':>6s} {'f32!=f64':>9s} {'GPU!=f32':>9s}")
    for label, rows, near, f64d, gpud in stats:
        tr.write_line(f"{label[:48]:48s} {rows:8d} {near:9d} {100.0 * near / rows:6.2f} {f64d:9d} {gpud:9d}")
