import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")


def pytest_collection_modifyitems(config, items):
    import torch
    if torch.cuda.is_available():
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for item in items:
        if "gpu" in item.keywords:
            item.add_marker(skip)


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """Measured parity margins: the largest relative distance error and the
    largest relative gap at the r-th neighbour among swapped keys, per
    workload, next to the tolerances (1e-3 / 1e-5 and 1e-4)."""
    try:
        import parity
    except ImportError:
        return
    if not parity.STATS:
        return
    terminalreporter.write_sep("-", "measured parity margins (GPU vs oracle)")
    for label, st in sorted(parity.STATS.items()):
        terminalreporter.write_line(
            f"{label}: rows {st['rows']}, max |dD|/D {st['max_dist_rel']:.3g}, "
            f"swaps {st['swaps']}, max swap gap / D_r {st['max_gap_rel']:.3g}")
