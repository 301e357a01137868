import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")


def pytest_collection_modifyitems(config, items):
    try:
        import torch
        has_gpu = torch.cuda.is_available()
    except Exception:  # pragma: no cover
        has_gpu = False
    if has_gpu:
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for item in items:
        if "gpu" in item.keywords:
            item.add_marker(skip)


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """Worst max / mean abs error of every bf16 output each parity test compared."""
    try:
        from tests import parity
    except Exception:  # pragma: no cover
        return
    if not parity.WORST:
        return
    terminalreporter.section("worst parity errors (bf16 outputs vs the fp64 oracle)")
    for (test, what), (mx, mean) in sorted(parity.WORST.items()):
        terminalreporter.write_line(f"{test}  {what}: max {mx:.3e}  mean {mean:.3e}")
