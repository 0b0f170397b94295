import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)
TESTS = os.path.dirname(os.path.abspath(__file__))
if TESTS not in sys.path:
    sys.path.insert(0, TESTS)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built libretrace")
    config.addinivalue_line("markers", "slow: full-size workloads (GPU tests only)")


def pytest_collection_modifyitems(config, items):
    # GPU tests cannot run without a device: skip them loudly instead of failing
    # when someone runs the whole suite on a CPU-only machine.
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


def pytest_terminal_summary(terminalreporter):
    # bf16 comparisons: how many elements needed the 1-ulp allowance above the
    # 2e-2 bound (|reference| >= 4), next to the largest error of each check
    parity = sys.modules.get("parity")
    rows = getattr(parity, "RELAXED", None)
    if not rows:
        return
    terminalreporter.section("bf16 elements above 2e-2 (allowed: 1 bf16 ulp where |ref| >= 4)")
    for what, count, total, worst in rows:
        terminalreporter.write_line(f"{what or '(unnamed)'}: {count} of {total} elements above 2e-2; "
                                    f"largest error {worst:.4g}")
