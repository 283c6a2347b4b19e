import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: large-size parity case")


def _cuda_available():
    try:
        import torch
        return torch.cuda.is_available()
    except Exception:
        return False


def pytest_collection_modifyitems(config, items):
    if _cuda_available():
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for item in items:
        if "gpu" in item.keywords:
            item.add_marker(skip)


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """The figures of every attention parity check of the run (max-abs, element-wise and
    per-row relative error against the fp64 oracle)."""
    try:
        from tests.parity import RECORDS
    except Exception:
        return
    if not RECORDS:
        return
    tr = terminalreporter
    tr.section("attention parity figures (bar 1e-2 each)")
    worst = {k: max(r[k] for _, r in RECORDS) for k in ("max_abs", "elem_rel", "max_rel")}
    tr.write_line(f"{len(RECORDS)} checks; worst max-abs {worst['max_abs']:.3e}, element-wise rel "
                  f"{worst['elem_rel']:.3e}, per-row rel {worst['max_rel']:.3e}")
    for what, r in sorted(RECORDS, key=lambda x: -x[1]["elem_rel"])[:40]:
        tr.write_line(f"  {r['max_abs']:.3e}  {r['elem_rel']:.3e}  {r['max_rel']:.3e}  {what}")
