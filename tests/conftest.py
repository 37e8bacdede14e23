import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built kvx library")
    config.addinivalue_line("markers", "slow: long-running case")


def pytest_collection_modifyitems(config, items):
    try:
        import torch
        has_gpu = torch.cuda.is_available()
    except Exception:
        has_gpu = False
    if has_gpu:
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for it in items:
        if "gpu" in it.keywords:
            it.add_marker(skip)


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """Summary of the session's parity comparisons: the worst rel-L2 and literal max-abs and the
    elements above 3e-2 (all within the element-wise bound 3e-2 + 2^-8 |ref| where they pass);
    the full list goes to the file KVX_PARITY_RECORD names, if set."""
    try:
        from harness import RECORD
    except Exception:
        return
    if not RECORD:
        return
    import json
    worst_rel = max(RECORD, key=lambda r: r["rel_l2"])
    worst_abs = max(RECORD, key=lambda r: r["max_abs"])
    above = sum(r["n_above_3e-2"] for r in RECORD)
    n = sum(r["n"] for r in RECORD)
    terminalreporter.write_line(
        f"parity: {len(RECORD)} comparisons over {n} elements; worst rel_l2 {worst_rel['rel_l2']:.3e} "
        f"({worst_rel['test']}); worst max_abs {worst_abs['max_abs']:.4e} ({worst_abs['test']}); "
        f"{above} elements above 3e-2")
    path = os.environ.get("KVX_PARITY_RECORD")
    if path:
        with open(path, "w") as f:
            for r in RECORD:
                f.write(json.dumps(r) + "\n")
