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
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: long-running GPU parity case at full size")


def pytest_collection_modifyitems(config, items):
    try:
        import torch

        have_gpu = torch.cuda.is_available()
    except Exception:  # pragma: no cover
        have_gpu = False
    if have_gpu:
        return
    skip = pytest.mark.skip(reason="no CUDA device in this process")
    for item in items:
        if "gpu" in item.keywords:
            item.add_marker(skip)


def pytest_sessionfinish(session, exitstatus):
    """Write the raw parity figures of the full-size checks (max and mean
    |err| against the oracle) to the file AOH_PARITY_LOG names, if any."""
    path = os.environ.get("AOH_PARITY_LOG")
    if not path:
        return
    mod = sys.modules.get("gpu_cases")
    figs = getattr(mod, "FIGURES", None) if mod else None
    if not figs:
        return
    import json
    with open(path, "w") as f:
        for name in sorted(figs):
            f.write(json.dumps(dict(check=name, **figs[name])) + "\n")
