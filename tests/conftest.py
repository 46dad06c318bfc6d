import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a GB300 (sm_103a) GPU and the built CUDA library")
    config.addinivalue_line("markers", "slow: long-running oracle comparison (opt-in via FBOB_SLOW=1)")


def pytest_collection_modifyitems(config, items):
    if os.environ.get("FBOB_SLOW") == "1":
        return
    skip = pytest.mark.skip(reason="slow oracle comparison: set FBOB_SLOW=1")
    for it in items:
        if "slow" in it.keywords:
            it.add_marker(skip)


def pytest_sessionfinish(session, exitstatus):
    out = os.environ.get("FBOB_PARITY_REPORT")
    if not out:
        return
    try:
        from tests import gpu_util
    except Exception:
        return
    import json
    with open(out, "w") as fh:
        json.dump([{"test": t, "tensor": n, "rel_fro": r, "max_abs_rel": m}
                   for t, n, r, m in gpu_util.RECORD], fh, indent=0)
