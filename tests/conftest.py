import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built libsimsd.so")


def pytest_sessionfinish(session, exitstatus):
    """With SIMSD_PARITY_LOG set, writes one JSON line per attention
    comparison (test id, error statistics, ratio to the derived bound)."""
    path = os.environ.get("SIMSD_PARITY_LOG")
    mod = sys.modules.get("tests._gpu")
    if not path or mod is None:
        return
    import json
    with open(path, "w") as f:
        for test, st in mod.PARITY_LOG:
            f.write(json.dumps({"test": test, **st}) + "\n")
