"""Shared pytest configuration: the ``gpu`` marker and repo-root import path."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: long-running (full-size workload) test")


import json  # noqa: E402

import pytest  # noqa: E402


@pytest.fixture
def parity_report(request):
    """Records measured deviations of a parity test (a dict per call).

    With TRACK_PARITY_REPORT naming a file, each record is appended to it as one
    JSON line with the test's id; otherwise records are only kept in the test's
    user properties."""
    path = os.environ.get("TRACK_PARITY_REPORT")

    def report(**fields):
        rec = {"test": request.node.nodeid, **fields}
        request.node.user_properties.append(("parity", rec))
        if path:
            with open(path, "a") as f:
                f.write(json.dumps(rec) + "\n")
    return report
