import json
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA device (GB300); parity tests through the C ABI")
    config.addinivalue_line("markers", "slow: longer CPU case")


def pytest_collection_modifyitems(config, items):
    import torch
    if torch.cuda.is_available():
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for it in items:
        if "gpu" in it.keywords:
            it.add_marker(skip)


def pytest_terminal_summary(terminalreporter):
    """The parity tests' exclusion counts per workload (ill-conditioned outputs, uncertain
    decisions, kept entries); also written as JSON to $EMR_PARITY_REPORT when set."""
    pu = sys.modules.get("parity_util")
    if pu is None or not pu.REPORT:
        return
    for line in pu.report_lines():
        terminalreporter.write_line(line)
    path = os.environ.get("EMR_PARITY_REPORT")
    if path:
        with open(path, "w") as f:
            json.dump(pu.REPORT, f, indent=1, sort_keys=True)
