import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a); runs through the C-ABI library")
    config.addinivalue_line("markers", "slow: full-size cases (seconds to minutes)")


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


@pytest.fixture
def tuning(monkeypatch):
    """Set GBMLA_* testing variables (kernel tiling) for one test.  The
    library reads them once per process, so each change is followed by
    mla_reload_tuning, and the defaults are restored and re-read afterwards."""
    from paper_2607_27269_gb300 import abi

    def apply(**env):
        for k, v in env.items():
            monkeypatch.setenv(k, str(v))
        abi.reload_tuning()

    yield apply
    monkeypatch.undo()
    abi.reload_tuning()
