import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line(
        "markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")
    config.addinivalue_line(
        "markers", "slow: long-running CPU test")


def cuda_available() -> bool:
    try:
        import torch
        return torch.cuda.is_available()
    except Exception:  # pragma: no cover
        return False


@pytest.fixture(scope="session")
def gpu():
    """Skip-free GPU guard: a gpu-marked test on a machine without a GPU is
    an error in the run configuration, so fail loudly instead of skipping."""
    if not cuda_available():
        pytest.fail("test marked gpu but no CUDA device is visible")
    import torch
    return torch.device("cuda:0")


def pytest_sessionfinish(session, exitstatus):
    """With LAMB_FLOOR_STATS set, write how often the parity tolerance floors
    decided a comparison (gpu_util.FLOOR_STATS) to that file as JSON."""
    path = os.environ.get("LAMB_FLOOR_STATS")
    if not path:
        return
    try:
        import gpu_util
    except Exception:  # pragma: no cover - CPU-only runs
        return
    import json
    with open(path, "w") as f:
        json.dump(gpu_util.FLOOR_STATS, f, indent=1, sort_keys=True)
