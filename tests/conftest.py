import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: long-running CPU test")


@pytest.fixture(scope="session")
def cuda_ok():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return True


@pytest.fixture(scope="session", autouse=True)
def _short_device_waits():
    """Kernels in the tests finish in milliseconds: give device-side waits a
    short budget so a stuck pipeline fails fast instead of waiting 2 s."""
    try:
        import torch
        if torch.cuda.is_available():
            from paper_2609_32415_gb300 import api, build
            build.build()
            api.refadapt_set_wait_budget_ns(500_000_000)
    except Exception:
        pass
    yield
