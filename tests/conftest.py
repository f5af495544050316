import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a GB300 (sm_103a) GPU and the CUDA library")


def gpu_available() -> bool:
    try:
        import torch
        return torch.cuda.is_available()
    except Exception:
        return False


@pytest.fixture(scope="session")
def davet():
    """The CUDA library binding; GPU tests fail loudly if it cannot load."""
    if not gpu_available():
        pytest.fail("gpu test selected but no CUDA device is visible")
    import paper_2608_01821_gb300 as pkg
    return pkg.load()
