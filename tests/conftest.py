import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a GB300 (sm_103a) and the CUDA library")
    config.addinivalue_line("markers", "slow: full-size cases (minutes on the CPU oracle)")


@pytest.fixture(scope="session")
def torch_threads():
    import torch
    torch.set_num_threads(min(16, os.cpu_count() or 1))
    return torch.get_num_threads()
