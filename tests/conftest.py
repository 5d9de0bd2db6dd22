import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built CUDA library")
    config.addinivalue_line("markers", "slow: full-size parity case (minutes of CPU oracle time)")


@pytest.fixture(scope="session")
def ppo():
    """The CPU oracle module, built on first use."""
    import oracle
    oracle.load()
    return oracle


@pytest.fixture(scope="session")
def pp():
    """The CUDA library binding; GPU tests fail (not skip) when it cannot load."""
    import torch
    if not torch.cuda.is_available():
        pytest.fail("GPU test run without a CUDA device")
    from paper_2605_28283_gb300 import binding
    binding.load()
    return binding
