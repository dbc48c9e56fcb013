import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (runs the sm_103a library)")


GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


@pytest.fixture(scope="session")
def golden_dir():
    return GOLDEN


@pytest.fixture(scope="session")
def p4q():
    """The CUDA binding, with the library built for sm_103a (GPU tests only)."""
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2609_34867_gb300 import build, p4q as binding
    build.build()
    binding.lib()
    return binding


@pytest.fixture(scope="session")
def dev():
    import torch
    return torch.device("cuda:0")
