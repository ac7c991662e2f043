import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)
TESTS = os.path.dirname(os.path.abspath(__file__))
if TESTS not in sys.path:
    sys.path.insert(0, TESTS)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built libasd.so")


@pytest.fixture(scope="session")
def oracle_lib():
    from oracle import oracle
    return oracle.load_library()


@pytest.fixture(scope="session")
def asd():
    """The CUDA binding; a GPU test fails loudly if the library or the GPU is missing."""
    import torch
    if not torch.cuda.is_available():
        pytest.fail("a gpu-marked test ran without a CUDA device")
    from paper_2608_03447_gb300 import asd as binding
    binding.load()
    return binding
