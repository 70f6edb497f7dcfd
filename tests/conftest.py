import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)
GOLDEN = os.path.join(ROOT, "tests", "golden")


def pytest_configure(config):
    config.addinivalue_line(
        "markers", "gpu: needs a CUDA GPU (sm_103a) and the built CUDA library")


@pytest.fixture(scope="session")
def cuda_lib():
    """The CUDA library, built in-tree.  GPU tests fail (never skip) when it or
    the GPU is missing, so a broken box cannot pass as green."""
    import torch
    if not torch.cuda.is_available():
        pytest.fail("CUDA is not available: GPU tests need a GB300")
    import paper_2607_16973_gb300 as tq
    tq.load()  # raises if libtq.so is missing
    return tq
