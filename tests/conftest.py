"""Shared pytest configuration: markers, the oracle build, and the GPU library handle."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA device (parity tests through the C-ABI)")
    config.addinivalue_line("markers", "slow: longer CPU test")


@pytest.fixture(scope="session")
def orc():
    """The CPU oracle module, built on first use."""
    from oracle import oracle as o
    o.build()
    return o


@pytest.fixture(scope="session")
def qs():
    """The CUDA library binding (GPU tests only)."""
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30950_gb300 as q
    q.load()
    return q
