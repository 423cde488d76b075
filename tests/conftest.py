import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built libtac.so")


@pytest.fixture(scope="session")
def orc():
    import oracle
    oracle.build()
    return oracle


@pytest.fixture(scope="session")
def tac_host():
    """libtac loaded for its host-only entry points (no GPU needed)."""
    from paper_2603_27467_gb300 import build as b
    b.build()
    import paper_2603_27467_gb300 as tac
    tac.load()
    return tac


@pytest.fixture(scope="session")
def tac_gpu():
    """libtac on a CUDA device; fails (never skips) when there is none."""
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2603_27467_gb300 import build as b
    b.build()
    import paper_2603_27467_gb300 as tac
    tac.load()
    torch.cuda.init()
    return tac
