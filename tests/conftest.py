import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA device (GB300, sm_103a) and the built library")


@pytest.fixture
def dw_schedule():
    """Forces the schedule of the weight-gradient work for one test ("split" or "tail")
    and restores the previous setting afterwards."""
    from paper_2406_06385_gb300 import lrqat as LQ
    before = LQ.dw_schedule()
    yield LQ.set_dw_schedule
    LQ.set_dw_schedule(before)


@pytest.fixture
def gemm_variant():
    """Forces the kernel of the forward and dX GEMMs for one test ("pair" or "single") and
    restores the previous setting afterwards."""
    from paper_2406_06385_gb300 import lrqat as LQ
    before = LQ.gemm_variant()
    yield LQ.set_gemm_variant
    LQ.set_gemm_variant(before)


@pytest.fixture
def lowrank_path():
    """Forces the source of the GEMMs' low-rank term for one test ("tile" or "codes") and
    restores the previous setting afterwards."""
    from paper_2406_06385_gb300 import lrqat as LQ
    before = LQ.lowrank_path()
    yield LQ.set_lowrank_path
    LQ.set_lowrank_path(before)
