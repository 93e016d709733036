import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: long-running on CPU")


@pytest.fixture
def force_plan():
    """Force a tile shape / chunk count of the full scan ("shape[,chunks]") or a
    chunk length of the channel-mean scan through libvmb's test-only controls
    (declared in paper_2412_16602_gb300/csrc/vmb_testing.h, not in the public
    header); the planners are restored when the test ends."""
    import ctypes
    import types

    import paper_2412_16602_gb300 as vmb

    lib = vmb.lib
    lib.vmb_testing_force_full_plan.argtypes = [ctypes.c_int, ctypes.c_int]
    lib.vmb_testing_force_full_plan.restype = ctypes.c_int
    lib.vmb_testing_force_mean_chunk.argtypes = [ctypes.c_int]
    lib.vmb_testing_force_mean_chunk.restype = ctypes.c_int

    def full(spec: str):
        shape, _, chunks = str(spec).partition(",")
        assert lib.vmb_testing_force_full_plan(int(shape), int(chunks or 0)) == 0

    def mean(tc):
        assert lib.vmb_testing_force_mean_chunk(int(tc)) == 0

    try:
        yield types.SimpleNamespace(full=full, mean=mean)
    finally:
        lib.vmb_testing_force_full_plan(-1, 0)
        lib.vmb_testing_force_mean_chunk(0)
