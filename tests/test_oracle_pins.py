"""The fp64 oracle against closed forms, hand-worked cases, invariants and brute force."""
import pytest

import oracle
from tests.oracle_pins import ALL_PINS


@pytest.mark.parametrize("pin", ALL_PINS, ids=[p.__name__ for p in ALL_PINS])
def test_oracle_pin(pin):
    pin(oracle.get())


def test_oracle_threading_does_not_change_results():
    """The oracle splits rows (full) and sequences (mean) over host threads; every
    work item is computed by one thread in order, so any thread count gives the
    same bits."""
    import numpy as np
    import workloads
    inp = workloads.make_inputs(workloads.small_case(B=2, D=12, N=4, H=5, W=6, seed=71))
    u = oracle.cross_scan(inp.x)
    args = (u, inp.draw, inp.A, inp.Bs, inp.Cs, inp.Dskip, inp.bias)
    y1 = oracle.selective_scan(*args, nthreads=1)
    y7 = oracle.selective_scan(*args, nthreads=7)
    assert np.array_equal(y1, y7)
    m1, b1 = oracle.mean_scan(*args, nthreads=1)
    m3, b3 = oracle.mean_scan(*args, nthreads=3)
    assert np.array_equal(m1, m3) and np.array_equal(b1, b3)
