"""The oracle against its committed regression fixtures (tests/golden/make_golden.py)."""
import os

import numpy as np
import pytest

from tests.golden.make_golden import HERE, tiny_outputs


def _load(name):
    path = os.path.join(HERE, f"oracle_tiny_{name}.txt")
    lines = open(path).read().splitlines()
    shape = tuple(int(s) for s in lines[1].split("shape ")[1].split(";")[0].split())
    return np.array([float(v) for v in lines[2:]]).reshape(shape)


@pytest.mark.parametrize("name", ["u", "y_full", "out_full", "y_mean", "ybar", "out_mean", "dA", "dBu", "scan_only",
                                  "scan_only_mean", "ybar_grouped3", "selection_delta", "selection_B"])
def test_oracle_matches_fixture(name):
    np.testing.assert_allclose(tiny_outputs()[name], _load(name), rtol=1e-13, atol=1e-15)
