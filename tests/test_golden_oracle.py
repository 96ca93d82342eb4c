"""The oracle against its stored values (tests/golden/, written by make_golden.py from
the oracle itself on seeded inputs): any change of the oracle's arithmetic shows up
here and has to be made deliberately, with the stored values rewritten in the same
commit. Integers must match exactly, floats to 1e-9 relative (BLAS summation order)."""
import json
import os

import numpy as np
import pytest

from tests.golden import make_golden as mg

HERE = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
INTS = {"topk_idx", "offsets", "schedule", "order"}


@pytest.mark.parametrize("name,fn", [("layer_tiny.json", mg.layer_values), ("train_tiny.json", mg.train_values)])
def test_oracle_matches_stored_values(name, fn):
    stored = json.load(open(os.path.join(HERE, name)))["values"]
    now = fn()
    assert set(now) == set(stored)
    for k, v in stored.items():
        if k in INTS:
            assert now[k] == v, k
        else:
            a, b = np.asarray(now[k], np.float64), np.asarray(v, np.float64)
            assert a.shape == b.shape, k
            assert np.allclose(a, b, rtol=1e-9, atol=1e-12 * max(1.0, np.abs(b).max())), k
