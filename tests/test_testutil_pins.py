"""CPU pins of the test helpers that stand in for the oracle at full size:
the SVD closed form of the Newton-Schulz iteration (lm_testutil.
ns_closed_form_rows) equals the oracle's recurrence (oracle.ns_polynomial)
to fp64 rounding, for wide, tall and square inputs, every row or a sample."""

import numpy as np
import pytest

import oracle as O
from tests.lm_testutil import ns_closed_form_rows, tall


@pytest.mark.parametrize("shape", [(300, 700), (700, 300), (256, 256), (64, 2000)])
@pytest.mark.parametrize("coeffs,steps", [(O.NS_QUINTIC, 5), ((1.5, -0.5, 0.0), 8), ((0.0, 1.0, 0.0), 1)])
def test_closed_form_equals_recurrence(shape, coeffs, steps):
    rng = np.random.default_rng(sum(shape))
    G = rng.standard_normal(shape) * 1e-3
    want = tall(O.ns_polynomial(G, steps, *coeffs, 1e-7))
    got = ns_closed_form_rows(G, steps, *coeffs, 1e-7)
    assert np.linalg.norm(got - want) <= 1e-10 * np.linalg.norm(want)
    rows = np.sort(rng.choice(max(shape), 37, replace=False))
    np.testing.assert_allclose(ns_closed_form_rows(G, steps, *coeffs, 1e-7, rows=rows), want[rows],
                               rtol=0, atol=1e-10 * np.abs(want).max())
