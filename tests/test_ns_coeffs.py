"""The product's coefficient tables for iteration-dependent msign polynomials
(paper_2605_19811_gb300/ns_coeffs.py, a Remez exchange) against the oracle's
independent construction (a linear program on a dense grid): the same
minimax polynomials and the same schedules."""

import numpy as np
import pytest

import oracle as O
from paper_2605_19811_gb300 import ns_coeffs as C


@pytest.mark.parametrize("lo,hi,degree", [(1e-3, 1.0, 5), (0.1, 1.0, 5), (0.02, 1.9, 5), (0.6, 1.3, 5),
                                          (0.2, 1.0, 3), (1e-3, 1.0, 3), (0.05, 1.7, 3)])
def test_remez_matches_lp_oracle(lo, hi, degree):
    q, E = C.remez_odd(lo, hi, degree)
    q_ref, E_ref = O.minimax_odd_polynomial(lo, hi, degree)
    np.testing.assert_allclose(q, q_ref, rtol=1e-6, atol=1e-9 * np.abs(q_ref).max())
    assert abs(E - E_ref) <= 1e-6 * max(E_ref, 1e-3)


@pytest.mark.parametrize("degree,steps", [(5, 5), (3, 6), (5, 3)])
def test_tables_match_oracle_schedule(degree, steps):
    got = C.minimax_table(steps, 1e-3, degree)
    want = O.minimax_schedule(steps, 1e-3, degree)
    assert len(got) == len(want) == steps
    np.testing.assert_allclose(np.array(got), np.array(want), rtol=1e-6, atol=1e-9)


def test_safety_factor_divides_each_polynomial():
    base = C.polar_express(1, 1e-2)
    safe = C.polar_express(1, 1e-2, safety=1.01)
    np.testing.assert_allclose(np.array(safe[0]) * 1.01, np.array(base[0]), rtol=1e-12)
    want = O.minimax_schedule(3, 1e-2, 5, safety=1.01)
    np.testing.assert_allclose(np.array(C.polar_express(3, 1e-2, safety=1.01)), np.array(want), rtol=1e-6)


def test_converged_tail_is_order_maximising_polynomial():
    t = C.polar_express(12, 1e-3)
    assert t[-1] == (1.875, -1.25, 0.375)
    # p(1) = 1, p'(1) = 0, p''(1) = 0 for the tail polynomial
    a, b, c = t[-1]
    assert abs(a + b + c - 1) < 1e-15 and abs(a + 3 * b + 5 * c) < 1e-15 and abs(6 * b + 20 * c) < 1e-15


def test_constant_tables_and_errors():
    assert C.constant(C.MUON_QUINTIC, 3) == (C.MUON_QUINTIC,) * 3
    with pytest.raises(ValueError):
        C.remez_odd(0.0, 1.0, 5)
    with pytest.raises(ValueError):
        C.remez_odd(0.1, 1.0, 4)
    with pytest.raises(ValueError):
        C.minimax_table(3, 1e-3, 5, safety=0.5)
