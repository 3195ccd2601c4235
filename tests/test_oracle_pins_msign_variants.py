"""Pins for the oracle's iteration-dependent msign polynomials (Section 2
names the minimax "Polar Express" and Chebyshev-type iterations beside
classical Newton-Schulz): the NS recurrence with a coefficient table, and the
minimax odd polynomial / coefficient schedule.  Each check rests on something
other than the oracle itself: an exactly known SVD with the singular-value
maps composed by hand, the closed form of the minimax odd cubic, the
equioscillation property of a minimax polynomial, random perturbations that
must not beat the optimum, and the interval bookkeeping of the schedule."""

import math

import numpy as np
import pytest

import oracle as O
from tests.test_oracle_pins import known_svd_matrix


def _cubic_minimax_closed_form(lo, hi):
    """Best odd cubic p(x) = alpha x + beta x^3 for 1 on [lo, hi], derived by
    hand from the alternation at lo (+E), x* (-E), hi (+E): p(lo) = p(hi),
    p'(x*) = 0, p(lo) + p(x*) = 2.  With S = hi^2 + hi lo + lo^2:
    x*^2 = S / 3, alpha = -beta S, beta = -2 / (lo (S - lo^2) + (2S/3) sqrt(S/3))."""
    S = hi * hi + hi * lo + lo * lo
    beta = -2.0 / (lo * (S - lo * lo) + (2.0 * S / 3.0) * math.sqrt(S / 3.0))
    alpha = -beta * S
    E = 1.0 - (alpha * lo + beta * lo ** 3)
    return np.array([alpha, beta]), E


@pytest.mark.parametrize("lo,hi", [(0.2, 1.0), (1e-3, 1.0), (0.05, 1.7), (0.5, 1.2)])
def test_minimax_cubic_matches_closed_form(lo, hi):
    q, E = O.minimax_odd_polynomial(lo, hi, 3)
    q_ref, E_ref = _cubic_minimax_closed_form(lo, hi)
    np.testing.assert_allclose(q, q_ref, rtol=2e-6)
    assert abs(E - E_ref) <= 2e-6 * max(E_ref, 1e-3)


def _odd_p_prime_roots(q, lo, hi):
    """Interior critical points of p(x) = sum q_j x^(2j+1): roots y = x^2 of
    sum (2j+1) q_j y^j inside (lo^2, hi^2)."""
    coef = [(2 * j + 1) * qj for j, qj in enumerate(q)]
    ys = np.roots(coef[::-1])
    xs = sorted(math.sqrt(y.real) for y in ys
                if abs(y.imag) < 1e-12 and lo * lo < y.real < hi * hi)
    return xs


@pytest.mark.parametrize("lo,hi", [(1e-3, 1.0), (0.1, 1.0), (0.02, 1.9), (0.6, 1.3)])
def test_minimax_quintic_equioscillates(lo, hi):
    """Chebyshev alternation: the error 1 - p of the best odd quintic takes
    +E, -E, +E, -E at lo, x1, x2, hi (x1 < x2 the critical points of p)."""
    q, E = O.minimax_odd_polynomial(lo, hi, 5)
    xs = _odd_p_prime_roots(q, lo, hi)
    assert len(xs) == 2
    pts = [lo, xs[0], xs[1], hi]
    err = 1.0 - O.odd_poly_eval(q, np.array(pts))
    want = np.array([E, -E, E, -E])
    np.testing.assert_allclose(err, want, rtol=0, atol=1e-6 * max(E, 1e-2))
    dense = np.linspace(lo, hi, 200001)
    assert np.abs(1.0 - O.odd_poly_eval(q, dense)).max() <= E * (1 + 1e-6)


@pytest.mark.parametrize("degree", [3, 5])
def test_minimax_is_not_beaten_by_perturbations(degree):
    lo, hi = 0.03, 1.0
    q, E = O.minimax_odd_polynomial(lo, hi, degree)
    x = np.linspace(lo, hi, 20001)
    r = np.random.default_rng(5)
    for _ in range(300):
        dq = q + r.normal(0, 1e-3, size=q.shape) * np.abs(q)
        assert np.abs(1.0 - O.odd_poly_eval(dq, x)).max() >= E - 1e-7


def test_ns_schedule_closed_form_on_known_svd():
    """NS with distinct (a_k, b_k, c_k) per iteration: each normalised
    singular value goes through phi_1, then phi_2, then phi_3 (composed by hand
    here), so the order of the table matters."""
    table = ((3.0, -3.2, 1.2), (2.0, -1.5, 0.45), (1.875, -1.25, 0.375))
    s, l = 16, 64
    sigma = np.linspace(0.1, 2.0, s)[::-1]
    for tall in (False, True):
        G, U, V = known_svd_matrix(s, l, sigma, seed=3, tall=tall)
        eps = 1e-7
        got = O.ns_polynomial_schedule(G, table, eps)
        x = sigma / (np.linalg.norm(sigma) + eps)
        x1 = 3.0 * x - 3.2 * x ** 3 + 1.2 * x ** 5
        x2 = 2.0 * x1 - 1.5 * x1 ** 3 + 0.45 * x1 ** 5
        x3 = 1.875 * x2 - 1.25 * x2 ** 3 + 0.375 * x2 ** 5
        want = U @ np.diag(x3) @ V.T
        if tall:
            want = want.T
        np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)
        np.testing.assert_allclose(O.ns_scalar_map_schedule(x, table), x3, rtol=0, atol=1e-15)


def test_ns_schedule_constant_table_is_classical_ns():
    r = np.random.default_rng(2)
    G = r.normal(size=(24, 40))
    np.testing.assert_allclose(O.ns_polynomial_schedule(G, (O.NS_QUINTIC,) * 5, 1e-7),
                               O.ns_polynomial(G, 5, *O.NS_QUINTIC, 1e-7), rtol=0, atol=1e-14)


@pytest.mark.parametrize("degree,steps", [(5, 5), (3, 6)])
def test_minimax_schedule_maps_interval_forward(degree, steps):
    """The construction keeps every singular value of [l_0, 1] inside the
    tracked interval: after k steps the composed map sends [l_0, 1] into
    [l_k, u_k], with l_k = composed map at l_0 (the bottom is the image of the
    bottom) and u_k - 1 = 1 - l_k (minimax equioscillation)."""
    lo = 1e-3
    table = O.minimax_schedule(steps, lo, degree)
    assert len(table) == steps
    x = np.concatenate([np.geomspace(lo, 1.0, 4001), np.linspace(lo, 1.0, 4001)])
    y = O.ns_scalar_map_schedule(x, table)
    l_k = O.ns_scalar_map_schedule(np.array([lo]), table)[0]
    # the LP works on a grid, so its polynomial equioscillates only to ~1e-7
    assert y.min() >= l_k - 1e-6
    assert y.max() <= 2.0 - l_k + 1e-5
    # every step moves the bottom of the interval up
    ls = [O.ns_scalar_map_schedule(np.array([lo]), table[:k])[0] for k in range(steps + 1)]
    assert all(b > a for a, b in zip(ls, ls[1:]))


def test_polar_express_beats_constant_quintic_on_spread_spectrum():
    """Section 2 lists the minimax iteration as a better-tuned variant of the
    same per-step cost: on singular values spread over [1e-3, 1] its 5-step
    table leaves a smaller worst-case distance to 1 than the constant
    quintic."""
    table = O.minimax_schedule(5, 1e-3, 5)
    x = np.geomspace(1e-3, 1.0, 2001)
    err_pe = np.abs(O.ns_scalar_map_schedule(x, table) - 1.0).max()
    err_q = np.abs(O.ns_scalar_map(x, 5, *O.NS_QUINTIC) - 1.0).max()
    assert err_pe < err_q


def test_bf16_storage_ns_on_hadamard_follows_hand_rounded_scalars():
    """For G = c H (H a 16 x 16 orthogonal Hadamard matrix, entries +-1/4)
    every intermediate is a scalar multiple of I or H, so the stored values
    follow a scalar recurrence whose roundings can be done by hand with
    torch's bf16 conversion: with eps = 0 the normalised singular value is
    x = 1/4 (||H||_F = 4), A = bf16(x^2) I, B = bf16(b A + c A^2) I and
    X <- bf16(a X + B X) entrywise."""
    import torch
    from tests.test_oracle_pins import hadamard

    def r(v):
        return float(torch.tensor(v, dtype=torch.float64).to(torch.bfloat16).to(torch.float64))

    H = hadamard(16)
    assert np.allclose(H @ H.T, np.eye(16))
    table = ((3.4445, -4.7750, 2.0315), (8.47, -25.1, 18.63), (2.0, -1.5, 0.45))
    got = O.ns_polynomial_schedule_storage(3.0 * H, table, 0.0, "bf16")
    # entries of X are +-h with h = x / 4 (x the singular value of X)
    h = r(3.0 * 0.25)              # X_0 = bf16(G): entries 3/4
    inv = 1.0 / 12.0               # ||3 H||_F = 12
    for k, (a, b, c) in enumerate(table):
        sa, sx = (inv * inv, inv) if k == 0 else (1.0, 1.0)
        A = r(sa * 16 * h * h)     # X X^T = 16 h^2 I
        B = r(b * A + c * A * A)
        h = r(sx * (a * h + B * h))
    want = h * (H * 4.0)           # H * 4 has entries +-1
    np.testing.assert_array_equal(got, want)


def test_bf16_storage_ns_tracks_exact_recurrence():
    """bf16 storage perturbs the constant quintic by about the bf16 spacing
    amplified a little, not by orders of magnitude, and not at all in the
    limit of no rounding (checked through the Hadamard case above)."""
    r = np.random.default_rng(4)
    G = r.normal(size=(64, 160))
    ex = O.ns_polynomial_schedule(G, (O.NS_QUINTIC,) * 5, 1e-7)
    em = O.ns_polynomial_schedule_storage(G, (O.NS_QUINTIC,) * 5, 1e-7, "bf16")
    e = np.linalg.norm(em - ex) / np.linalg.norm(ex)
    assert 2.0 ** -10 < e < 5e-2
    ef = O.ns_polynomial_schedule_storage(G, (O.NS_QUINTIC,) * 5, 1e-7, "f32")
    e32 = np.linalg.norm(ef - ex) / np.linalg.norm(ex)
    assert 2.0 ** -26 < e32 < 1e-5
