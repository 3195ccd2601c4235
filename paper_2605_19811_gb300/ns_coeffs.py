"""Coefficient tables for the odd-polynomial msign iterations (Section 2:
classical Newton-Schulz, the minimax-optimised "Polar Express" iteration and
Chebyshev-type accelerations all map each singular value s of the normalised
matrix by s -> a_k s + b_k s^3 + c_k s^5 per iteration, at the same cost).

A table is a tuple of (a_k, b_k, c_k) triples, one per iteration, passed to
``LionMuon(..., ns_coeffs=table)`` or ``msign_ns_coeffs``.  This is host code
that runs once when a configuration is made; the GPU kernels only read the
triples.

The minimax tables are built by the Remez exchange algorithm: for the current
interval [l, u] of singular values, the best odd polynomial of degree 3 or 5
approximating 1 in the max norm is the one whose error 1 - p alternates in
sign with equal magnitude E at l, at the interior critical points of p, and
at u (Chebyshev's alternation theorem).  The exchange solves that linear
system, moves the interior points to the critical points of the new p, and
repeats until they stop moving.  The next interval is the image of the
current one: l' = p(l) = 1 - E and u' = max p = 1 + E (divided by the safety
factor when one is used).  After the Frobenius normalisation that the NS
kernels apply, the first interval is [l_0, 1].
"""

from __future__ import annotations

import math
from typing import Tuple

import numpy as np

Triple = Tuple[float, float, float]

MUON_QUINTIC: Triple = (3.4445, -4.7750, 2.0315)
NEWTON_SCHULZ_CUBIC: Triple = (1.5, -0.5, 0.0)


def constant(triple: Triple, steps: int) -> Tuple[Triple, ...]:
    """The same polynomial in every iteration (classical NS)."""
    return tuple(tuple(float(v) for v in triple) for _ in range(steps))


def _critical_points(q: np.ndarray, lo: float, hi: float):
    """Roots of p'(x) = sum_j (2j+1) q_j x^(2j) in (lo, hi), via y = x^2."""
    dcoef = [(2 * j + 1) * q[j] for j in range(len(q))]      # in powers of y
    if len(dcoef) == 2:
        ys = [-dcoef[0] / dcoef[1]] if dcoef[1] != 0 else []
    else:
        ys = [complex(y) for y in np.roots(dcoef[::-1])]
    xs = []
    for y in ys:
        y = complex(y)
        if abs(y.imag) <= 1e-12 * max(1.0, abs(y.real)) and lo * lo < y.real < hi * hi:
            xs.append(math.sqrt(y.real))
    return sorted(xs)


def remez_odd(lo: float, hi: float, degree: int, max_iter: int = 200, tol: float = 1e-15):
    """Minimax odd polynomial of degree 3 or 5 for the constant 1 on
    [lo, hi] (0 < lo < hi).  Returns (q, E): q the coefficients of x, x^3
    [, x^5] and E the equal-ripple error."""
    if degree not in (3, 5):
        raise ValueError("degree must be 3 or 5")
    if not (0.0 < lo < hi):
        raise ValueError("need 0 < lo < hi")
    d = (degree + 1) // 2            # number of coefficients
    # reference: lo, d - 1 interior points, hi
    inner = [lo + (hi - lo) * 0.5 * (1 - math.cos(math.pi * i / d)) for i in range(1, d)]
    q = np.zeros(d)
    E = 0.0
    for _ in range(max_iter):
        pts = [lo] + inner + [hi]
        M = np.zeros((d + 1, d + 1))
        for i, x in enumerate(pts):
            for j in range(d):
                M[i, j] = x ** (2 * j + 1)
            M[i, d] = (-1.0) ** i           # p(x_i) + (-1)^i E = 1
        sol = np.linalg.solve(M, np.ones(d + 1))
        q, E = sol[:d], float(sol[d])
        crit = _critical_points(q, lo, hi)
        if len(crit) != d - 1:
            break
        moved = max(abs(a - b) for a, b in zip(crit, inner))
        inner = crit
        if moved <= tol * hi:
            break
    return q, abs(E)


def minimax_table(steps: int, lo: float = 1e-3, degree: int = 5, safety: float = 1.0):
    """Per-iteration minimax coefficients for ``steps`` iterations starting
    from singular values in [lo, 1]; degree 5 is the Polar Express
    construction, degree 3 the Chebyshev-type (cubic) one.  ``safety`` >= 1
    divides every polynomial (a margin against rounding in low precision)."""
    if safety < 1.0:
        raise ValueError("safety must be >= 1")
    out = []
    l, u = float(lo), 1.0
    for _ in range(steps):
        q, E = remez_odd(l, u, degree)
        q = q / safety
        trip = (float(q[0]), float(q[1]), float(q[2]) if degree == 5 else 0.0)
        out.append(trip)
        l_next = sum(q[j] * l ** (2 * j + 1) for j in range(len(q)))
        u = (1.0 + E) / safety
        l = float(l_next)
        if not (0.0 < l < u):
            raise ValueError("interval collapsed; use fewer steps or a larger lo")
        if u - l < 1e-9:
            # interval converged to 1: the remaining iterations keep it there
            # with the polynomial of maximal order at 1
            tail = (1.875, -1.25, 0.375) if degree == 5 else NEWTON_SCHULZ_CUBIC
            out.extend([tail] * (steps - len(out)))
            break
    return tuple(out)


def polar_express(steps: int = 5, lo: float = 1e-3, safety: float = 1.0):
    """Degree-5 minimax (Polar Express) table."""
    return minimax_table(steps, lo, 5, safety)


def chebyshev_cubic(steps: int = 5, lo: float = 1e-3, safety: float = 1.0):
    """Degree-3 minimax (Chebyshev-type) table; c_k = 0."""
    return minimax_table(steps, lo, 3, safety)
