"""Pins for the oracle's adaptive Muon/Lion selection (Appendix G: Muon on a
matrix whose momentum has stable rank ||M||_F^2 / sigma_1_hat^2 at most
alpha * min(m, n), sigma_1 from a few power-iteration steps): the published
first outputs of SplitMix64, the power-iteration estimate on an exactly
known SVD written out in closed form, the Rayleigh bound, matrices whose
stable rank is known exactly, the threshold, and the step routing."""

import numpy as np
import pytest

import oracle as O
from tests.test_oracle_pins import known_svd_matrix, orth


def test_splitmix64_published_outputs():
    """The first three outputs from seed 0 of the reference SplitMix64."""
    assert O.splitmix64(0, 3) == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_start_vector_range_and_determinism():
    v = O.power_start_vector(1000, 7)
    assert v.shape == (1000,) and np.all(v >= -1.0) and np.all(v < 1.0)
    np.testing.assert_array_equal(v, O.power_start_vector(1000, 7))
    assert abs(v.mean()) < 0.1 and 0.25 < v.var() < 0.42          # uniform on [-1, 1): var 1/3
    z = O.splitmix64(7, 1)[0]
    assert v[0] == 2.0 * ((z >> 11) * 2.0 ** -53) - 1.0


@pytest.mark.parametrize("iters", [1, 2, 3, 5])
def test_power_estimate_closed_form_on_known_svd(iters):
    """M = U diag(sigma) V^T, c = V^T v0 / ||v0||: after k passes the estimate
    is v^T (M^T M)^(2k-1) v / v^T (M^T M)^(2k-2) v with v = v0 / ||v0||, i.e.
    sum c_i^2 sigma_i^(4(k-1)+2) / sum c_i^2 sigma_i^(4(k-1)) for k > 1 and
    sum c_i^2 sigma_i^2 for k = 1 (the denominator is then ||v||^2 = 1, null
    space included)."""
    s, l = 16, 64
    sigma = np.linspace(0.3, 2.0, s)[::-1]
    for tall in (False, True):
        M, U, V = known_svd_matrix(s, l, sigma, seed=5, tall=tall)
        n = M.shape[1]
        v0 = O.power_start_vector(n, 3)
        fro2, sig2 = O.stable_rank_estimate(M, iters, v0)
        right = U if tall else V                                  # right singular vectors of M
        c = right.T @ (v0 / np.linalg.norm(v0))
        p = 4 * (iters - 1)
        den = 1.0 if iters == 1 else np.sum(c ** 2 * sigma ** p)
        want = np.sum(c ** 2 * sigma ** (p + 2)) / den
        assert abs(sig2 - want) <= 1e-12 * want
        assert abs(fro2 - np.sum(sigma ** 2)) <= 1e-12 * fro2


def test_estimate_never_exceeds_sigma1_and_converges():
    r = np.random.default_rng(0)
    M = r.normal(size=(60, 90))
    s1 = np.linalg.svd(M, compute_uv=False)[0]
    last = 0.0
    for k in range(1, 40):
        _, sig2 = O.stable_rank_estimate(M, k, O.power_start_vector(90, 0))
        assert sig2 <= s1 * s1 * (1 + 1e-12)
        assert sig2 >= last * (1 - 1e-12)                         # monotone in k
        last = sig2
    # the top singular values of a Gaussian matrix lie close together, so convergence is slow
    assert abs(last - s1 * s1) <= 1e-2 * s1 * s1


def test_exact_stable_ranks():
    """Rank one a b^T: stable rank 1 from the second pass on (the first pass
    gives ||a||^2 (b . v)^2 for the unit start v); a multiple of an orthogonal
    matrix: stable rank n for any start and any number of passes."""
    a = np.arange(1.0, 13.0)
    b = np.linspace(-1, 2, 20)
    v = O.power_start_vector(20, 1)
    fro2, sig2 = O.stable_rank_estimate(np.outer(a, b), 1, v)
    assert abs(sig2 - (a @ a) * (b @ v / np.linalg.norm(v)) ** 2) <= 1e-12 * sig2
    for k in (2, 4):
        fro2, sig2 = O.stable_rank_estimate(np.outer(a, b), k, v)
        assert abs(fro2 / sig2 - 1.0) < 1e-12
    Q = 3.0 * orth(16, 4)                                         # square: exact from the first pass
    for k in (1, 3):
        fro2, sig2 = O.stable_rank_estimate(Q, k, O.power_start_vector(16, 2))
        assert abs(fro2 / sig2 - 16.0) < 1e-10
    Qw = 3.0 * orth(32, 4)[:16, :]            # 16 x 32: exact once v has left the null space (pass 2 on)
    for k in (2, 3):
        fro2, sig2 = O.stable_rank_estimate(Qw, k, O.power_start_vector(32, 2))
        assert abs(fro2 / sig2 - 16.0) < 1e-10
    fro2, sig2 = O.stable_rank_estimate(Qw, 1, O.power_start_vector(32, 2))
    assert fro2 / sig2 > 16.0


def test_threshold_and_zero_buffer():
    """sigma = (4, 1, 1, ...): stable rank (16 + 15) / 16 = 31/16 for a 16 x 48
    matrix, known exactly once the power iteration has converged; Muon iff
    alpha * 16 >= 31/16."""
    sigma = np.array([4.0] + [1.0] * 15)
    M, _, _ = known_svd_matrix(16, 64, sigma, seed=9)
    cfg = O.Config(schedule="stable_rank", srank_iters=30)
    srank = 31.0 / 16.0
    for alpha, want in [(srank / 16 * 1.01, True), (srank / 16 * 0.99, False), (1.0, True), (0.01, False)]:
        cfg.srank_alpha = alpha
        assert O.srank_takes_muon(M, cfg) is want
    assert O.srank_takes_muon(np.zeros((8, 12)), cfg) is True


def test_step_routes_matrices_by_stable_rank():
    """Under schedule="stable_rank" a matrix whose buffer is rank one takes the
    Muon branch and a full-rank noise buffer the Lion branch, at any t; vectors
    keep the Lion step."""
    r = np.random.default_rng(1)
    cfg = O.Config(schedule="stable_rank", srank_alpha=0.05, period=2)
    shapes = [(24, 40), (24, 40), (40,)]
    W = [r.normal(size=s) for s in shapes]
    G = [r.normal(size=s) for s in shapes]
    M = [np.outer(r.normal(size=24), r.normal(size=40)), r.normal(size=(24, 40)), r.normal(size=40)]
    for t in (1, 2):                                              # a Lion step and a Muon step of P = 2
        P1, M1 = O.lionmuon_step(W, G, M, t, cfg)
        gh = [O.interpolated_direction(M[i], G[i], cfg.beta1) for i in range(3)]
        np.testing.assert_allclose(P1[0], O.muon_update(W[0], gh[0], cfg), rtol=0, atol=1e-15)
        np.testing.assert_allclose(P1[1], O.lion_update(W[1], gh[1], cfg.eta_lion, cfg.weight_decay),
                                   rtol=0, atol=1e-15)
        np.testing.assert_allclose(P1[2], O.lion_update(W[2], gh[2], cfg.eta_lion, cfg.weight_decay),
                                   rtol=0, atol=1e-15)
        for i in range(3):
            np.testing.assert_allclose(M1[i], O.momentum_update(M[i], G[i], cfg.beta2), rtol=0, atol=1e-15)


def test_decision_uses_the_buffer_before_the_update():
    """At a zero M_{t-1} the rule takes Muon (the zero-buffer reading), while
    the updated buffer (1 - beta2) G of a noise gradient would select Lion."""
    r = np.random.default_rng(2)
    cfg = O.Config(schedule="stable_rank", srank_alpha=0.05, period=2)
    W = [r.normal(size=(24, 40))]
    G = [r.normal(size=(24, 40))]
    P1, _ = O.lionmuon_step(W, G, [np.zeros((24, 40))], 1, cfg)
    gh = O.interpolated_direction(np.zeros((24, 40)), G[0], cfg.beta1)
    np.testing.assert_allclose(P1[0], O.muon_update(W[0], gh, cfg), rtol=0, atol=1e-15)
    assert not O.srank_takes_muon(O.momentum_update(np.zeros((24, 40)), G[0], cfg.beta2), cfg)
