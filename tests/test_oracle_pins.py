"""Pins for the CPU oracle: closed forms, invariants and special cases that the
paper and the mathematics fix, chosen so that a plausible slip in the oracle
(a dropped term, a wrong sign, a transposed operand, the post-update buffer,
a wrong branch) fails at least one of them.  CPU only."""

import math

import numpy as np
import pytest

import oracle as O


# ---------------------------------------------------------------------------
# helpers: exactly orthogonal matrices
# ---------------------------------------------------------------------------

def hadamard(n):
    """Sylvester Hadamard matrix scaled to be orthogonal; exact in binary
    floating point when n is a power of 4 (scale 1/2, 1/4, 1/8 ...)."""
    H = np.array([[1.0]])
    while H.shape[0] < n:
        H = np.block([[H, H], [H, -H]])
    assert H.shape[0] == n
    return H / math.sqrt(n)


def signed_perm(n, seed):
    r = np.random.default_rng(seed)
    P = np.zeros((n, n))
    P[np.arange(n), r.permutation(n)] = r.choice([-1.0, 1.0], size=n)
    return P


def orth(n, seed):
    """Exactly orthogonal: signed permutation times a scaled Hadamard."""
    return signed_perm(n, seed) @ hadamard(n) @ signed_perm(n, seed + 1000)


def known_svd_matrix(s, l, sigma, seed, tall=False):
    U = orth(s, seed)
    V = orth(l, seed + 7)[:, :s]
    G = U @ np.diag(sigma) @ V.T
    if tall:
        return G.T, U, V
    return G, U, V


# ---------------------------------------------------------------------------
# bf16 rounding and sign
# ---------------------------------------------------------------------------

def test_bf16_round_known_values():
    one = np.float32(1.0)
    cases = {
        1.0: 1.0,
        1.0 + 2.0 ** -8: 1.0,                        # tie -> even mantissa 0
        1.0 + 3 * 2.0 ** -8: 1.0 + 2.0 ** -6,        # tie -> even mantissa 2
        1.0 + 2.0 ** -8 + 2.0 ** -20: 1.0 + 2.0 ** -7,  # above tie -> up
        -(1.0 + 3 * 2.0 ** -8): -(1.0 + 2.0 ** -6),
        3.4028234663852886e38: float("inf"),         # max float32 rounds up
        3.3895313892515355e38: 3.3895313892515355e38,  # max bf16 is exact
        0.0: 0.0,
    }
    for x, want in cases.items():
        got = float(O.bf16_round(np.array([x], dtype=np.float32))[0])
        assert got == want, (x, got, want)
    assert np.isnan(O.bf16_round(np.array([np.nan], dtype=np.float32))[0])
    assert one == 1.0


def test_bf16_round_matches_torch_cpu_conversion():
    torch = pytest.importorskip("torch")
    r = np.random.default_rng(5)
    x = np.concatenate([
        r.standard_normal(20000).astype(np.float32) * np.float32(0.02),
        (r.standard_normal(20000) * 1e-39).astype(np.float32),   # subnormals
        r.uniform(-3.4e38, 3.4e38, 20000).astype(np.float32),
        np.array([0.0, -0.0, np.inf, -np.inf], dtype=np.float32),
    ])
    want = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    got = O.bf16_round(x)
    np.testing.assert_array_equal(got.view(np.uint32), want.view(np.uint32))


def test_sign_conventions():
    x = np.array([2.5, -1e-30, 0.0, -0.0, np.nan, np.inf])
    s = O.sign(x)
    assert list(s[:4]) == [1.0, -1.0, 0.0, 0.0]
    assert np.isnan(s[4]) and s[5] == 1.0


# ---------------------------------------------------------------------------
# Newton-Schulz and msign
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("s,l,tall", [(4, 16, False), (16, 64, False), (16, 16, False),
                                      (4, 64, True), (16, 64, True)])
@pytest.mark.parametrize("coeffs,steps", [(O.NS_QUINTIC, 5), (O.NS_CUBIC, 7), ((2.0, -1.3, 0.4), 3)])
def test_ns_closed_form_on_known_svd(s, l, tall, coeffs, steps):
    """For G = U diag(sigma) V^T, NS_K(G) = U diag(phi^K(sigma/(||sigma||+eps))) V^T."""
    r = np.random.default_rng(s * 100 + l)
    sigma = np.sort(r.uniform(0.05, 3.0, size=s))[::-1]
    G, U, V = known_svd_matrix(s, l, sigma, seed=s + l, tall=tall)
    eps = 1e-7
    a, b, c = coeffs
    got = O.ns_polynomial(G, steps, a, b, c, eps)
    phi = O.ns_scalar_map(sigma / (np.linalg.norm(sigma) + eps), steps, a, b, c)
    want = U @ np.diag(phi) @ V.T
    if tall:
        want = want.T
    assert got.shape == G.shape
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)


def test_ns_rank_one():
    u = np.array([1.0, -2.0, 2.0]) / 3.0
    v = np.array([2.0, 3.0, 6.0, 0.0]) / 7.0
    G = 5.0 * np.outer(u, v)
    eps = 1e-7
    got = O.ns_polynomial(G, 5, *O.NS_QUINTIC, eps)
    phi = O.ns_scalar_map(np.array([5.0 / (5.0 + eps)]), 5, *O.NS_QUINTIC)[0]
    np.testing.assert_allclose(got, phi * np.outer(u, v), atol=1e-13)


def test_ns_transpose_identity():
    r = np.random.default_rng(1)
    G = r.standard_normal((24, 40))
    a = O.ns_polynomial(G, 5, *O.NS_QUINTIC)
    b = O.ns_polynomial(G.T, 5, *O.NS_QUINTIC)
    np.testing.assert_allclose(a, b.T, atol=1e-12)


def test_ns_orthogonal_equivariance():
    r = np.random.default_rng(2)
    G = r.standard_normal((12, 20))
    Q, _ = np.linalg.qr(r.standard_normal((12, 12)))
    R, _ = np.linalg.qr(r.standard_normal((20, 20)))
    lhs = O.ns_polynomial(Q @ G @ R, 5, *O.NS_QUINTIC)
    rhs = Q @ O.ns_polynomial(G, 5, *O.NS_QUINTIC) @ R
    np.testing.assert_allclose(lhs, rhs, atol=1e-11)


def test_ns_scale_invariance():
    r = np.random.default_rng(3)
    G = r.standard_normal((10, 30))
    a = O.ns_polynomial(G, 5, *O.NS_QUINTIC, eps=0.0)
    b = O.ns_polynomial(37.5 * G, 5, *O.NS_QUINTIC, eps=0.0)
    np.testing.assert_allclose(a, b, atol=1e-12)


def test_ns_zero_steps_is_normalisation():
    r = np.random.default_rng(4)
    G = r.standard_normal((6, 9))
    got = O.ns_polynomial(G, 0, *O.NS_QUINTIC, eps=1e-7)
    np.testing.assert_allclose(got, G / (np.linalg.norm(G) + 1e-7), atol=1e-15)


def test_cubic_ns_converges_to_svd_msign():
    r = np.random.default_rng(6)
    s, l = 8, 20
    U, _ = np.linalg.qr(r.standard_normal((s, s)))
    V, _ = np.linalg.qr(r.standard_normal((l, s)))
    sigma = np.linspace(1.0, 0.4, s)
    G = U @ np.diag(sigma) @ V.T
    got = O.ns_polynomial(G, 60, *O.NS_CUBIC, eps=0.0)
    np.testing.assert_allclose(got, O.msign_svd(G), atol=1e-10)
    np.testing.assert_allclose(O.msign_svd(G), U @ V.T, atol=1e-12)


def test_msign_svd_brute_force_2x2_and_rank_deficient():
    G = np.array([[3.0, 0.0], [0.0, -0.5]])
    np.testing.assert_allclose(O.msign_svd(G), np.diag([1.0, -1.0]), atol=1e-15)
    # a rotation times a positive diagonal: msign is the rotation
    th = 0.3
    Rm = np.array([[math.cos(th), -math.sin(th)], [math.sin(th), math.cos(th)]])
    np.testing.assert_allclose(O.msign_svd(Rm @ np.diag([2.0, 0.1])), Rm, atol=1e-14)
    # rank one: msign(s u v^T) = u v^T
    u = np.array([3.0, 4.0]) / 5.0
    v = np.array([1.0, 0.0, 0.0])
    np.testing.assert_allclose(O.msign_svd(7 * np.outer(u, v)), np.outer(u, v), atol=1e-14)


def test_msign_svd_is_polar_factor():
    """For full column rank G, msign(G) = G (G^T G)^{-1/2} (computed with an
    eigendecomposition, a different library routine)."""
    r = np.random.default_rng(8)
    G = r.standard_normal((15, 6))
    w, Q = np.linalg.eigh(G.T @ G)
    polar = G @ (Q @ np.diag(w ** -0.5) @ Q.T)
    np.testing.assert_allclose(O.msign_svd(G), polar, atol=1e-12)


# ---------------------------------------------------------------------------
# The update rules of Algorithm 1
# ---------------------------------------------------------------------------

def test_dispatch_rule():
    assert O.is_muon_step(0, 1) and O.is_muon_step(5, 1)
    assert [O.is_muon_step(t, 3) for t in range(7)] == [True, False, False, True, False, False, True]
    assert not any(O.is_muon_step(t, 0) for t in range(10))   # P = infinity
    with pytest.raises(ValueError):
        O.is_muon_step(-1, 2)


def test_direction_uses_pre_update_buffer():
    """beta1=0.9, beta2=0.5, M_{t-1}=1, G=-2: the pre-update direction is
    0.9 - 0.2 = +0.7; the post-update one would be 0.45 - 1.1 < 0."""
    cfg = O.Config(beta1=0.9, beta2=0.5, eta_lion=1.0, weight_decay=0.0, period=0)
    W1, M1 = O.lionmuon_param_step(np.zeros(1), np.array([-2.0]), np.array([1.0]), 1, cfg)
    assert W1[0] == -1.0
    assert M1[0] == 0.5 * 1.0 + 0.5 * -2.0


def test_lion_step_magnitude_invariant():
    r = np.random.default_rng(9)
    W = r.standard_normal(1000)
    G = r.standard_normal(1000)
    M = r.standard_normal(1000)
    G[:50] = 0.0
    M[:50] = 0.0               # forced ties: G_hat exactly 0
    cfg = O.Config(eta_lion=0.01, weight_decay=0.3, period=0)
    W1, _ = O.lionmuon_param_step(W, G, M, 3, cfg)
    step = W1 - (1 - cfg.eta_lion * cfg.weight_decay) * W
    np.testing.assert_allclose(np.abs(step[50:]), cfg.eta_lion, rtol=1e-12)
    np.testing.assert_allclose(step[:50], 0.0, atol=1e-15)
    Ghat = cfg.beta1 * M + (1 - cfg.beta1) * G
    assert np.all(np.sign(step[50:]) == -np.sign(Ghat[50:]))


def test_momentum_closed_form_constant_gradient():
    """Constant G from M_{-1} = 0: M_t = (1 - beta2^(t+1)) G."""
    cfg = O.Config(beta1=0.8, beta2=0.95, period=0)
    G = np.array([1.5, -2.0, 0.25])
    M = np.zeros(3)
    W = np.zeros(3)
    for t in range(12):
        W, M = O.lionmuon_param_step(W, G, M, t, cfg)
        np.testing.assert_allclose(M, (1 - cfg.beta2 ** (t + 1)) * G, rtol=1e-14)


def test_muon_step_closed_form_on_known_svd():
    """One Muon step on G_hat with known SVD: the update direction is
    0.2 sqrt(max(m,n)) U phi^K(sigma) V^T, decay not scaled."""
    s, l = 16, 64
    sigma = np.linspace(2.0, 0.5, s)
    G, U, V = known_svd_matrix(s, l, sigma, seed=11, tall=True)   # tall 64 x 16
    cfg = O.Config(beta1=0.9, eta_muon=0.01, weight_decay=0.2, period=1)
    W = np.random.default_rng(1).standard_normal(G.shape)
    W1, _ = O.lionmuon_param_step(W, G, np.zeros_like(G), 0, cfg)
    # G_hat = (1 - beta1) G: same singular vectors, scaled singular values
    ghat_sigma = (1 - cfg.beta1) * sigma
    phi = O.ns_scalar_map(ghat_sigma / (np.linalg.norm(ghat_sigma) + cfg.ns_eps), 5, *O.NS_QUINTIC)
    dirn = (U @ np.diag(phi) @ V.T).T
    want = W - 0.01 * (0.2 * math.sqrt(64) * dirn + 0.2 * W)
    np.testing.assert_allclose(W1, want, atol=1e-12)


def test_vectors_take_lion_step_on_muon_steps():
    cfg = O.Config(eta_lion=0.5, eta_muon=9.0, weight_decay=0.0, period=1)
    W1, _ = O.lionmuon_param_step(np.zeros(4), np.array([1.0, -1.0, 0.0, 2.0]), np.zeros(4), 0, cfg)
    np.testing.assert_array_equal(W1, [-0.5, 0.5, 0.0, -0.5])


def _run(params, grads_per_step, cfg, steps):
    P = [p.copy() for p in params]
    M = [np.zeros_like(p) for p in params]
    for t in range(steps):
        P, M = O.lionmuon_step(P, grads_per_step[t], M, t, cfg)
    return P, M


def _problem(seed=0, steps=6):
    r = np.random.default_rng(seed)
    shapes = [(8, 12), (20, 6), (5,)]
    params = [r.standard_normal(s) for s in shapes]
    grads = [[r.standard_normal(s) for s in shapes] for _ in range(steps)]
    return params, grads


def test_reduction_P_infinity_beta_equal_is_signum():
    """Table 1: beta1 = beta2 with P = infinity is Signum:
    W <- W - eta (sign(M_t) + lambda W) with M_t the EMA of the gradients."""
    params, grads = _problem(1)
    beta = 0.9
    cfg = O.Config(beta1=beta, beta2=beta, eta_lion=0.01, weight_decay=0.1, period=0)
    got, _ = _run(params, grads, cfg, 6)
    W = [p.copy() for p in params]
    M = [np.zeros_like(p) for p in params]
    for t in range(6):
        for i in range(len(W)):
            M[i] = beta * M[i] + (1 - beta) * grads[t][i]
            W[i] = W[i] - 0.01 * (np.sign(M[i]) + 0.1 * W[i])
    for g, w in zip(got, W):
        np.testing.assert_allclose(g, w, atol=1e-14)


def test_reduction_P_infinity_is_lion():
    """Table 1: P = infinity with beta1 != beta2 is Lion (dual EMA); no matrix
    ever takes the Muon step."""
    params, grads = _problem(2)
    cfg = O.Config(beta1=0.9, beta2=0.99, eta_lion=0.01, eta_muon=123.0, weight_decay=0.1, period=0)
    got, _ = _run(params, grads, cfg, 6)
    W = [p.copy() for p in params]
    M = [np.zeros_like(p) for p in params]
    for t in range(6):
        for i in range(len(W)):
            d = np.sign(0.9 * M[i] + 0.1 * grads[t][i])
            W[i] = W[i] - 0.01 * (d + 0.1 * W[i])
            M[i] = 0.99 * M[i] + 0.01 * grads[t][i]
    for g, w in zip(got, W):
        np.testing.assert_allclose(g, w, atol=1e-14)


def test_reduction_P1_beta_equal_is_muon():
    """Table 1: beta1 = beta2, P = 1 is Muon with EMA momentum (no Nesterov):
    every matrix takes W <- W - eta (s NS(M_t) + lambda W) with M_t the EMA."""
    params, grads = _problem(3)
    beta = 0.9
    cfg = O.Config(beta1=beta, beta2=beta, eta_muon=0.02, eta_lion=0.001, weight_decay=0.1, period=1)
    got, _ = _run(params, grads, cfg, 5)
    W = [p.copy() for p in params]
    M = [np.zeros_like(p) for p in params]
    for t in range(5):
        for i in range(len(W)):
            M[i] = beta * M[i] + (1 - beta) * grads[t][i]
            if W[i].ndim == 2:
                X = O.ns_polynomial(M[i], 5, *O.NS_QUINTIC, 1e-7)
                W[i] = W[i] - 0.02 * (0.2 * math.sqrt(max(W[i].shape)) * X + 0.1 * W[i])
            else:
                W[i] = W[i] - 0.001 * (np.sign(M[i]) + 0.1 * W[i])
    for g, w in zip(got, W):
        np.testing.assert_allclose(g, w, atol=1e-13)


def test_period_alternation_pattern():
    """With P = 3, steps 0, 3 are Muon and 1, 2, 4 Lion: a matrix's Lion steps
    move every entry by exactly eta_L (lambda = 0), its Muon steps do not."""
    params, grads = _problem(4)
    cfg = O.Config(eta_lion=1e-3, eta_muon=1e-2, weight_decay=0.0, period=3)
    P = [p.copy() for p in params]
    M = [np.zeros_like(p) for p in params]
    for t in range(5):
        P1, M = O.lionmuon_step(P, grads[t], M, t, cfg)
        d = np.abs(P1[0] - P[0])
        if t % 3 == 0:
            assert not np.allclose(d, 1e-3)
        else:
            np.testing.assert_allclose(d, 1e-3, rtol=1e-9)
        P = P1


def test_heavy_ball_equals_ema_signmuon():
    """Appendix F: heavy-ball M = mu M + G and EMA M' = beta M' + (1-beta) G
    with mu = beta satisfy M' = (1-beta) M, so the sign and msign directions
    agree and the iterates coincide (up to the eps of the NS normalisation)."""
    params, grads = _problem(5, steps=6)
    beta = 0.9
    cfg = O.Config(beta1=beta, beta2=beta, eta_muon=0.02, eta_lion=0.01, weight_decay=0.1, period=2)
    got, _ = _run(params, grads, cfg, 6)
    W = [p.copy() for p in params]
    Mhb = [np.zeros_like(p) for p in params]
    for t in range(6):
        for i in range(len(W)):
            Mhb[i] = beta * Mhb[i] + grads[t][i]
            if W[i].ndim == 2 and t % 2 == 0:
                X = O.ns_polynomial(Mhb[i], 5, *O.NS_QUINTIC, 0.0)
                W[i] = W[i] - 0.02 * (0.2 * math.sqrt(max(W[i].shape)) * X + 0.1 * W[i])
            else:
                W[i] = W[i] - 0.01 * (np.sign(Mhb[i]) + 0.1 * W[i])
    for g, w in zip(got, W):
        np.testing.assert_allclose(g, w, atol=1e-7)


def test_decay_frank_wolfe_rewrite():
    """Appendix B: with U the step direction (sign or msign of G_hat) and
    LMO_{B(1/lambda)}(G_hat) = -U / lambda,
    W - eta (U + lambda W) = (1 - eta lambda) W + eta lambda LMO_{B(1/lambda)}(G_hat)."""
    r = np.random.default_rng(12)
    W = r.standard_normal((7, 9))
    Ghat = r.standard_normal((7, 9))
    eta, lam = 0.03, 0.2
    for U in (np.sign(Ghat), O.msign_svd(Ghat)):
        a = W - eta * (U + lam * W)
        b = (1 - eta * lam) * W + eta * lam * (-U / lam)
        np.testing.assert_allclose(a, b, atol=1e-15)
    cfg = O.Config(eta_lion=eta, weight_decay=lam, period=0)
    W1, _ = O.lionmuon_param_step(W, Ghat, np.zeros_like(W), 1, cfg)
    # LMO of the l_inf ball of radius 1/lambda is -sign(G_hat)/lambda
    lmo = -np.sign((1 - cfg.beta1) * Ghat) / lam
    np.testing.assert_allclose(W1, (1 - eta * lam) * W + eta * lam * lmo, atol=1e-15)


def test_state_is_one_buffer_per_parameter():
    """Section 3, Implementation notes: the only persisted state is one buffer
    of |W| entries per parameter."""
    params, grads = _problem(6)
    cfg = O.Config(period=2)
    M = [np.zeros_like(p) for p in params]
    P, M = O.lionmuon_step(params, grads[0], M, 0, cfg)
    assert [m.shape for m in M] == [p.shape for p in params]
    assert sum(m.size for m in M) == sum(p.size for p in params)


# ---------------------------------------------------------------------------
# Same-order fp32 Lion step
# ---------------------------------------------------------------------------

def test_lion_f32_matches_fp64_within_rounding():
    r = np.random.default_rng(13)
    n = 50000
    w = r.standard_normal(n).astype(np.float32)
    g = r.standard_normal(n).astype(np.float32)
    m = r.standard_normal(n).astype(np.float32)
    beta1, beta2, eta, lam = 0.9, 0.99, 0.02, 0.1
    w32, m32 = O.lion_step_f32(w, g, m, beta1, beta2, eta, lam, w_dtype="f32")
    cfg = O.Config(beta1=beta1, beta2=beta2, eta_lion=eta, weight_decay=lam, period=0)
    w64, m64 = O.lionmuon_param_step(w.astype(np.float64), g.astype(np.float64), m.astype(np.float64), 1, cfg)
    ghat = 0.9 * m.astype(np.float64) + 0.1 * g.astype(np.float64)
    safe = np.abs(ghat) > 1e-5        # away from sign ties
    # error bound: a few float32 ulps of the largest operand of the last
    # subtraction (w and eta*(u + lambda*w)), plus the rounding of the constants
    mag = np.maximum(np.abs(w).astype(np.float64), eta * (1 + lam * np.abs(w)))
    ulp = np.spacing(mag.astype(np.float32)).astype(np.float64)
    assert np.all(np.abs(w32[safe] - w64[safe]) <= 3 * ulp[safe])
    mmag = np.maximum(np.abs(m), np.abs(g)).astype(np.float64)
    mulp = np.spacing(mmag.astype(np.float32)).astype(np.float64)
    assert np.all(np.abs(m32 - m64) <= 3 * mulp)


def test_lion_f32_order_is_separately_rounded():
    """Each float32 product and sum is rounded once: recompute the same
    sequence with float64 arithmetic (exact for these products/sums of
    float32 values) and explicit rounding to float32 after every operation."""
    r = np.random.default_rng(14)
    n = 20000
    w = O.bf16_round(r.standard_normal(n).astype(np.float32) * np.float32(0.05))
    g = O.bf16_round(r.standard_normal(n).astype(np.float32) * np.float32(1e-3))
    m = (r.standard_normal(n) * 1e-3).astype(np.float32)
    beta1, beta2, eta, lam = 0.9, 0.99, 2e-5, 0.1
    w32, m32 = O.lion_step_f32(w, g, m, beta1, beta2, eta, lam, w_dtype="bf16")
    f = np.float32
    b1, c1, b2, c2, eL, la = (np.float64(f(beta1)), np.float64(f(1 - beta1)), np.float64(f(beta2)),
                              np.float64(f(1 - beta2)), np.float64(f(eta)), np.float64(f(lam)))
    R = lambda x: np.asarray(x, dtype=np.float64).astype(np.float32).astype(np.float64)
    W, G, M = w.astype(np.float64), g.astype(np.float64), m.astype(np.float64)
    gh = R(R(b1 * M) + R(c1 * G))
    u = np.sign(gh)
    wn = R(W - R(eL * R(u + R(la * W))))
    mn = R(R(b2 * M) + R(c2 * G))
    np.testing.assert_array_equal(w32, O.bf16_round(wn.astype(np.float32)))
    np.testing.assert_array_equal(m32, mn.astype(np.float32))


def test_ns_flop_count():
    assert O.ns_flops(128, 256, 1, symmetric=False) == 4 * 128 * 128 * 256 + 2 * 128 ** 3
    assert O.ns_flops(256, 128, 5, symmetric=True) == 5 * (3 * 128 * 128 * 256 + 128 ** 3)


def test_storage_mode_sign_decision_matches_f32_lion():
    """Storage-modelled mode decides Lion signs on the float32 G_hat: its
    weights then agree with the same-order float32 Lion step to within the
    final bf16 rounding (one bf16 ulp), including near-tie entries."""
    r = np.random.default_rng(21)
    n = 20000
    w = O.bf16_round(r.standard_normal(n).astype(np.float32) * np.float32(0.02))
    g = O.bf16_round(r.standard_normal(n).astype(np.float32) * np.float32(1e-3))
    m = (r.standard_normal(n) * 1e-3).astype(np.float32)
    # near ties: G_hat almost exactly 0 in float64 but not in float32
    g[:100] = O.bf16_round(np.float32(-9.0) * m[:100])
    cfg = O.Config(beta1=0.9, beta2=0.99, eta_lion=1e-2, weight_decay=0.1, period=0)
    P, M = O.lionmuon_step([w.astype(np.float64)], [g.astype(np.float64)], [m.astype(np.float64)], 1,
                           cfg, param_dtypes=["bf16"])
    w32, m32 = O.lion_step_f32(w, g, m, 0.9, 0.99, 1e-2, 0.1, w_dtype="bf16")
    ulp = np.spacing(np.abs(w32)) * 65536.0
    assert np.all(np.abs(P[0] - w32) <= ulp)
    # fp64 EMA rounded once vs the float32 same-order EMA: within two ulps of
    # the larger addend
    mag = np.maximum(np.abs(m), np.abs(g)).astype(np.float32)
    assert np.all(np.abs(M[0] - m32.astype(np.float64)) <= 2 * np.spacing(mag).astype(np.float64))


def test_quintic_iterates_stay_within_its_range():
    """The published quintic phi(x) = a x + b x^3 + c x^5 maps [0, 1] into
    [0, 1.2024] (its maximum on [0, 1], at x^2 = (3|b| - sqrt(9 b^2 - 20 a c))
    / (10 c), is 1.20237) and keeps [0, 1.2024] there, so every singular
    value of an NS output lies in [0, 1.2024]: the validity bound the GPU
    tests apply to rank-deficient inputs."""
    a, b, c = O.NS_QUINTIC
    x2 = (-3 * b - np.sqrt(9 * b * b - 20 * a * c)) / (10 * c)
    xm = np.sqrt(x2)
    peak = a * xm + b * xm ** 3 + c * xm ** 5
    assert 1.2023 < peak < 1.2025
    x = np.linspace(0.0, 1.0, 200001)
    for _ in range(5):
        x = a * x + b * x ** 3 + c * x ** 5
        assert x.min() >= 0.0 and x.max() <= peak + 1e-12
