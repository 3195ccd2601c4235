"""Pins for the oracle's AdamW fallback for 1-D parameters (Section 3: biases
and norm gains take AdamW with a small fixed learning rate; Table 5: 1e-3 and
AdamW betas (0.8, 0.999)): against torch.optim.AdamW in float64 (a library
routine), closed forms for a constant and a zero gradient, the float32
same-order variant within its rounding, and the LionMuon step routing
vectors to AdamW and matrices to Algorithm 1."""

import numpy as np
import pytest

import oracle as O

LR, B1, B2, EPS, WD = 1e-3, 0.8, 0.999, 1e-8, 0.1


def _torch_adamw(W0, grads, lr, betas, eps, wd):
    import torch
    p = torch.nn.Parameter(torch.tensor(W0, dtype=torch.float64))
    opt = torch.optim.AdamW([p], lr=lr, betas=betas, eps=eps, weight_decay=wd)
    out = []
    for g in grads:
        p.grad = torch.tensor(g, dtype=torch.float64)
        opt.step()
        out.append(p.detach().numpy().copy())
    st = opt.state[p]
    return out, st["exp_avg"].numpy(), st["exp_avg_sq"].numpy()


@pytest.mark.parametrize("wd", [0.0, WD])
def test_adamw_matches_torch_adamw_float64(wd):
    r = np.random.default_rng(0)
    W = r.normal(0, 0.02, size=257)
    grads = [r.standard_t(3, size=257) * 1e-3 for _ in range(7)]
    want, m_ref, v_ref = _torch_adamw(W, grads, LR, (B1, B2), EPS, wd)
    m = np.zeros_like(W)
    v = np.zeros_like(W)
    for k, g in enumerate(grads):
        W, m, v = O.adamw_update(W, g, m, v, k + 1, LR, B1, B2, EPS, wd)
        np.testing.assert_allclose(W, want[k], rtol=1e-13, atol=1e-17)
    # torch forms the moments with lerp / addcmul: same values to fp64 rounding
    np.testing.assert_allclose(m, m_ref, rtol=1e-12)
    np.testing.assert_allclose(v, v_ref, rtol=1e-12)


def test_adamw_constant_gradient_closed_form():
    """With a constant gradient g the bias-corrected moments are exactly g and
    g^2 at every step, so without decay W_t = W_0 - t lr g / (|g| + eps)."""
    W0 = np.array([0.5, -0.25, 0.125, 0.0])
    g = np.array([3e-3, -1e-4, 0.0, 2.0])
    W, m, v = W0.copy(), np.zeros(4), np.zeros(4)
    for t in range(1, 9):
        W, m, v = O.adamw_update(W, g, m, v, t, LR, B1, B2, EPS, 0.0)
        np.testing.assert_allclose(W, W0 - t * LR * g / (np.abs(g) + EPS), rtol=1e-12, atol=1e-18)


def test_adamw_zero_gradient_is_pure_decay():
    W0 = np.linspace(-1, 1, 9)
    W, m, v = O.adamw_update(W0, np.zeros(9), np.zeros(9), np.zeros(9), 1, LR, B1, B2, EPS, WD)
    np.testing.assert_array_equal(W, W0 - LR * WD * W0)
    assert not m.any() and not v.any()


def test_adamw_first_step_is_sign_like():
    """Step 1 from zero moments: m_hat = g, v_hat = g^2, so the update is
    lr g / (|g| + eps) (plus decay)."""
    g = np.array([1e-2, -1e-6, 5.0])
    W0 = np.array([0.1, 0.2, -0.3])
    W, _, _ = O.adamw_update(W0, g, np.zeros(3), np.zeros(3), 1, LR, B1, B2, EPS, WD)
    np.testing.assert_allclose(W, W0 - LR * WD * W0 - LR * g / (np.abs(g) + EPS), rtol=1e-14)


def test_adamw_f32_matches_fp64_within_rounding():
    r = np.random.default_rng(1)
    n = 4096
    w32 = r.normal(0, 0.02, size=n).astype(np.float32)
    m32 = np.zeros(n, np.float32)
    v32 = np.zeros(n, np.float32)
    W, m, v = w32.astype(np.float64), np.zeros(n), np.zeros(n)
    for t in range(1, 6):
        g = (r.standard_t(3, size=n) * 1e-3).astype(np.float32)
        w32, m32, v32 = O.adamw_step_f32(w32, g, m32, v32, t, LR, B1, B2, EPS, WD, w_dtype="f32")
        W, m, v = O.adamw_update(W, g.astype(np.float64), m, v, t, LR, B1, B2, EPS, WD)
    # each step moves w by at most about lr (|m_hat| / sqrt(v_hat) <= 1 / sqrt(1 - b2) bounds it loosely);
    # float32 rounding of a few operations per step stays far below 1e-6 relative to |w| + lr
    assert np.max(np.abs(w32 - W) / (np.abs(W) + LR)) < 1e-5
    # m = b1 m + c1 g can cancel: its float32 error is relative to |c1 g| ~ 2e-4, not to |m|
    np.testing.assert_allclose(m32, m, rtol=1e-5, atol=1e-9)
    np.testing.assert_allclose(v32, v, rtol=1e-5, atol=1e-15)


def test_lionmuon_step_routes_vectors_to_adamw():
    cfg = O.Config(vector_rule="adamw", period=2)
    r = np.random.default_rng(3)
    shapes = [(8, 12), (12,)]
    P = [r.normal(size=s) for s in shapes]
    M = [np.zeros(s) for s in shapes]
    V = [np.zeros(s) for s in shapes]
    ref_lion = O.Config(period=2)
    Pl, Ml = [p.copy() for p in P], [m.copy() for m in M]
    vec_W, vec_m, vec_v = P[1].copy(), np.zeros(12), np.zeros(12)
    for t in range(4):
        G = [r.normal(size=s) for s in shapes]
        P, M, V = O.lionmuon_step(P, G, M, t, cfg, seconds=V)
        Pl, Ml = O.lionmuon_step(Pl, G, Ml, t, ref_lion)
        vec_W, vec_m, vec_v = O.adamw_update(vec_W, G[1], vec_m, vec_v, t + 1, cfg.adamw_lr, cfg.adamw_beta1,
                                             cfg.adamw_beta2, cfg.adamw_eps, cfg.adamw_weight_decay)
        np.testing.assert_array_equal(P[0], Pl[0])     # the matrix follows Algorithm 1 unchanged
        np.testing.assert_array_equal(P[1], vec_W)
        np.testing.assert_array_equal(M[1], vec_m)
        np.testing.assert_array_equal(V[1], vec_v)
    with pytest.raises(ValueError):
        O.lionmuon_step(P, G, M, 0, cfg)
