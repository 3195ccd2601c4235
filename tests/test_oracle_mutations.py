"""Plant plausible mistakes in the oracle (on the CPU) and check that the pins
in test_oracle_pins.py catch each of them: the pins are only worth something
if a dropped term, a wrong sign, a transposed operand, the post-update buffer
or a wrong branch makes at least one of them fail."""

import math

import numpy as np
import pytest

import oracle
import oracle.lionmuon_oracle as OM
from tests import test_oracle_pins as pins
from tests import test_oracle_pins_msign_variants as vpins
from tests import test_oracle_pins_adamw as apins
from tests import test_oracle_pins_srank as spins

# every pin, with representative arguments for the parametrised ones
PIN_CALLS = [
    (pins.test_ns_closed_form_on_known_svd, (16, 64, False, oracle.NS_QUINTIC, 5)),
    (pins.test_ns_closed_form_on_known_svd, (16, 64, True, oracle.NS_CUBIC, 7)),
    (pins.test_ns_closed_form_on_known_svd, (16, 16, False, (2.0, -1.3, 0.4), 3)),
    (pins.test_ns_rank_one, ()),
    (pins.test_ns_transpose_identity, ()),
    (pins.test_ns_orthogonal_equivariance, ()),
    (pins.test_ns_scale_invariance, ()),
    (pins.test_ns_zero_steps_is_normalisation, ()),
    (pins.test_cubic_ns_converges_to_svd_msign, ()),
    (pins.test_msign_svd_brute_force_2x2_and_rank_deficient, ()),
    (pins.test_msign_svd_is_polar_factor, ()),
    (pins.test_dispatch_rule, ()),
    (pins.test_direction_uses_pre_update_buffer, ()),
    (pins.test_lion_step_magnitude_invariant, ()),
    (pins.test_momentum_closed_form_constant_gradient, ()),
    (pins.test_muon_step_closed_form_on_known_svd, ()),
    (pins.test_vectors_take_lion_step_on_muon_steps, ()),
    (pins.test_reduction_P_infinity_beta_equal_is_signum, ()),
    (pins.test_reduction_P_infinity_is_lion, ()),
    (pins.test_reduction_P1_beta_equal_is_muon, ()),
    (pins.test_period_alternation_pattern, ()),
    (pins.test_heavy_ball_equals_ema_signmuon, ()),
    (pins.test_decay_frank_wolfe_rewrite, ()),
    (pins.test_bf16_round_known_values, ()),
    (pins.test_lion_f32_matches_fp64_within_rounding, ()),
    (vpins.test_minimax_cubic_matches_closed_form, (0.2, 1.0)),
    (vpins.test_minimax_quintic_equioscillates, (0.1, 1.0)),
    (vpins.test_ns_schedule_closed_form_on_known_svd, ()),
    (vpins.test_ns_schedule_constant_table_is_classical_ns, ()),
    (vpins.test_minimax_schedule_maps_interval_forward, (5, 5)),
    (vpins.test_bf16_storage_ns_on_hadamard_follows_hand_rounded_scalars, ()),
    (apins.test_adamw_matches_torch_adamw_float64, (0.1,)),
    (apins.test_adamw_constant_gradient_closed_form, ()),
    (apins.test_adamw_zero_gradient_is_pure_decay, ()),
    (apins.test_adamw_first_step_is_sign_like, ()),
    (spins.test_splitmix64_published_outputs, ()),
    (spins.test_power_estimate_closed_form_on_known_svd, (3,)),
    (spins.test_exact_stable_ranks, ()),
    (spins.test_threshold_and_zero_buffer, ()),
    (spins.test_step_routes_matrices_by_stable_rank, ()),
    (spins.test_decision_uses_the_buffer_before_the_update, ()),
]


def _ns_factory(variant):
    def ns(G, steps, a, b, c, eps=1e-7):
        X = np.array(G, dtype=np.float64)
        tr = X.shape[0] > X.shape[1]
        if tr:
            X = X.T.copy()
        if variant != "no_normalisation":
            X = X / (np.linalg.norm(X) + eps)
        n = steps + 1 if variant == "extra_iteration" else steps
        for _ in range(n):
            A = X.T @ X if variant == "transposed_gram" and X.shape[0] == X.shape[1] else X @ X.T
            if variant == "dropped_c":
                B = b * A
            elif variant == "wrong_sign_c":
                B = b * A - c * (A @ A)
            else:
                B = b * A + c * (A @ A)
            X = a * X + (X @ B if variant == "right_multiply" else B @ X)
        return X.T.copy() if tr else X
    return ns


def _patch(monkeypatch, name, fn):
    monkeypatch.setattr(OM, name, fn)
    monkeypatch.setattr(oracle, name, fn)


def _mutations():
    muts = {}
    for v in ("no_normalisation", "extra_iteration", "transposed_gram", "dropped_c", "wrong_sign_c",
              "right_multiply"):
        muts["ns_" + v] = [("ns_polynomial", _ns_factory(v))]
    muts["post_update_buffer"] = [("lionmuon_param_step", _post_update_step)]
    muts["lion_missing_decay"] = [("lion_update", lambda W, Gh, eta, lam: W - eta * OM.sign(Gh))]
    muts["lion_wrong_sign"] = [("lion_update", lambda W, Gh, eta, lam: W + eta * (OM.sign(Gh) - lam * W))]
    muts["momentum_uses_beta1"] = [("momentum_update", lambda M, G, b2: 0.9 * M + 0.1 * G)]
    muts["dispatch_off_by_one"] = [("is_muon_step", lambda t, P: P != 0 and t % P == 1 % max(P, 1))]
    muts["scale_uses_min"] = [("muon_update", _muon_min_scale)]
    muts["bf16_truncates"] = [("bf16_round", _bf16_truncate)]
    muts["schedule_reversed"] = [("ns_polynomial_schedule", _schedule_factory(reverse=True)),
                                 ("ns_scalar_map_schedule", _scalar_schedule_factory(reverse=True))]
    muts["schedule_first_only"] = [("ns_polynomial_schedule", _schedule_factory(first_only=True)),
                                   ("ns_scalar_map_schedule", _scalar_schedule_factory(first_only=True))]
    muts["minimax_least_squares"] = [("minimax_odd_polynomial", _least_squares_poly)]
    muts["minimax_no_interval_update"] = [("minimax_schedule", _schedule_fixed_interval)]
    muts["storage_ns_unrounded_B"] = [("ns_polynomial_schedule_storage", _storage_ns_unrounded_B)]
    muts["adamw_no_bias_correction"] = [("adamw_update", _adamw_variant("no_bias"))]
    muts["adamw_coupled_decay"] = [("adamw_update", _adamw_variant("coupled"))]
    muts["adamw_eps_inside_sqrt"] = [("adamw_update", _adamw_variant("eps_in_sqrt"))]
    muts["adamw_beta_swap"] = [("adamw_update", _adamw_variant("swap"))]
    muts["srank_threshold_max_dim"] = [("srank_takes_muon", _srank_max_dim)]
    muts["srank_estimate_from_w"] = [("stable_rank_estimate", _srank_estimate_w)]
    muts["srank_post_update_buffer"] = [("lionmuon_step", _srank_post_update_step)]
    muts["splitmix_shift_29"] = [("splitmix64", _splitmix_shift29)]
    return muts


def _order(coeffs, reverse, first_only):
    coeffs = list(coeffs)
    if first_only:
        return [coeffs[0]] * len(coeffs)
    return coeffs[::-1] if reverse else coeffs


def _schedule_factory(reverse=False, first_only=False):
    def f(G, coeffs, eps=1e-7):
        X = np.array(G, dtype=np.float64)
        tr = X.shape[0] > X.shape[1]
        if tr:
            X = X.T.copy()
        X = X / (np.linalg.norm(X) + eps)
        for a, b, c in _order(coeffs, reverse, first_only):
            A = X @ X.T
            X = a * X + (b * A + c * (A @ A)) @ X
        return X.T.copy() if tr else X
    return f


def _scalar_schedule_factory(reverse=False, first_only=False):
    def f(x, coeffs):
        x = np.array(x, dtype=np.float64)
        for a, b, c in _order(coeffs, reverse, first_only):
            x = a * x + b * x ** 3 + c * x ** 5
        return x
    return f


def _least_squares_poly(lo, hi, degree, grid=20001):
    x = np.linspace(lo, hi, grid)
    d = (degree + 1) // 2
    V = np.stack([x ** (2 * j + 1) for j in range(d)], axis=1)
    q = np.linalg.lstsq(V, np.ones(grid), rcond=None)[0]
    return q, float(np.abs(1 - V @ q).max())


def _schedule_fixed_interval(steps, lo, degree=5, safety=1.0):
    q, _ = OM.minimax_odd_polynomial(lo, 1.0, degree)
    tr = (float(q[0]), float(q[1]), float(q[2]) if len(q) > 2 else 0.0)
    return (tr,) * steps


def _post_update_step(W, G, M_prev, t, cfg, sign_in_f32=False, take_muon=None):
    W = np.asarray(W, dtype=np.float64)
    G = np.asarray(G, dtype=np.float64)
    M_new = OM.momentum_update(np.asarray(M_prev, dtype=np.float64), G, cfg.beta2)
    G_hat = OM.interpolated_direction(M_new, G, cfg.beta1)
    muon = OM.is_muon_step(t, cfg.period) if take_muon is None else take_muon
    if OM.is_matrix(W.shape) and muon:
        return OM.muon_update(W, G_hat, cfg), M_new
    return OM.lion_update(W, G_hat, cfg.eta_lion, cfg.weight_decay), M_new


def _muon_min_scale(W, G_hat, cfg):
    O = OM.ns_polynomial(G_hat, cfg.ns_steps, cfg.ns_a, cfg.ns_b, cfg.ns_c, cfg.ns_eps)
    return W - cfg.eta_muon * (cfg.shape_scale * math.sqrt(min(W.shape)) * O + cfg.weight_decay * W)


def _bf16_truncate(x):
    f = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    u = f.view(np.uint32) & np.uint32(0xFFFF0000)
    return u.view(np.float32).copy()


def _adamw_variant(kind):
    def f(W, G, m_prev, v_prev, step, lr, beta1, beta2, eps, weight_decay):
        W = np.asarray(W, dtype=np.float64)
        G = np.asarray(G, dtype=np.float64)
        if kind == "swap":
            beta1, beta2 = beta2, beta1
        g_eff = G + weight_decay * W if kind == "coupled" else G
        m = beta1 * m_prev + (1 - beta1) * g_eff
        v = beta2 * v_prev + (1 - beta2) * g_eff * g_eff
        bc1, bc2 = (1.0, 1.0) if kind == "no_bias" else (1 - beta1 ** step, 1 - beta2 ** step)
        den = np.sqrt(v / bc2 + eps) if kind == "eps_in_sqrt" else np.sqrt(v / bc2) + eps
        decay = 0.0 if kind == "coupled" else lr * weight_decay * W
        return W - decay - lr * (m / bc1) / den, m, v
    return f


def _srank_max_dim(M_prev, cfg):
    m, n = np.shape(M_prev)
    fro2, sig2 = OM.stable_rank_estimate(M_prev, cfg.srank_iters, OM.power_start_vector(n, cfg.srank_seed))
    return fro2 == 0.0 or fro2 <= cfg.srank_alpha * max(m, n) * sig2


def _srank_estimate_w(M, iters, v0):
    M = np.asarray(M, dtype=np.float64)
    v = v0 / np.linalg.norm(v0)
    sig2 = 0.0
    for _ in range(iters):
        w = M.T @ (M @ v)
        sig2 = float(np.linalg.norm(w))
        v = w / np.linalg.norm(w)
    return float(np.sum(M * M)), sig2


def _srank_post_update_step(params, grads, moms, t, cfg, param_dtypes=None, seconds=None):
    new_p, new_m = [], []
    for W, G, M in zip(params, grads, moms):
        M1 = OM.momentum_update(np.asarray(M, dtype=np.float64), np.asarray(G, dtype=np.float64), cfg.beta2)
        take = OM.srank_takes_muon(M1, cfg) if OM.is_matrix(np.shape(W)) else None
        W1, M1 = OM.lionmuon_param_step(W, G, M, t, cfg, take_muon=take)
        new_p.append(W1)
        new_m.append(M1)
    return new_p, new_m


def _splitmix_shift29(seed, count):
    out, st, U = [], seed, (1 << 64) - 1
    for _ in range(count):
        st = (st + 0x9E3779B97F4A7C15) & U
        z = ((st ^ (st >> 29)) * 0xBF58476D1CE4E5B9) & U
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & U
        out.append(z ^ (z >> 31))
    return out


def _storage_ns_unrounded_B(G, coeffs, eps=1e-7, storage="bf16"):
    rd = lambda v: OM.bf16_round(v).astype(np.float64)
    G = np.array(G, dtype=np.float64)
    tr = G.shape[0] > G.shape[1]
    if tr:
        G = G.T.copy()
    inv = 1.0 / (np.linalg.norm(G) + eps)
    X = rd(G)
    for k, (a, b, c) in enumerate(coeffs):
        sa, sx = (inv * inv, inv) if k == 0 else (1.0, 1.0)
        A = rd(sa * (X @ X.T))
        B = b * A + c * (A @ A)
        X = rd(sx * (a * X + B @ X))
    return X.T.copy() if tr else X


@pytest.mark.filterwarnings("ignore::RuntimeWarning")
@pytest.mark.parametrize("name", sorted(_mutations()))
def test_each_planted_mistake_is_caught(name, monkeypatch):
    for fn_name, fn in _mutations()[name]:
        _patch(monkeypatch, fn_name, fn)
    caught = []
    for pin, args in PIN_CALLS:
        try:
            pin(*args)
        except (AssertionError, ValueError):
            caught.append(pin.__name__)
    assert caught, f"no pin detects the mutation {name}"

