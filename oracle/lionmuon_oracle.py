"""CPU oracle for the LionMuon optimizer step (arXiv 2605.19811).

TEST INFRASTRUCTURE ONLY.  This module is the slow, plain restatement of the
paper's update that the CUDA library is checked against.  Only the test suite,
``__graft_entry__.smoke()`` and the ``cpu_baseline`` / ``--impl reference`` legs
of ``bench.py`` may import it.  It shares no code with the CUDA path and never
imports the product package.

Everything is numpy in float64 unless a function says otherwise.  Each function
names the passage of the paper it restates:

* Algorithm 1 ("LionMuon and SignMuon for a single 2D parameter"): the
  interpolated direction G_hat from the *pre-update* buffer M_{t-1}, the
  branch on ``t mod P``, the Muon step with NS_{K_NS}, the Lion sign step,
  decoupled weight decay on both branches, and the momentum update on every
  step.
* Section 2 (Related works, "Spectral methods" / "Approximating the matrix
  sign") and the Notations of Section 2.1: msign(X) = U V^T, computed by an
  odd-polynomial Newton-Schulz iteration.
* Table 5 (full experimental configuration): K_NS = 5 and the NS output
  scaling 0.2 * sqrt(max(m, n)).
* Section 3, Implementation notes: one persisted buffer per parameter.

Readings taken where the paper is silent:

* NS coefficients: the paper gives none; the default is the widely used
  quintic (a, b, c) = (3.4445, -4.7750, 2.0315), constant over iterations.
* The NS input is pre-normalised as X / (||X||_F + eps), eps = 1e-7.
* For a tall matrix (m > n) the iteration runs on X^T and the result is
  transposed back; p(X X^T) X = X p(X^T X) makes this the same function.
* The 0.2*sqrt(max(m,n)) factor multiplies the NS output inside the eta_M
  bracket; the decay term is not scaled.
* sign(0) = 0 and sign(NaN) = NaN.
* 1-D parameters (vectors) take the Lion step on every step by default; the
  AdamW fallback of Section 3 is the ``vector_rule="adamw"`` option, with
  Table 5's 1-D learning rate 1e-3 and AdamW betas (0.8, 0.999), weight decay
  0.1 (Table 5's), eps 1e-8, bias correction with the update count t + 1.
* P = infinity is encoded as ``period = 0``.
* The adaptive schedule of Appendix G decides on M_{t-1}, the buffer at hand
  when the step starts; its power iteration starts from a SplitMix64 vector
  (seed a parameter), makes ``srank_iters`` passes (5 by default: "a few"),
  and a zero buffer takes Muon.
* Iteration-dependent NS coefficients (the minimax / Chebyshev-type msign
  iterations of Section 2) keep the Frobenius normalisation, so the first
  interval of singular values is [l_0, 1] with l_0 a parameter; the minimax
  table is the per-interval best odd polynomial with the interval mapped
  forward, optionally divided by a safety factor.

Parity status: the fp64 update rules are pinned by closed forms and
invariants in tests/test_oracle_pins.py.  The end-to-end trajectory values are
pinned only through those invariants: the paper prints no worked example of
an update, so the exact trajectory of the paper's implementation (whose NS
coefficients it does not state) is "parity unpinned".
"""

from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Sequence, Tuple

import numpy as np

# Quintic Newton-Schulz coefficients used as the default reading (the paper
# cites the Muon iteration but prints no coefficients).
NS_QUINTIC = (3.4445, -4.7750, 2.0315)
# Classic cubic Newton-Schulz iteration X <- 1.5 X - 0.5 X X^T X, which
# converges to msign(X) for ||X||_2 < sqrt(3).
NS_CUBIC = (1.5, -0.5, 0.0)


@dataclasses.dataclass
class Config:
    """Hyper-parameters named in the Require line of Algorithm 1."""

    beta1: float = 0.9
    beta2: float = 0.99
    eta_muon: float = 3e-3
    eta_lion: float = 2e-5
    weight_decay: float = 0.1
    period: int = 2            # P >= 1; 0 encodes P = infinity (never Muon)
    ns_steps: int = 5          # K_NS (Table 5)
    ns_a: float = NS_QUINTIC[0]
    ns_b: float = NS_QUINTIC[1]
    ns_c: float = NS_QUINTIC[2]
    ns_eps: float = 1e-7
    shape_scale: float = 0.2   # NS scaling 0.2*sqrt(max(m,n)) (Table 5)
    # Optional per-iteration coefficients ((a_0, b_0, c_0), ...): when set they
    # replace (ns_a, ns_b, ns_c) and their count replaces ns_steps.
    ns_coeffs: Optional[Tuple[Tuple[float, float, float], ...]] = None
    # 1-D parameters: "lion" (the Lion step of Algorithm 1 every step) or
    # "adamw" (Section 3's fallback for biases and norm gains, with Table 5's
    # 1-D learning rate 1e-3 and AdamW betas (0.8, 0.999)).
    vector_rule: str = "lion"
    # Muon/Lion selection for matrices: "period" (Algorithm 1, t mod P) or
    # "stable_rank" (Appendix G): Muon where the stable rank of M_{t-1},
    # ||M||_F^2 / sigma_1_hat^2, is at most alpha * min(m, n).
    schedule: str = "period"
    srank_alpha: float = 0.01
    srank_iters: int = 5        # passes over M of the power iteration
    srank_seed: int = 0         # SplitMix64 seed of the start vector
    adamw_lr: float = 1e-3
    adamw_beta1: float = 0.8
    adamw_beta2: float = 0.999
    adamw_eps: float = 1e-8
    adamw_weight_decay: float = 0.1


# ---------------------------------------------------------------------------
# Scalar building blocks
# ---------------------------------------------------------------------------

def sign(x: np.ndarray) -> np.ndarray:
    """Element-wise sign, the l_inf LMO of Section 2.1 (up to the minus sign).

    sign(+-0) = 0, sign(NaN) = NaN (numpy's definition, written out so the
    choice is visible)."""
    x = np.asarray(x)
    out = np.where(x > 0, 1.0, np.where(x < 0, -1.0, 0.0)).astype(x.dtype)
    return np.where(np.isnan(x), x, out)


def is_muon_step(t: int, period: int) -> bool:
    """Branch condition of Algorithm 1: Muon iff ``t mod P == 0``.

    P = infinity (``period == 0``) never takes the Muon branch."""
    if t < 0:
        raise ValueError("t must be >= 0")
    if period < 0:
        raise ValueError("period must be >= 0 (0 encodes infinity)")
    return period != 0 and t % period == 0


def interpolated_direction(M_prev, G, beta1):
    """G_hat_t = beta1 * M_{t-1} + (1 - beta1) * G_t (Algorithm 1, uses the
    buffer *before* this step's momentum update)."""
    return beta1 * M_prev + (1.0 - beta1) * G


def momentum_update(M_prev, G, beta2):
    """M_t = beta2 * M_{t-1} + (1 - beta2) * G_t (Algorithm 1, every step)."""
    return beta2 * M_prev + (1.0 - beta2) * G


# ---------------------------------------------------------------------------
# Matrix sign
# ---------------------------------------------------------------------------

def ns_polynomial(G: np.ndarray, steps: int, a: float, b: float, c: float,
                  eps: float = 1e-7) -> np.ndarray:
    """NS_K(G): odd-polynomial Newton-Schulz approximation of msign(G).

    Section 2 ("Spectral methods", "Approximating the matrix sign") names the
    iteration; the polynomial form used is, per step,
        A = X X^T,  B = b A + c A A,  X <- a X + B X,
    which maps every singular value s of X to a s + b s^3 + c s^5.
    The input is first divided by (||G||_F + eps).  A tall input (m > n) is
    iterated in its transposed (wide) orientation and transposed back.
    """
    X = np.array(G, dtype=np.float64)
    if X.ndim != 2:
        raise ValueError("NS needs a 2-D matrix")
    transposed = X.shape[0] > X.shape[1]
    if transposed:
        X = X.T.copy()
    X = X / (np.linalg.norm(X) + eps)
    for _ in range(steps):
        A = X @ X.T
        B = b * A + c * (A @ A)
        X = a * X + B @ X
    return X.T.copy() if transposed else X


def ns_polynomial_schedule(G: np.ndarray, coeffs, eps: float = 1e-7) -> np.ndarray:
    """NS with an odd polynomial that changes from iteration to iteration:
    iteration k (k = 0, 1, ...) uses coeffs[k] = (a_k, b_k, c_k), i.e.
        A = X X^T,  B = b_k A + c_k A A,  X <- a_k X + B X,
    mapping each singular value s to a_k s + b_k s^3 + c_k s^5.  This is the
    shape of the minimax-optimised (Polar Express) and Chebyshev-type msign
    iterations that Section 2 names next to classical Newton-Schulz; they
    differ from it only in the coefficient table.  Normalisation and the
    tall-matrix orientation are as in ns_polynomial."""
    X = np.array(G, dtype=np.float64)
    if X.ndim != 2:
        raise ValueError("NS needs a 2-D matrix")
    transposed = X.shape[0] > X.shape[1]
    if transposed:
        X = X.T.copy()
    X = X / (np.linalg.norm(X) + eps)
    for a_k, b_k, c_k in coeffs:
        A = X @ X.T
        B = b_k * A + c_k * (A @ A)
        X = a_k * X + B @ X
    return X.T.copy() if transposed else X


def ns_polynomial_schedule_storage(G: np.ndarray, coeffs, eps: float = 1e-7,
                                   storage: str = "bf16") -> np.ndarray:
    """The NS recurrence with every stored intermediate rounded to the
    storage type ("bf16" or "f32"), as an implementation that keeps them in
    that type does (the precision reading "bf16 operands, fp32 accumulation",
    or the fp32 mode): X_0 = rd(G); per iteration A = rd(X X^T),
    B = rd(b_k A + c_k A A), X <- rd(a_k X + B X), products and sums in fp64;
    the normalisation 1/(||G||_F + eps) (of the unrounded G) is applied to A
    (squared) and to X in iteration 0.  It measures how far the storage
    precision alone moves a given coefficient table from the exact
    recurrence."""
    def rd(v):
        if storage == "bf16":
            return bf16_round(v).astype(np.float64)
        if storage == "f32":
            return np.asarray(v, dtype=np.float32).astype(np.float64)
        raise ValueError("storage must be 'bf16' or 'f32'")
    G = np.array(G, dtype=np.float64)
    transposed = G.shape[0] > G.shape[1]
    if transposed:
        G = G.T.copy()
    inv = 1.0 / (np.linalg.norm(G) + eps)
    X = rd(G)
    for k, (a_k, b_k, c_k) in enumerate(coeffs):
        s_a, s_x = (inv * inv, inv) if k == 0 else (1.0, 1.0)
        A = rd(s_a * (X @ X.T))
        B = rd(b_k * A + c_k * (A @ A))
        X = rd(s_x * (a_k * X + B @ X))
    if len(coeffs) == 0:
        X = X * inv
    return X.T.copy() if transposed else X


def ns_scalar_map_schedule(x: np.ndarray, coeffs) -> np.ndarray:
    """phi_K o ... o phi_1 (x) with phi_k(x) = a_k x + b_k x^3 + c_k x^5,
    applied in iteration order."""
    x = np.array(x, dtype=np.float64)
    for a_k, b_k, c_k in coeffs:
        x = a_k * x + b_k * x ** 3 + c_k * x ** 5
    return x


def odd_poly_eval(q, x):
    """p(x) = sum_j q_j x^(2j+1)."""
    x = np.asarray(x, dtype=np.float64)
    return sum(qj * x ** (2 * j + 1) for j, qj in enumerate(q))


def minimax_odd_polynomial(lo: float, hi: float, degree: int, grid: int = 20001):
    """The odd polynomial p of the given degree (3 or 5) that minimises
    max_{x in [lo, hi]} |1 - p(x)|: the per-iteration polynomial of the
    minimax ("Polar Express") msign iteration and, at degree 3, of the
    Chebyshev-type iteration (Section 2 names both).  Solved as written, as a
    linear program over a dense grid (Chebyshev-spaced, endpoints included):
        minimise E  subject to  -E <= 1 - p(x_i) <= E  for every grid point.
    scipy's LP solver (HiGHS) is the library primitive.  Returns (q, E) with
    q the coefficients of x, x^3[, x^5]."""
    from scipy.optimize import linprog
    if degree not in (3, 5) or not (0 < lo < hi):
        raise ValueError("degree 3 or 5 on 0 < lo < hi")
    d = (degree + 1) // 2
    t = np.cos(np.pi * np.arange(grid) / (grid - 1))
    x = np.sort(0.5 * (lo + hi) + 0.5 * (hi - lo) * t)
    V = np.stack([x ** (2 * j + 1) for j in range(d)], axis=1)
    ones = np.ones((grid, 1))
    # variables (q_0 .. q_{d-1}, E); constraints  p - E <= 1  and  -p - E <= -1
    A_ub = np.vstack([np.hstack([V, -ones]), np.hstack([-V, -ones])])
    b_ub = np.concatenate([np.ones(grid), -np.ones(grid)])
    cost = np.zeros(d + 1)
    cost[-1] = 1.0
    res = linprog(cost, A_ub=A_ub, b_ub=b_ub, bounds=[(None, None)] * (d + 1), method="highs")
    if not res.success:
        raise RuntimeError("minimax LP failed: " + res.message)
    return res.x[:d].copy(), float(res.x[d])


def minimax_schedule(steps: int, lo: float, degree: int = 5, safety: float = 1.0):
    """Coefficient table of the minimax msign iteration after the
    Frobenius normalisation (singular values in [lo, 1]): iteration k uses the
    minimax odd polynomial on the current interval [l_k, u_k], divided by
    ``safety`` (>= 1), and the next interval is that polynomial's image,
    l_{k+1} = p_k(l_k) and u_{k+1} = max of p_k on [l_k, u_k] (taken on the
    LP grid).  Degree 5 is the Polar Express construction, degree 3 the
    Chebyshev-type one.  Returns ((a_k, b_k, c_k), ...)."""
    out = []
    l, u = float(lo), 1.0
    for _ in range(steps):
        q, _E = minimax_odd_polynomial(l, u, degree)
        q = q / safety
        grid = np.linspace(l, u, 20001)
        l, u = float(odd_poly_eval(q, l)), float(odd_poly_eval(q, grid).max())
        out.append((float(q[0]), float(q[1]), float(q[2]) if len(q) > 2 else 0.0))
    return tuple(out)


def msign_svd(G: np.ndarray) -> np.ndarray:
    """Exact msign(G) = U V^T from the thin SVD G = U S V^T (Section 2,
    "msign(X) = U V^T"; Section 2.1, LMO of the spectral norm).  Zero singular
    values contribute nothing (the minimum-norm element of the subdifferential).
    LAPACK's SVD is the library primitive."""
    G = np.asarray(G, dtype=np.float64)
    U, s, Vt = np.linalg.svd(G, full_matrices=False)
    tol = s.max(initial=0.0) * max(G.shape) * np.finfo(np.float64).eps
    keep = s > tol
    return (U[:, keep] @ Vt[keep, :])


def ns_scalar_map(x: np.ndarray, steps: int, a: float, b: float, c: float) -> np.ndarray:
    """phi^K(x) with phi(x) = a x + b x^3 + c x^5: what NS does to each
    normalised singular value."""
    x = np.array(x, dtype=np.float64)
    for _ in range(steps):
        x = a * x + b * x ** 3 + c * x ** 5
    return x


# ---------------------------------------------------------------------------
# The two update rules of Algorithm 1 (fp64)
# ---------------------------------------------------------------------------

def lion_update(W, G_hat, eta_lion, weight_decay):
    """Lion branch of Algorithm 1: W <- W - eta_L (sign(G_hat) + lambda W)
    (in fp64 whatever the precision G_hat was formed in)."""
    return W - eta_lion * (sign(G_hat).astype(np.float64) + weight_decay * W)


def muon_update(W, G_hat, cfg: Config):
    """Muon branch of Algorithm 1 with Table 5's NS scaling:
    W <- W - eta_M (0.2 sqrt(max(m,n)) NS_K(G_hat) + lambda W)."""
    if cfg.ns_coeffs is not None:
        O = ns_polynomial_schedule(G_hat, cfg.ns_coeffs, cfg.ns_eps)
    else:
        O = ns_polynomial(G_hat, cfg.ns_steps, cfg.ns_a, cfg.ns_b, cfg.ns_c, cfg.ns_eps)
    scale = cfg.shape_scale * math.sqrt(max(W.shape))
    return W - cfg.eta_muon * (scale * O + cfg.weight_decay * W)


def adamw_update(W, G, m_prev, v_prev, step: int, lr, beta1, beta2, eps, weight_decay):
    """AdamW with decoupled weight decay (Loshchilov and Hutter), the update
    Section 3 gives 1-D parameters (biases, norm gains) in the LionMuon hybrid;
    ``step`` counts this parameter's AdamW updates, 1 for the first:
        m = beta1 m + (1 - beta1) G,   v = beta2 v + (1 - beta2) G^2
        m_hat = m / (1 - beta1^step),  v_hat = v / (1 - beta2^step)
        W <- W - lr lambda W - lr m_hat / (sqrt(v_hat) + eps)
    Returns (W_new, m, v), fp64."""
    if step < 1:
        raise ValueError("step counts updates from 1")
    W = np.asarray(W, dtype=np.float64)
    G = np.asarray(G, dtype=np.float64)
    m = beta1 * np.asarray(m_prev, dtype=np.float64) + (1.0 - beta1) * G
    v = beta2 * np.asarray(v_prev, dtype=np.float64) + (1.0 - beta2) * G * G
    m_hat = m / (1.0 - beta1 ** step)
    v_hat = v / (1.0 - beta2 ** step)
    W_new = W - lr * weight_decay * W - lr * m_hat / (np.sqrt(v_hat) + eps)
    return W_new, m, v


# ---------------------------------------------------------------------------
# Adaptive Muon/Lion selection (Appendix G)
# ---------------------------------------------------------------------------

_U64 = (1 << 64) - 1
_GOLDEN = 0x9E3779B97F4A7C15


def splitmix64(seed: int, count: int) -> List[int]:
    """The first ``count`` outputs of SplitMix64 (Steele, Lea and Flood,
    2014) started from ``seed``: the state advances by 0x9E3779B97F4A7C15 and
    each output is the state passed through the two xor-shift-multiply
    rounds (multipliers 0xBF58476D1CE4E5B9, 0x94D049BB133111EB) and a final
    xor-shift by 31.  Output j depends only on seed + (j + 1) * golden, so it
    is a counter-based generator."""
    out = []
    state = seed & _U64
    for _ in range(count):
        state = (state + _GOLDEN) & _U64
        z = state
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _U64
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _U64
        out.append(z ^ (z >> 31))
    return out


def power_start_vector(n: int, seed: int) -> np.ndarray:
    """Start vector of the power iteration (the paper leaves it open):
    entry j = 2 * (top 53 bits of SplitMix64 output j) / 2^53 - 1, in [-1, 1)."""
    return np.array([2.0 * ((z >> 11) * 2.0 ** -53) - 1.0 for z in splitmix64(seed, n)], dtype=np.float64)


def stable_rank_estimate(M: np.ndarray, iters: int, v0: np.ndarray):
    """||M||_F^2 and the power-iteration estimate of sigma_1(M)^2 (Appendix G:
    sigma_1 "approximated by a few power-iteration steps").  With
    v = v0 / ||v0||, each of the ``iters`` passes forms u = M v and takes
    ||u||^2 as the estimate; every pass but the last also forms w = M^T u and
    v = w / ||w||.  So the estimate is the Rayleigh quotient of M^T M at
    (M^T M)^(iters-1) v0, never above sigma_1^2.  Returns (fro2, sigma2)."""
    M = np.asarray(M, dtype=np.float64)
    fro2 = float(np.sum(M * M))
    v = np.asarray(v0, dtype=np.float64)
    v = v / np.linalg.norm(v)
    sigma2 = 0.0
    for k in range(iters):
        u = M @ v
        sigma2 = float(u @ u)
        if k + 1 < iters:
            w = M.T @ u
            nw = np.linalg.norm(w)
            if nw == 0.0:
                break
            v = w / nw
    return fro2, sigma2


def srank_takes_muon(M_prev: np.ndarray, cfg: "Config") -> bool:
    """Appendix G's rule on the momentum buffer M_{t-1}: Muon iff the stable
    rank estimate ||M||_F^2 / sigma_1_hat^2 <= alpha * min(m, n), decided as
    ||M||_F^2 <= alpha * min(m, n) * sigma_1_hat^2.  A zero buffer (t = 0)
    takes Muon, as step 0 does under the fixed period."""
    m, n = np.shape(M_prev)
    fro2, sigma2 = stable_rank_estimate(M_prev, cfg.srank_iters, power_start_vector(n, cfg.srank_seed))
    if fro2 == 0.0:
        return True
    return fro2 <= cfg.srank_alpha * min(m, n) * sigma2


def is_matrix(shape: Sequence[int]) -> bool:
    """A parameter is a hidden matrix (takes Muon steps) unless it is a vector
    (one of its two dimensions is 1)."""
    return len(shape) == 2 and shape[0] > 1 and shape[1] > 1


def lionmuon_param_step(W, G, M_prev, t: int, cfg: Config, sign_in_f32: bool = False,
                        take_muon: Optional[bool] = None):
    """One iteration of Algorithm 1 for one parameter, fp64.

    With ``sign_in_f32`` the Lion branch decides sign(G_hat) on the float32
    value of G_hat formed as fl(fl(b1*M) + fl(c1*G)) with float32 constants
    (the order the CUDA library uses), so both sides take the same integer
    decision near ties; the update itself stays fp64.
    ``take_muon`` overrides the branch of a matrix (the adaptive schedule).
    Returns (W_{t+1}, M_t)."""
    W = np.asarray(W, dtype=np.float64)
    G = np.asarray(G, dtype=np.float64)
    M_prev = np.asarray(M_prev, dtype=np.float64)
    G_hat = interpolated_direction(M_prev, G, cfg.beta1)
    muon = is_muon_step(t, cfg.period) if take_muon is None else take_muon
    if is_matrix(W.shape) and muon:
        W_new = muon_update(W, G_hat, cfg)
    else:
        direction = G_hat
        if sign_in_f32:
            b1, c1 = np.float32(cfg.beta1), np.float32(1.0 - cfg.beta1)
            direction = (b1 * M_prev.astype(np.float32)) + (c1 * G.astype(np.float32))
        W_new = lion_update(W, direction, cfg.eta_lion, cfg.weight_decay)
    M_new = momentum_update(M_prev, G, cfg.beta2)
    return W_new, M_new


# ---------------------------------------------------------------------------
# Storage modelling (bf16 / fp32 rounding of the persisted state)
# ---------------------------------------------------------------------------

def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round to the nearest bfloat16 value, ties to even, returned as float32.

    Written from the IEEE-754 binary32 layout: bfloat16 keeps the top 16 bits.
    Adding 0x7FFF plus the lowest kept bit to the 32-bit pattern and
    truncating rounds to nearest with ties to even; the carry into the
    exponent handles overflow to infinity.  NaN stays NaN (quiet)."""
    f = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    u = f.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    r = ((u + 0x7FFF + lsb) >> 16) << 16
    out = (r & 0xFFFFFFFF).astype(np.uint32).view(np.float32)
    return np.where(np.isnan(f), np.float32(np.nan), out).astype(np.float32)


def round_to_storage(x: np.ndarray, dtype: str) -> np.ndarray:
    """Round fp64 values to what a buffer of ``dtype`` ('bf16' or 'f32') holds,
    returned as float64 for further fp64 arithmetic."""
    if dtype == "f32":
        return np.asarray(x, dtype=np.float32).astype(np.float64)
    if dtype == "bf16":
        return bf16_round(np.asarray(x, dtype=np.float64).astype(np.float32)).astype(np.float64)
    raise ValueError(f"unknown storage dtype {dtype!r}")


def lionmuon_step(params: List[np.ndarray], grads: List[np.ndarray],
                  moms: List[np.ndarray], t: int, cfg: Config,
                  param_dtypes: Optional[List[str]] = None,
                  seconds: Optional[List[np.ndarray]] = None):
    """One LionMuon step over a list of parameters (Algorithm 1 applied to
    each matrix; vectors take the Lion step every step, or AdamW when
    ``cfg.vector_rule == "adamw"``, with M as AdamW's first moment, the
    second moments in ``seconds`` and the update count t + 1).

    With ``param_dtypes`` given, the new weights are rounded to their storage
    dtype, the momentum (and second moments) to float32, and Lion signs are
    decided on the float32 G_hat (storage-modelled mode); otherwise the state
    stays in fp64 (exact mode).  Returns (new_params, new_moms), plus
    new_seconds when ``seconds`` is given."""
    if not (len(params) == len(grads) == len(moms)):
        raise ValueError("params, grads and moms must have equal length")
    adamw = cfg.vector_rule == "adamw"
    if cfg.vector_rule not in ("lion", "adamw"):
        raise ValueError("vector_rule must be 'lion' or 'adamw'")
    if adamw and seconds is None:
        raise ValueError("the AdamW rule needs the second moments")
    if cfg.schedule not in ("period", "stable_rank"):
        raise ValueError("schedule must be 'period' or 'stable_rank'")
    new_p, new_m, new_v = [], [], []
    for i, (W, G, M) in enumerate(zip(params, grads, moms)):
        if np.shape(W) != np.shape(G) or np.shape(W) != np.shape(M):
            raise ValueError(f"shape mismatch at parameter {i}")
        V1 = None if seconds is None else seconds[i]
        if adamw and not is_matrix(np.shape(W)):
            W1, M1, V1 = adamw_update(W, G, M, seconds[i], t + 1, cfg.adamw_lr, cfg.adamw_beta1,
                                      cfg.adamw_beta2, cfg.adamw_eps, cfg.adamw_weight_decay)
        else:
            take = None
            if cfg.schedule == "stable_rank" and is_matrix(np.shape(W)):
                take = srank_takes_muon(M, cfg)
            W1, M1 = lionmuon_param_step(W, G, M, t, cfg, sign_in_f32=param_dtypes is not None,
                                         take_muon=take)
        if param_dtypes is not None:
            W1 = round_to_storage(W1, param_dtypes[i])
            M1 = round_to_storage(M1, "f32")
            if V1 is not None:
                V1 = round_to_storage(V1, "f32")
        new_p.append(W1)
        new_m.append(M1)
        new_v.append(V1)
    if seconds is not None:
        return new_p, new_m, new_v
    return new_p, new_m


# ---------------------------------------------------------------------------
# Same-order float32 Lion step (bit-level reference)
# ---------------------------------------------------------------------------

def lion_constants_f32(beta1, beta2, eta_lion, weight_decay):
    """The six float32 constants of the Lion step, each rounded once from
    float64: (beta1, 1-beta1, beta2, 1-beta2, eta_L, lambda)."""
    f = np.float32
    return (f(beta1), f(1.0 - beta1), f(beta2), f(1.0 - beta2), f(eta_lion), f(weight_decay))


def lion_step_f32(w: np.ndarray, g: np.ndarray, m: np.ndarray, beta1, beta2,
                  eta_lion, weight_decay, w_dtype: str = "bf16"):
    """Lion branch + momentum update of Algorithm 1 evaluated in float32 with a
    fixed operation order, every product and sum rounded separately (no fused
    multiply-add):

        gh = b1*m + c1*g ;  u = sign(gh)
        w  = w - eL*(u + lam*w)      (then bf16 round-to-nearest-even if bf16)
        m  = b2*m + c2*g

    ``w`` and ``g`` hold the stored values (bf16 values as float32), ``m`` is
    float32.  numpy evaluates each float32 operation with one rounding, which
    is what makes this a bit-level reference.  Returns (w_new, m_new) as
    float32 arrays."""
    b1, c1, b2, c2, eL, lam = lion_constants_f32(beta1, beta2, eta_lion, weight_decay)
    w = np.asarray(w, dtype=np.float32)
    g = np.asarray(g, dtype=np.float32)
    m = np.asarray(m, dtype=np.float32)
    gh = (b1 * m) + (c1 * g)
    u = sign(gh).astype(np.float32)
    w_new = w - eL * (u + lam * w)
    m_new = (b2 * m) + (c2 * g)
    if w_dtype == "bf16":
        w_new = bf16_round(w_new)
    elif w_dtype != "f32":
        raise ValueError(f"unknown w dtype {w_dtype!r}")
    return w_new.astype(np.float32), m_new.astype(np.float32)


def adamw_constants_f32(step: int, lr, beta1, beta2, eps, weight_decay):
    """The float32 constants of one AdamW step, each rounded once from its
    double value: b1, 1 - b1, b2, 1 - b2, lr / (1 - beta1^step),
    1 / sqrt(1 - beta2^step), lr * lambda, eps (powers and roots in double,
    by the C library's pow and sqrt)."""
    f = np.float32
    bc1 = 1.0 - math.pow(beta1, step)
    bc2 = 1.0 - math.pow(beta2, step)
    return (f(beta1), f(1.0 - beta1), f(beta2), f(1.0 - beta2), f(lr / bc1), f(1.0 / math.sqrt(bc2)),
            f(lr * weight_decay), f(eps))


def adamw_step_f32(w, g, m, v, step: int, lr, beta1, beta2, eps, weight_decay, w_dtype: str = "bf16"):
    """AdamW step in float32 with a fixed operation order, every operation
    rounded once (no fused multiply-add; sqrt and division correctly
    rounded):
        m = b1*m + c1*g ;  v = b2*v + c2*(g*g)
        w = w - lrwd*w ;   den = sqrt(v)*rbc2 + eps ;  w = w - step_size*(m/den)
    then bf16 round-to-nearest-even of w for bf16 parameters.  Returns
    (w, m, v) as float32 arrays."""
    b1, c1, b2, c2, st, rbc2, lrwd, e = adamw_constants_f32(step, lr, beta1, beta2, eps, weight_decay)
    w = np.asarray(w, dtype=np.float32)
    g = np.asarray(g, dtype=np.float32)
    m = (b1 * np.asarray(m, dtype=np.float32)) + (c1 * g)
    v = (b2 * np.asarray(v, dtype=np.float32)) + (c2 * (g * g))
    w = w - lrwd * w
    den = (np.sqrt(v) * rbc2) + e
    w = w - st * (m / den)
    if w_dtype == "bf16":
        w = bf16_round(w)
    elif w_dtype != "f32":
        raise ValueError(f"unknown w dtype {w_dtype!r}")
    return w.astype(np.float32), m.astype(np.float32), v.astype(np.float32)


# ---------------------------------------------------------------------------
# Cost model (for reporting; FLOP counts of the method's contractions)
# ---------------------------------------------------------------------------

def ns_flops(m: int, n: int, steps: int, symmetric: bool = True) -> float:
    """FLOPs of NS_K on an m x n matrix, s = min, l = max.  Per iteration:
    X X^T (s^2 l with the symmetric half, 2 s^2 l dense), A A (s^3 / 2 s^3),
    B X (2 s^2 l)."""
    s, l = min(m, n), max(m, n)
    per = (3 * s * s * l + s ** 3) if symmetric else (4 * s * s * l + 2 * s ** 3)
    return float(steps) * per
