"""GPU parity of whole LionMuon steps (Algorithm 1) through lm_create/lm_step
against the storage-modelled fp64 oracle: weights within 1e-3 relative
(Frobenius) after 8 steps with the fp32 Newton-Schulz path, and within the
bound the 2e-2 NS tolerance implies with the bf16 tensor-core path (and the
2e-5 one with the three-piece tensor-core mode, ns_precision 2); momentum
bit-exact (same-order fp32 EMA); the Muon direction itself within the NS
tolerance; plus the state-size invariant, status flags and argument errors."""

import numpy as np
import pytest

import oracle as O
from paper_2605_19811_gb300 import synth
from tests.lm_testutil import (bits, host_tensor, make_problem, rel_fro, run_trajectory_gpu,
                               run_trajectory_oracle, stored_values)

pytestmark = pytest.mark.gpu

TINY = synth.PARAM_SETS["tiny"]


def _cfg_pair(**kw):
    gpu = dict(kw)
    ora = O.Config(**{k: v for k, v in kw.items() if k != "ns_precision"})
    return gpu, ora


NS_TOL_BF16 = 2e-2     # relative Frobenius tolerance of the bf16 NS output
NS_TOL_F32TC = 2e-5    # the same for the three-piece tensor-core mode
F32TC = 2              # LM_NS_F32_TC
BF16_ULP = 2.0 ** -8   # relative spacing of bf16 values (upper bound)


def _check(Wg, Wo, Mg, Mo, tol):
    """tol: one float for every parameter, or a list with one per parameter."""
    tols = tol if isinstance(tol, (list, tuple)) else [tol] * len(Wo)
    worst = []
    for wg, wo, mg, mo, tl in zip(Wg, Wo, Mg, Mo, tols):
        if wo.size == 0:
            continue
        e = rel_fro(wg, wo)
        worst.append((e, tl))
        # the momentum EMA is the same float32 formula on both sides
        np.testing.assert_array_equal(mg.astype(np.float32).view(np.uint32),
                                      mo.astype(np.float32).view(np.uint32))
    assert all(e <= tl for e, tl in worst), worst
    return worst


def _bf16_ns_bounds(W0, grads, dtype, cfg: O.Config, steps, Wo, tau_ns=NS_TOL_BF16, storage="bf16", floor=1e-3):
    """Weight tolerance implied by the NS tolerance for the bf16 tensor-core
    path.  The gradients do not depend on W, so the momentum and G_hat are the
    same on both sides and a weight difference only comes from the Muon
    updates: each adds at most eta_M * s * tau * ||NS(G_hat)||_F (s the shape
    scale, tau = 2e-2), carried forward with the decay factor (1 - eta lambda)
    <= 1.  For bf16 parameters a pre-rounding difference d of relative size r
    also flips the bf16 rounding of about a fraction r/u of the entries (u the
    bf16 spacing), which adds sqrt(r u) in relative Frobenius terms.  The
    bound per parameter is 1e-3 + r + sqrt(r u) (the last term for bf16).
    tau_ns, storage, floor: the same bound for another NS mode (the
    three-piece mode: 2e-5, fp32 storage, floor 1e-6 for fp32 W)."""
    P = [stored_values(host_tensor(w, dtype)) for w in W0]
    M = [np.zeros_like(p) for p in P]
    acc = [0.0] * len(P)
    for t in range(steps):
        G = [stored_values(host_tensor(g, dtype)) for g in grads[t]]
        for i, (p, g, m) in enumerate(zip(P, G, M)):
            if O.is_matrix(p.shape) and O.is_muon_step(t, cfg.period):
                gh = O.interpolated_direction(m, g, cfg.beta1)
                tau = tau_ns
                if cfg.ns_coeffs is not None:
                    o = O.ns_polynomial_schedule(gh, cfg.ns_coeffs, cfg.ns_eps)
                    # the table's own sensitivity to storage (see test_gpu_msign.table_tolerance)
                    d = rel_fro(O.ns_polynomial_schedule_storage(gh, cfg.ns_coeffs, cfg.ns_eps, storage), o)
                    tau = max(tau, 1.5 * d)
                else:
                    o = O.ns_polynomial(gh, cfg.ns_steps, cfg.ns_a, cfg.ns_b, cfg.ns_c, cfg.ns_eps)
                acc[i] += cfg.eta_muon * cfg.shape_scale * np.sqrt(max(p.shape)) * tau * np.linalg.norm(o)
            M[i] = O.momentum_update(m, g, cfg.beta2)
    out = []
    for a, w in zip(acc, Wo):
        r = a / max(np.linalg.norm(w), 1e-30)
        out.append(floor + r + (np.sqrt(r * BF16_ULP) if dtype == "bf16" else 0.0))
    return out


def _momentum_same_order(grads, shapes, beta2, steps):
    """fp32 momentum after ``steps`` steps, evaluated with the same-order rule."""
    M = [np.zeros(s, dtype=np.float32) for s in shapes]
    for t in range(steps):
        for i in range(len(shapes)):
            _, M[i] = O.lion_step_f32(np.zeros(shapes[i], np.float32), grads[t][i], M[i],
                                      0.9, beta2, 0.0, 0.0, w_dtype="f32")
    return M


def _f32tc_bounds(W0, grads, dtype, cfg, steps, Wo):
    return _bf16_ns_bounds(W0, grads, dtype, cfg, steps, Wo, tau_ns=NS_TOL_F32TC, storage="f32",
                           floor=1e-3 if dtype == "bf16" else 1e-6)


@pytest.mark.parametrize("precision", [1, 0, F32TC])
def test_tiny_config_4_steps(precision):
    """The Tiny set: fp32 params, N(0,1) grads from seed 0, P=2, 4 steps,
    beta=(0.9,0.99), eta=0.02, lambda=0.1, NS per the paper (K=5)."""
    steps = 4
    W0, grads = make_problem(TINY.shapes, "normal", steps)
    gcfg, ocfg = _cfg_pair(beta1=0.9, beta2=0.99, eta_muon=0.02, eta_lion=0.02, weight_decay=0.1,
                           period=2, ns_precision=precision)
    Wg, Mg, flags = run_trajectory_gpu(W0, grads, "f32", gcfg, steps)
    Wo, _ = run_trajectory_oracle(W0, grads, "f32", ocfg, steps)
    Mo = _momentum_same_order([[stored_values(host_tensor(g, "f32")).astype(np.float32) for g in gs]
                               for gs in grads], TINY.shapes, 0.99, steps)
    tol = (1e-5 if precision == 0 else _f32tc_bounds(W0, grads, "f32", ocfg, steps, Wo) if precision == F32TC
           else _bf16_ns_bounds(W0, grads, "f32", ocfg, steps, Wo))
    _check(Wg, Wo, Mg, Mo, tol)
    assert flags == 0


SMALL_GPT = synth.scaled_set("small_gpt", layers=2, d=128, vocab=1000)


@pytest.mark.parametrize("period", [2, 1, 4])
@pytest.mark.parametrize("precision", [1, 0, F32TC])
def test_small_gpt_8_steps(period, precision):
    """bf16 GPT-style set (2 layers, d=128, vocab 1000, heavy-tailed grads):
    weights after 8 steps within 1e-3 of the storage-modelled oracle."""
    steps = 8
    shapes = SMALL_GPT.shapes
    W0, grads = make_problem(shapes, "student_t", steps)
    gcfg, ocfg = _cfg_pair(eta_muon=3e-3, eta_lion=2e-5, weight_decay=0.1, period=period,
                           ns_precision=precision)
    Wg, Mg, flags = run_trajectory_gpu(W0, grads, "bf16", gcfg, steps)
    Wo, _ = run_trajectory_oracle(W0, grads, "bf16", ocfg, steps)
    Mo = _momentum_same_order([[stored_values(host_tensor(g, "bf16")).astype(np.float32) for g in gs]
                               for gs in grads], shapes, 0.99, steps)
    tol = (1e-3 if precision == 0 else _f32tc_bounds(W0, grads, "bf16", ocfg, steps, Wo) if precision == F32TC
           else _bf16_ns_bounds(W0, grads, "bf16", ocfg, steps, Wo))
    worst = _check(Wg, Wo, Mg, Mo, tol)
    # the measured relative weight error per parameter, beside its bound (-s shows it)
    print(f"P={period} ns_precision={precision}: " +
          "; ".join(f"{tuple(s)} {e:.2e} <= {tl:.2e}" for s, (e, tl) in zip(shapes, worst)))
    assert flags == 0


@pytest.mark.parametrize("precision,tau", [(1, NS_TOL_BF16), (0, 1e-5), (F32TC, NS_TOL_F32TC)])
def test_muon_step_direction_within_ns_tolerance(precision, tau):
    """One Muon step on fp32 parameters (Algorithm 1, Muon branch): the
    direction recovered from the weight change,
    O = (W_t - W_{t+1} - eta lambda W_t) / (eta s), matches the oracle's
    NS_5(G_hat) within the NS tolerance (wide, tall and square matrices)."""
    shapes = [(192, 640), (640, 192), (256, 256), (300, 130)]
    W0, grads = make_problem(shapes, "student_t", 1, w_std=1.0)
    eta, lam = 1.0, 0.1
    gcfg, ocfg = _cfg_pair(eta_muon=eta, weight_decay=lam, period=1, ns_precision=precision)
    Wg, _, flags = run_trajectory_gpu(W0, grads, "f32", gcfg, 1)
    for w0, g, w1, shp in zip(W0, grads[0], Wg, shapes):
        w0 = w0.astype(np.float64)
        s = 0.2 * np.sqrt(max(shp))
        o_gpu = (w0 - w1 - eta * lam * w0) / (eta * s)
        o_ref = O.ns_polynomial(0.1 * g.astype(np.float64), 5, *O.NS_QUINTIC, 1e-7)
        # fp32 storage of W adds about |W| * 2^-24 / (eta s) to the recovered O
        slack = 4 * np.linalg.norm(w0) * 2.0 ** -24 / (eta * s) / np.linalg.norm(o_ref)
        assert rel_fro(o_gpu, o_ref) <= tau + slack
    assert flags == 0


@pytest.mark.parametrize("precision,tau", [(1, NS_TOL_BF16), (0, 1e-5), (F32TC, NS_TOL_F32TC)])
def test_muon_step_degenerate_gradients(precision, tau):
    """The method's degenerate inputs on a Muon step (Algorithm 1, Muon
    branch).  A zero gradient: G_hat = 0, X_0 = 0 / (0 + eps) = 0, every NS
    output is 0 and the step is pure decay.  Rank-one gradients s u v^T, wide,
    tall and square: the exact NS output is phi^5(x) u v^T / (|u| |v|), but
    NS raises any singular value near 0 about 480-fold over five quintic
    iterations, so the rounding of X_0 alone fills the null space with
    directions that differ from run to run (the oracle's storage model puts a
    bf16 result 117% and an fp32 one 1.7e-5 away from the exact output).  What
    is unique is checked: the component u^T O v along the input's singular
    pair, within the NS tolerance of the oracle's (the storage model: at most
    2.2e-3 bf16, 1e-8 fp32); the rest must be a valid NS output, every
    singular value within the quintic's range [0, 1.2024].  Momentum
    bit-exact; no status flag."""
    shapes = [(192, 640), (640, 192), (256, 256), (200, 72), (72, 200)]
    rng = np.random.default_rng(21)
    W0 = [rng.standard_normal(s).astype(np.float32) for s in shapes]
    u = [rng.standard_normal(s[0]) for s in shapes]
    v = [rng.standard_normal(s[1]) for s in shapes]
    scale = [0.0, 1.0, 1e-3, 1.0, 1e-3]
    G = [(c * np.outer(a, b)).astype(np.float32) for c, a, b in zip(scale, u, v)]
    eta, lam = 1.0, 0.1
    gcfg, _ = _cfg_pair(eta_muon=eta, weight_decay=lam, period=1, ns_precision=precision)
    Wg, Mg, flags = run_trajectory_gpu(W0, [G], "f32", gcfg, 1)
    assert flags == 0
    for w0, g, w1, m1, shp, a, b in zip(W0, G, Wg, Mg, shapes, u, v):
        w0 = w0.astype(np.float64)
        s = 0.2 * np.sqrt(max(shp))
        o_gpu = (w0 - w1 - eta * lam * w0) / (eta * s)
        # fp32 storage of W moves the recovered direction by |W| 2^-24 / (eta s) per entry
        slack = 4 * np.linalg.norm(w0) * 2.0 ** -24 / (eta * s)
        if not g.any():
            assert np.linalg.norm(o_gpu) <= slack
        else:
            o_ref = O.ns_polynomial(0.1 * g.astype(np.float64), 5, *O.NS_QUINTIC, 1e-7)
            uh, vh = a / np.linalg.norm(a), b / np.linalg.norm(b)
            p_gpu, p_ref = uh @ o_gpu @ vh, uh @ o_ref @ vh
            assert abs(p_gpu - p_ref) <= tau * abs(p_ref) + slack, (shp, p_gpu, p_ref)
            assert np.linalg.norm(o_gpu, 2) <= 1.2024 + 1e-2 + slack
        _, m_ref = O.lion_step_f32(np.zeros_like(g), g, np.zeros_like(g), 0.9, 0.99, 0.0, 0.0, w_dtype="f32")
        np.testing.assert_array_equal(m1.astype(np.float32).view(np.uint32), m_ref.view(np.uint32))


def test_p_infinity_matrices_take_lion_steps_bit_exact():
    """period = 0 (P = infinity): every parameter, matrices included, takes
    the Lion step; bit-exact against the same-order oracle."""
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    shapes = [(96, 200), (200, 96), (96,)]
    W0, grads = make_problem(shapes, "student_t", 3)
    params = [host_tensor(w, "bf16").cuda() for w in W0]
    opt = L.LionMuon(params, period=0, eta_lion=1e-3)
    rw = [host_tensor(w, "bf16").float().numpy() for w in W0]
    rm = [np.zeros(s, np.float32) for s in shapes]
    for t in range(3):
        gh = [host_tensor(g, "bf16") for g in grads[t]]
        opt.step([g.cuda() for g in gh], t)
        for i in range(3):
            rw[i], rm[i] = O.lion_step_f32(rw[i], gh[i].float().numpy(), rm[i], 0.9, 0.99, 1e-3, 0.1)
    torch.cuda.synchronize()
    for i in range(3):
        np.testing.assert_array_equal(bits(params[i]), bits(torch.from_numpy(rw[i]).to(torch.bfloat16)))
    opt.close()


def test_state_bytes_is_one_fp32_buffer_per_parameter():
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    shapes = SMALL_GPT.shapes
    params = [torch.zeros(s, dtype=torch.bfloat16, device="cuda") for s in shapes]
    opt = L.LionMuon(params)
    assert opt.state_bytes() == 4 * sum(int(np.prod(s)) for s in shapes)
    assert opt.workspace_bytes() > 0
    m = opt.momentum(0)
    assert m.shape == params[0].shape and m.dtype == torch.float32
    assert float(m.abs().sum()) == 0.0      # M_{-1} = 0
    opt.close()


def test_nonfinite_gradient_sets_flag():
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    p = [torch.zeros((64, 96), dtype=torch.bfloat16, device="cuda")]
    opt = L.LionMuon(p, period=1)
    g = torch.randn((64, 96), device="cuda").to(torch.bfloat16)
    g[5, 7] = float("inf")
    opt.step([g], 0)
    assert opt.status() & L.LM_FLAG_NONFINITE
    assert opt.status() == 0          # flags are cleared by the read
    opt.close()


def test_step_argument_errors():
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    p = [torch.zeros((32, 48), dtype=torch.bfloat16, device="cuda"), torch.zeros(48, device="cuda")]
    opt = L.LionMuon(p)
    with pytest.raises(L.LionMuonError) as e:
        opt.step([torch.zeros((32, 48), dtype=torch.bfloat16, device="cuda")], 0)
    assert e.value.status == 1
    with pytest.raises(L.LionMuonError) as e:
        opt.step([torch.zeros((48, 32), dtype=torch.bfloat16, device="cuda"),
                  torch.zeros(48, device="cuda")], 0)
    assert e.value.status == 1
    with pytest.raises(L.LionMuonError) as e:
        opt.step([torch.zeros((32, 48), device="cuda"), torch.zeros(48, device="cuda")], 0)
    assert e.value.status == 2
    with pytest.raises(L.LionMuonError) as e:
        opt.step([torch.zeros((32, 48), dtype=torch.bfloat16, device="cuda"),
                  torch.zeros(48, device="cuda")], -1)
    assert e.value.status == 1
    opt.close()


def test_set_lr_and_checkpoint_resume():
    """Restoring M and passing the same t resumes the trajectory exactly."""
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    shapes = [(64, 192), (192,)]
    W0, grads = make_problem(shapes, "student_t", 4)

    def run(split):
        params = [host_tensor(w, "bf16").cuda() for w in W0]
        opt = L.LionMuon(params, period=2, eta_muon=1e-2, eta_lion=1e-3)
        for t in range(4):
            if t == split:
                saved = [opt.momentum(i).clone() for i in range(2)]
                snap = [p.clone() for p in params]
                opt.close()
                params = snap
                opt = L.LionMuon(params, period=2, eta_muon=1e-2, eta_lion=1e-3)
                for i in range(2):
                    opt.set_momentum(i, saved[i])
            opt.step([host_tensor(g, "bf16").cuda() for g in grads[t]], t)
        torch.cuda.synchronize()
        out = [p.cpu() for p in params]
        opt.close()
        return out

    a, b = run(-1), run(2)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(bits(x), bits(y))


def test_fused_parameter_write_matches_finalize_kernel_bit_exact():
    """The Muon parameter write W <- W - eta_M (s X_K + lambda W) runs in the
    last Newton-Schulz epilogue when every matrix is bf16 with a column count
    divisible by 8, and in a separate kernel otherwise; both evaluate the same
    float32 expression on the same bf16 X_K, so the weights agree bit for bit.
    A 40 x 36 matrix added to the set switches the fusion off.  The fused
    write loads and stores W in 64-column boxes of 128 (load) or 32 (store)
    rows: the shapes put box edges past W's last row and column, partly
    (300 x 136: rows 288-299 of a 32-row box, columns 128-135 of a 64-column
    box) and wholly (384 x 256, 136 x 520), in both orientations."""
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    shapes = [(256, 384), (384, 256), (320, 320), (300, 136), (136, 520), (128,)]
    W0, grads = make_problem(shapes + [(40, 36)], "student_t", 2)
    out = []
    for n in (len(shapes), len(shapes) + 1):
        params = [host_tensor(w, "bf16").cuda() for w in W0[:n]]
        opt = L.LionMuon(params, period=2, eta_muon=0.02, weight_decay=0.1)
        for t in range(2):
            opt.step([host_tensor(g, "bf16").cuda() for g in grads[t][:n]], t)
        torch.cuda.synchronize()
        assert opt.status() == 0
        out.append([bits(p) for p in params[:len(shapes)]])
        opt.close()
    for a, b in zip(*out):
        np.testing.assert_array_equal(a, b)


@pytest.mark.parametrize("table_name", ["polar_express", "chebyshev_cubic"])
@pytest.mark.parametrize("precision", [1, 0, F32TC])
def test_small_gpt_8_steps_polar_express_table(precision, table_name):
    """Whole steps with an iteration-dependent NS table (the degree-5 minimax
    schedule from l_0 = 1e-3, or the degree-3 one, whose iterations have
    c = 0 and run without the polynomial launch, the parameter write fused
    into an APPLY that reads A): weights after 8 steps against the
    storage-modelled oracle run with the same table."""
    from paper_2605_19811_gb300 import ns_coeffs as C
    table = {"polar_express": C.polar_express, "chebyshev_cubic": C.chebyshev_cubic}[table_name](5, 1e-3)
    steps = 8
    shapes = SMALL_GPT.shapes
    W0, grads = make_problem(shapes, "student_t", steps)
    gcfg, ocfg = _cfg_pair(eta_muon=3e-3, eta_lion=2e-5, weight_decay=0.1, period=2,
                           ns_precision=precision, ns_coeffs=table)
    Wg, Mg, flags = run_trajectory_gpu(W0, grads, "bf16", gcfg, steps)
    Wo, _ = run_trajectory_oracle(W0, grads, "bf16", ocfg, steps)
    Mo = _momentum_same_order([[stored_values(host_tensor(g, "bf16")).astype(np.float32) for g in gs]
                               for gs in grads], shapes, 0.99, steps)
    tol = (1e-3 if precision == 0 else _f32tc_bounds(W0, grads, "bf16", ocfg, steps, Wo) if precision == F32TC
           else _bf16_ns_bounds(W0, grads, "bf16", ocfg, steps, Wo))
    _check(Wg, Wo, Mg, Mo, tol)
    assert flags == 0


def test_coefficient_table_rejected_when_not_finite():
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    p = [torch.zeros((32, 48), dtype=torch.bfloat16, device="cuda")]
    with pytest.raises(L.LionMuonError) as e:
        L.LionMuon(p, ns_coeffs=[(1.0, 0.0, 0.0), (float("inf"), 0.0, 0.0)])
    assert e.value.status == 1
