"""GPU parity of the adaptive Muon/Lion selection (LM_SCHEDULE_STABLE_RANK,
Appendix G): the per-matrix stable-rank estimates and decisions against the
oracle on the same momentum buffers (low-rank and full-rank buffers set
through lm_set_momentum; wide, tall, square, columns not divisible by 4, more
than 8192 columns); whole mixed steps against the storage-modelled oracle
(Lion-selected matrices and vectors bit-exact, Muon-selected ones within the
NS-derived bound); the zero buffer at t = 0; the period schedule's report;
argument errors."""

import numpy as np
import pytest

import oracle as O
from tests.lm_testutil import bits, host_tensor, rel_fro, stored_values

pytestmark = pytest.mark.gpu

SHAPES = [(96, 200), (200, 96), (128, 128), (64, 250), (16, 9000), (300, 1280), (200,)]


def _buffer(shape, kind, r):
    m, n = shape
    if kind == "lowrank":      # two directions plus a little noise: stable rank ~1
        a = r.normal(size=(m, 2)) @ np.diag([3.0, 1.0]) @ r.normal(size=(2, n))
        return (a + 0.01 * r.normal(size=shape)).astype(np.float32) * 1e-3
    return r.normal(size=shape).astype(np.float32) * 1e-3    # full rank: stable rank ~ min(m, n) / 4


def _state(shapes, kinds, seed, **cfg):
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    r = np.random.default_rng(seed)
    W0 = [r.normal(0, 0.02, size=s).astype(np.float32) for s in shapes]
    M0 = [(_buffer(s, k, r) if len(s) == 2 else r.normal(size=s).astype(np.float32) * 1e-3)
          for s, k in zip(shapes, kinds)]
    params = [host_tensor(w, "bf16").cuda() for w in W0]
    opt = L.LionMuon(params, schedule=L.LM_SCHEDULE_STABLE_RANK, **cfg)
    for i, m in enumerate(M0):
        opt.set_momentum(i, torch.from_numpy(m).cuda())
    torch.cuda.synchronize()
    return opt, params, W0, M0


@pytest.mark.parametrize("scale", [1e-16, 1e9])
def test_estimates_hold_at_extreme_momentum_scales(scale):
    """Momentum entries of 1e-16 or 1e9 (the power-iteration vectors M^T u then
    have entries near 1e-30 or 1e21, whose squares leave the fp32 range): the
    estimates still match the fp64 oracle."""
    import torch
    kinds = ["lowrank", "noise", "lowrank", "noise", "lowrank", "noise", None]
    opt, params, _, M0 = _state(SHAPES, kinds, 4, srank_alpha=0.08, srank_iters=5)
    for i, m in enumerate(M0):
        M0[i] = (m.astype(np.float64) * (scale / 1e-3)).astype(np.float32)
        opt.set_momentum(i, torch.from_numpy(M0[i]).cuda())
    g = [torch.zeros(s, dtype=torch.bfloat16, device="cuda") for s in SHAPES]
    opt.step(g, 3)
    took, est = opt.selection()
    for i, s in enumerate(SHAPES):
        if len(s) == 1:
            continue
        M = M0[i].astype(np.float64)
        fro2, sig2 = O.stable_rank_estimate(M, 5, O.power_start_vector(s[1], 0))
        want = fro2 / sig2
        assert np.isfinite(est[i]) and abs(est[i] - want) <= 1e-4 * want, (s, scale, est[i], want)
    assert opt.status() == 0
    opt.close()


@pytest.mark.parametrize("iters", [1, 2, 5])
def test_estimates_and_decisions_match_oracle(iters):
    import torch
    kinds = ["lowrank", "noise", "lowrank", "noise", "lowrank", "noise", None]
    alpha = 0.08
    opt, params, _, M0 = _state(SHAPES, kinds, 3, srank_alpha=alpha, srank_iters=iters)
    g = [torch.zeros(s, dtype=torch.bfloat16, device="cuda") for s in SHAPES]
    opt.step(g, 7)
    took, est = opt.selection()
    cfg = O.Config(schedule="stable_rank", srank_alpha=alpha, srank_iters=iters)
    for i, s in enumerate(SHAPES):
        if len(s) == 1:
            assert not took[i] and np.isnan(est[i])
            continue
        M = M0[i].astype(np.float64)
        fro2, sig2 = O.stable_rank_estimate(M, iters, O.power_start_vector(s[1], 0))
        want = fro2 / sig2
        assert abs(est[i] - want) <= 1e-4 * want, (s, est[i], want)
        thr = alpha * min(s)
        if abs(want - thr) > 1e-3 * thr:                       # decide away from the threshold only
            assert took[i] == O.srank_takes_muon(M, cfg), (s, want, thr)
    # from two passes on the low-rank buffers select Muon and the noise buffers
    # Lion at this alpha; one pass leaves the start vector mostly outside a
    # rank-2 row space, so every estimate is large and all take Lion
    want = [True, False, True, False, True, False] if iters >= 2 else [False] * 6
    assert [took[i] for i in range(6)] == want
    opt.close()


@pytest.mark.parametrize("precision", [0, 2])
def test_mixed_steps_match_oracle_fp32_ns(precision):
    """Three mixed steps from designed buffers with the fp32 NS path: each
    matrix takes the branch the rule selects on its current buffer; weights of
    Lion-selected matrices and of the vector bit-exact against the same-order
    float32 step, of Muon-selected matrices within the fp32 NS tolerance (1e-5
    CUDA cores, 2e-5 three-piece tensor cores)
    carried into W; momentum bit-exact.  (The low-rank buffers are badly
    conditioned: storing their NS intermediates in bf16 alone moves the
    output by 30-45%, so the bf16 path is checked against the plain Muon
    step instead, below.)"""
    import torch
    kinds = ["lowrank", "noise", "lowrank", "noise", "lowrank", "noise", None]
    shapes = SHAPES
    eta_M, eta_L, lam, alpha = 3e-3, 2e-5, 0.1, 0.08
    opt, params, W0, M0 = _state(shapes, kinds, 5, srank_alpha=alpha, eta_muon=eta_M, eta_lion=eta_L,
                                 weight_decay=lam, ns_precision=precision)
    r = np.random.default_rng(9)
    W = [stored_values(host_tensor(w, "bf16")).astype(np.float32) for w in W0]
    M = [m.copy() for m in M0]
    cfg = O.Config(schedule="stable_rank", srank_alpha=alpha, eta_muon=eta_M, eta_lion=eta_L, weight_decay=lam)
    n_muon = 0
    for t in range(1, 4):
        G = [stored_values(host_tensor(r.normal(size=s) * 1e-4, "bf16")).astype(np.float32) for s in shapes]
        opt.step([host_tensor(x, "bf16").cuda() for x in G], t)
        torch.cuda.synchronize()
        took, _ = opt.selection()
        for i, s in enumerate(shapes):
            if len(s) == 2:
                assert took[i] == O.srank_takes_muon(M[i].astype(np.float64), cfg)
            wg = stored_values(params[i]).astype(np.float32)
            if len(s) == 1 or not took[i]:
                w_ref, m_ref = O.lion_step_f32(W[i], G[i], M[i], 0.9, 0.99, eta_L, lam)
                np.testing.assert_array_equal(bits(params[i]), bits(torch.from_numpy(w_ref).to(torch.bfloat16)))
            else:
                n_muon += 1
                gh = O.interpolated_direction(M[i].astype(np.float64), G[i].astype(np.float64), 0.9)
                w_ref = O.round_to_storage(O.muon_update(W[i].astype(np.float64), gh, cfg), "bf16")
                o = O.ns_polynomial(gh, 5, *O.NS_QUINTIC, 1e-7)
                d = rel_fro(O.ns_polynomial_schedule_storage(gh, (O.NS_QUINTIC,) * 5, 1e-7, "f32"), o)
                tau = max(1e-5 if precision == 0 else 2e-5, 1.5 * d)
                r_w = eta_M * 0.2 * np.sqrt(max(s)) * tau * np.linalg.norm(o) / np.linalg.norm(w_ref)
                assert rel_fro(wg, w_ref) <= 1e-4 + r_w + np.sqrt(r_w * 2.0 ** -8), (s, rel_fro(wg, w_ref))
                _, m_ref = O.lion_step_f32(W[i], G[i], M[i], 0.9, 0.99, 0.0, 0.0, w_dtype="f32")
            np.testing.assert_array_equal(stored_values(opt.momentum(i)).astype(np.float32).view(np.uint32),
                                          m_ref.view(np.uint32))
            W[i] = wg
            M[i] = m_ref
    assert n_muon == 9                                   # three low-rank matrices, three steps
    assert opt.status() == 0
    opt.close()


@pytest.mark.parametrize("precision", [1, 0, 2])
def test_mixed_step_muon_matrices_equal_plain_muon_step(precision):
    """From identical weights and buffers, one mixed step (stable-rank
    schedule) and one plain Muon step (period 1): every matrix the rule sends
    to Muon ends bit-identical to the plain step's result (skipping the tiles
    of the other matrices changes nothing in the ones that run), and the rest
    bit-identical to the Lion step."""
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    kinds = ["lowrank", "noise", "lowrank", "noise", "lowrank", "noise", None]
    opt_a, pa, W0, M0 = _state(SHAPES, kinds, 11, srank_alpha=0.08, ns_precision=precision)
    pb = [host_tensor(w, "bf16").cuda() for w in W0]
    opt_b = L.LionMuon(pb, period=1, ns_precision=precision)
    for i, m in enumerate(M0):
        opt_b.set_momentum(i, torch.from_numpy(m).cuda())
    r = np.random.default_rng(12)
    G = [host_tensor(r.normal(size=s) * 1e-4, "bf16") for s in SHAPES]
    opt_a.step([g.cuda() for g in G], 4)
    opt_b.step([g.cuda() for g in G], 4)
    torch.cuda.synchronize()
    took, _ = opt_a.selection()
    assert took[:6] == [True, False, True, False, True, False]
    W = [stored_values(host_tensor(w, "bf16")).astype(np.float32) for w in W0]
    for i, s in enumerate(SHAPES):
        if took[i]:
            np.testing.assert_array_equal(bits(pa[i]), bits(pb[i]))
        else:
            w_ref, _ = O.lion_step_f32(W[i], stored_values(G[i]).astype(np.float32), M0[i], 0.9, 0.99,
                                       2e-5, 0.1)
            np.testing.assert_array_equal(bits(pa[i]), bits(torch.from_numpy(w_ref).to(torch.bfloat16)))
    assert opt_a.status() == 0 and opt_b.status() == 0
    opt_a.close()
    opt_b.close()


def test_no_matrix_selected_equals_pure_lion_steps():
    """With an alpha no buffer meets, every step is a Lion step: three mixed
    steps end bit-identical (weights and momentum) to three steps with
    period 0 (P = infinity, Algorithm 1's pure Lion reduction).  The masked
    Newton-Schulz launches then hold no selected tile anywhere, and every CTA
    pair leaves before any set-up."""
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    kinds = ["lowrank", "noise", "lowrank", "noise", "lowrank", "noise", None]
    opt_a, pa, W0, M0 = _state(SHAPES, kinds, 21, srank_alpha=1e-12)
    pb = [host_tensor(w, "bf16").cuda() for w in W0]
    opt_b = L.LionMuon(pb, period=0)
    for i, m in enumerate(M0):
        opt_b.set_momentum(i, torch.from_numpy(m).cuda())
    r = np.random.default_rng(22)
    for t in range(1, 4):
        G = [host_tensor(r.normal(size=s) * 1e-3, "bf16").cuda() for s in SHAPES]
        opt_a.step(G, t)
        opt_b.step(G, t)
        torch.cuda.synchronize()
        assert not any(opt_a.selection()[0]), t
    for i in range(len(SHAPES)):
        np.testing.assert_array_equal(bits(pa[i]), bits(pb[i]))
        assert torch.equal(opt_a.momentum(i), opt_b.momentum(i)), i
    assert opt_a.status() == 0 and opt_b.status() == 0
    opt_a.close()
    opt_b.close()


def test_zero_buffer_takes_muon_at_t0():
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    p = [torch.zeros((64, 96), dtype=torch.bfloat16, device="cuda"), torch.zeros(96, device="cuda")]
    opt = L.LionMuon(p, schedule=L.LM_SCHEDULE_STABLE_RANK)
    opt.step([torch.randn((64, 96), device="cuda").to(torch.bfloat16), torch.randn(96, device="cuda")], 0)
    took, est = opt.selection()
    assert took == [True, False] and est[0] == 0.0 and np.isnan(est[1])
    opt.close()


def test_period_schedule_reports_its_branch():
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    p = [torch.zeros((64, 96), dtype=torch.bfloat16, device="cuda"), torch.zeros(96, device="cuda")]
    opt = L.LionMuon(p, period=2)
    g = [torch.zeros((64, 96), dtype=torch.bfloat16, device="cuda"), torch.zeros(96, device="cuda")]
    with pytest.raises(L.LionMuonError):
        opt.selection()                                  # no step yet
    for t, want in [(0, True), (1, False), (2, True)]:
        opt.step(g, t)
        took, est = opt.selection()
        assert took == [want, False] and all(np.isnan(x) for x in est)
    opt.close()


def test_stable_rank_argument_errors():
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    p = [torch.zeros((32, 48), dtype=torch.bfloat16, device="cuda")]
    for bad in (dict(srank_alpha=0.0), dict(srank_iters=0), dict(srank_iters=65), dict(schedule=2)):
        kw = dict(schedule=L.LM_SCHEDULE_STABLE_RANK)
        kw.update(bad)
        with pytest.raises(L.LionMuonError) as e:
            L.LionMuon(p, **kw)
        assert e.value.status == 1
    wide = [torch.zeros((2, 16400), dtype=torch.bfloat16, device="cuda")]
    with pytest.raises(L.LionMuonError) as e:
        L.LionMuon(wide, schedule=L.LM_SCHEDULE_STABLE_RANK)
    assert e.value.status == 6                           # LM_ERR_UNSUPPORTED


def test_stable_rank_schedule_with_adamw_vectors():
    """Both options together: matrices take the branch the rule selects (Lion
    ones bit-exact), the vector takes AdamW (bit-exact against the same-order
    float32 AdamW step with its update count t + 1), momentum bit-exact."""
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    kinds = ["lowrank", "noise", "lowrank", "noise", "lowrank", "noise", None]
    opt, params, W0, M0 = _state(SHAPES, kinds, 21, srank_alpha=0.08, vector_rule=L.LM_VECTOR_ADAMW)
    r = np.random.default_rng(22)
    W = [stored_values(host_tensor(w, "bf16")).astype(np.float32) for w in W0]
    M = [m.copy() for m in M0]
    V = np.zeros(SHAPES[-1], np.float32)
    cfg = O.Config(schedule="stable_rank", srank_alpha=0.08)
    for t in (3, 4):
        G = [stored_values(host_tensor(r.normal(size=s) * 1e-4, "bf16")).astype(np.float32) for s in SHAPES]
        opt.step([host_tensor(x, "bf16").cuda() for x in G], t)
        torch.cuda.synchronize()
        took, _ = opt.selection()
        assert took[:6] == [True, False, True, False, True, False]
        for i, s in enumerate(SHAPES):
            if len(s) == 1:
                w_ref, m_ref, V = O.adamw_step_f32(W[i], G[i], M[i], V, t + 1, 1e-3, 0.8, 0.999, 1e-8, 0.1)
                np.testing.assert_array_equal(bits(params[i]), bits(torch.from_numpy(w_ref).to(torch.bfloat16)))
                np.testing.assert_array_equal(stored_values(opt.second_moment(i)).astype(np.float32).view(np.uint32),
                                              V.view(np.uint32))
            elif not took[i]:
                w_ref, m_ref = O.lion_step_f32(W[i], G[i], M[i], 0.9, 0.99, 2e-5, 0.1)
                np.testing.assert_array_equal(bits(params[i]), bits(torch.from_numpy(w_ref).to(torch.bfloat16)))
            else:
                _, m_ref = O.lion_step_f32(W[i], G[i], M[i], 0.9, 0.99, 0.0, 0.0, w_dtype="f32")
                assert O.srank_takes_muon(M[i].astype(np.float64), cfg)
            np.testing.assert_array_equal(stored_values(opt.momentum(i)).astype(np.float32).view(np.uint32),
                                          m_ref.view(np.uint32))
            W[i] = stored_values(params[i]).astype(np.float32)
            M[i] = m_ref
    assert opt.status() == 0
    opt.close()
