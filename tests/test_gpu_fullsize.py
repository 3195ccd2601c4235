"""Full-size parity on the 720M-shaped parameter set (772 M parameters), in
the launch configuration bench.py times: one Muon step (t = 0) and one Lion
step (t = 1), checked on sampled outputs the oracle computes directly:

* momentum and Lion-step weights of sampled tensors bit-exact against the
  same-order float32 oracle;
* the Muon direction of one matrix of each hidden shape (wide, square, tall)
  against the fp64 NS recurrence within the NS tolerance;
* for the 50304 x 1280 embedding, a property that holds at any size: the
  singular values of the direction equal phi^5(sigma_i(G_hat)/||G_hat||_F)
  (phi the quintic map), compared from the two 1280 x 1280 Gram spectra."""

import math

import numpy as np
import pytest

import oracle as O
from paper_2605_19811_gb300 import synth
from tests.lm_testutil import bits, rel_fro

pytestmark = pytest.mark.gpu

NS_TOL = 2e-2


def _host(t):
    return t.detach().float().cpu().numpy()


def test_720m_muon_then_lion_sampled():
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    ps = synth.PARAM_SETS["gpt_720m"]
    shapes = [tuple(s) for s in ps.shapes]
    dev = torch.device("cuda", 0)
    params = synth.device_weights_torch(shapes, seed=1, device=dev, dtype=torch.bfloat16)
    g0 = synth.device_grads_torch(shapes, "student_t", seed=10, device=dev, dtype=torch.bfloat16)
    g1 = synth.device_grads_torch(shapes, "student_t", seed=11, device=dev, dtype=torch.bfloat16)

    def first(shape):
        return next(i for i, s in enumerate(shapes) if s == shape)
    emb = first((50304, 1280))
    mats = [first((1280, 1280)), first((1280, 3840)), first((1280, 5120)), first((5120, 1280))]
    vec = first((1280,))
    sample = mats + [emb, vec]
    W0 = {i: _host(params[i]) for i in sample}
    G0 = {i: _host(g0[i]) for i in sample}
    G1 = {i: _host(g1[i]) for i in sample}

    eta_M, eta_L, lam = 1.0, 1e-3, 0.0        # a large Muon step exposes the direction
    opt = L.LionMuon(params, period=2, eta_muon=eta_M, eta_lion=eta_L, weight_decay=lam)
    opt.step(g0, 0)
    torch.cuda.synchronize()
    W1 = {i: _host(params[i]) for i in sample}
    M1 = {i: _host(opt.momentum(i)) for i in sample}

    # momentum after the first step: fl(c2 * g) from M = 0 (bit-exact)
    for i in sample:
        _, m_ref = O.lion_step_f32(np.zeros_like(G0[i]), G0[i], np.zeros_like(G0[i]), 0.9, 0.99, 0.0, 0.0,
                                   w_dtype="f32")
        np.testing.assert_array_equal(M1[i].view(np.uint32), m_ref.view(np.uint32))
    # the vector took the Lion step
    w_ref, _ = O.lion_step_f32(W0[vec], G0[vec], np.zeros_like(G0[vec]), 0.9, 0.99, eta_L, lam)
    np.testing.assert_array_equal(bits(torch.from_numpy(W1[vec]).to(torch.bfloat16)),
                                  bits(torch.from_numpy(w_ref).to(torch.bfloat16)))
    # Muon directions of the sampled hidden matrices
    for i in mats:
        s = 0.2 * math.sqrt(max(shapes[i]))
        o_gpu = (W0[i].astype(np.float64) - W1[i].astype(np.float64)) / (eta_M * s)
        o_ref = O.ns_polynomial(0.1 * G0[i].astype(np.float64), 5, *O.NS_QUINTIC, 1e-7)
        # W1 is stored in bf16: its rounding adds up to 2^-9 |W1| / (eta s)
        slack = 2.0 ** -9 * np.linalg.norm(W1[i]) / (eta_M * s) / np.linalg.norm(o_ref)
        assert rel_fro(o_gpu, o_ref) <= NS_TOL + slack, (shapes[i], rel_fro(o_gpu, o_ref))
    # embedding: spectrum of the direction vs the scalar map of G_hat's spectrum
    s = 0.2 * math.sqrt(50304)
    o_emb = (W0[emb].astype(np.float64) - W1[emb].astype(np.float64)) / (eta_M * s)
    gh = 0.1 * G0[emb].astype(np.float64)
    sig_g = np.sqrt(np.clip(np.linalg.eigvalsh(gh.T @ gh), 0, None))
    sig_o = np.sqrt(np.clip(np.linalg.eigvalsh(o_emb.T @ o_emb), 0, None))
    want = np.sort(O.ns_scalar_map(sig_g / (np.linalg.norm(sig_g) + 1e-7), 5, *O.NS_QUINTIC))
    slack = 2.0 ** -9 * np.linalg.norm(W1[emb]) / (eta_M * s) / np.linalg.norm(want)
    assert np.linalg.norm(np.sort(sig_o) - want) / np.linalg.norm(want) <= NS_TOL + slack

    # t = 1 is a Lion step for every parameter: bit-exact on the samples
    opt.step(g1, 1)
    torch.cuda.synchronize()
    for i in sample:
        w_ref, m_ref = O.lion_step_f32(W1[i], G1[i], M1[i], 0.9, 0.99, eta_L, lam)
        np.testing.assert_array_equal(bits(params[i]), bits(torch.from_numpy(w_ref).to(torch.bfloat16)))
        np.testing.assert_array_equal(_host(opt.momentum(i)).view(np.uint32), m_ref.view(np.uint32))
    assert opt.status() == 0
    opt.close()


def _muon_then_lion(set_name, period, check_shapes, spectrum_shape=None):
    """One Muon step (t = 0) and one Lion step (t = 1, or t = period - 1 when
    that is not a Muon step) of a whole parameter set in the bench's
    configuration; sampled checks as in the 720M test above."""
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    ps = synth.PARAM_SETS[set_name]
    shapes = [tuple(s) for s in ps.shapes]
    dev = torch.device("cuda", 0)
    params = synth.device_weights_torch(shapes, seed=1, device=dev, dtype=torch.bfloat16)
    g0 = synth.device_grads_torch(shapes, ps.grad_kind, seed=10, device=dev, dtype=torch.bfloat16)
    idx = {s: next(i for i, x in enumerate(shapes) if x == s) for s in check_shapes}
    vecs = [i for i, s in enumerate(shapes) if len(s) == 1][:1]
    sample = list(idx.values()) + vecs + ([shapes.index(spectrum_shape)] if spectrum_shape else [])
    W0 = {i: _host(params[i]) for i in sample}
    G0 = {i: _host(g0[i]) for i in sample}
    eta_M, eta_L, lam = 1.0, 1e-3, 0.0
    opt = L.LionMuon(params, period=period, eta_muon=eta_M, eta_lion=eta_L, weight_decay=lam)
    opt.step(g0, 0)
    torch.cuda.synchronize()
    W1 = {i: _host(params[i]) for i in sample}
    M1 = {i: _host(opt.momentum(i)) for i in sample}
    for i in sample:
        _, m_ref = O.lion_step_f32(np.zeros_like(G0[i]), G0[i], np.zeros_like(G0[i]), 0.9, 0.99, 0.0, 0.0,
                                   w_dtype="f32")
        np.testing.assert_array_equal(M1[i].view(np.uint32), m_ref.view(np.uint32))
    for i in vecs:
        w_ref, _ = O.lion_step_f32(W0[i], G0[i], np.zeros_like(G0[i]), 0.9, 0.99, eta_L, lam)
        np.testing.assert_array_equal(bits(torch.from_numpy(W1[i]).to(torch.bfloat16)),
                                      bits(torch.from_numpy(w_ref).to(torch.bfloat16)))
    for shp, i in idx.items():
        s = 0.2 * math.sqrt(max(shp))
        o_gpu = (W0[i].astype(np.float64) - W1[i].astype(np.float64)) / (eta_M * s)
        o_ref = O.ns_polynomial(0.1 * G0[i].astype(np.float64), 5, *O.NS_QUINTIC, 1e-7)
        slack = 2.0 ** -9 * np.linalg.norm(W1[i]) / (eta_M * s) / np.linalg.norm(o_ref)
        assert rel_fro(o_gpu, o_ref) <= NS_TOL + slack, (set_name, shp, rel_fro(o_gpu, o_ref))
    if spectrum_shape:
        i = shapes.index(spectrum_shape)
        s = 0.2 * math.sqrt(max(spectrum_shape))
        o = (W0[i].astype(np.float64) - W1[i].astype(np.float64)) / (eta_M * s)
        gh = 0.1 * G0[i].astype(np.float64)
        sig_g = np.sqrt(np.clip(np.linalg.eigvalsh(gh.T @ gh), 0, None))
        sig_o = np.sqrt(np.clip(np.linalg.eigvalsh(o.T @ o), 0, None))
        want = np.sort(O.ns_scalar_map(sig_g / (np.linalg.norm(sig_g) + 1e-7), 5, *O.NS_QUINTIC))
        slack = 2.0 ** -9 * np.linalg.norm(W1[i]) / (eta_M * s) / np.linalg.norm(want)
        assert np.linalg.norm(np.sort(sig_o) - want) / np.linalg.norm(want) <= NS_TOL + slack
    # a Lion step for every parameter: bit-exact on the samples
    t1 = 1 if period != 1 else None
    if t1 is not None:
        g1 = synth.device_grads_torch(shapes, ps.grad_kind, seed=11, device=dev, dtype=torch.bfloat16)
        G1 = {i: _host(g1[i]) for i in sample}
        opt.step(g1, t1)
        torch.cuda.synchronize()
        for i in sample:
            w_ref, m_ref = O.lion_step_f32(W1[i], G1[i], M1[i], 0.9, 0.99, eta_L, lam)
            np.testing.assert_array_equal(bits(params[i]), bits(torch.from_numpy(w_ref).to(torch.bfloat16)))
            np.testing.assert_array_equal(_host(opt.momentum(i)).view(np.uint32), m_ref.view(np.uint32))
        del g1
    assert opt.status() == 0
    opt.close()
    del params, g0
    torch.cuda.empty_cache()


def test_124m_muon_then_lion_sampled():
    _muon_then_lion("gpt2_124m", 2, [(768, 2304), (768, 768), (3072, 768)], spectrum_shape=(50304, 768))


@pytest.mark.parametrize("period", [1, 4])
def test_355m_muon_then_lion_sampled(period):
    _muon_then_lion("gpt_355m", period, [(1024, 3072), (4096, 1024)])


def test_stress_7b_muon_then_lion_sampled():
    """The 7B-style stress set (7.79 G parameters, outlier gradients, P = 8):
    the Muon direction of a 4096 x 4096 and a 14336 x 4096 matrix against the
    fp64 recurrence, the Lion step bit-exact."""
    _muon_then_lion("stress_7b", 8, [(4096, 4096), (14336, 4096)])


def test_720m_three_piece_fp32_mode_directions_sampled():
    """The 720M-shaped set with ns_precision = LM_NS_F32_TC and fp32
    parameters and gradients (so that W's storage does not hide the NS
    error): the Muon
    direction of one matrix of each hidden shape against the fp64 recurrence
    within the three-piece tolerance 5e-5, and the embedding's singular values
    against the scalar map, after one Muon step of the whole set."""
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    tol = 5e-5
    ps = synth.PARAM_SETS["gpt_720m"]
    shapes = [tuple(s) for s in ps.shapes]
    dev = torch.device("cuda", 0)
    params = synth.device_weights_torch(shapes, seed=1, device=dev, dtype=torch.float32)
    g0 = synth.device_grads_torch(shapes, "student_t", seed=10, device=dev, dtype=torch.float32)

    def first(shape):
        return next(i for i, s in enumerate(shapes) if s == shape)
    emb = first((50304, 1280))
    mats = [first((1280, 1280)), first((1280, 3840)), first((1280, 5120)), first((5120, 1280))]
    sample = mats + [emb]
    W0 = {i: _host(params[i]) for i in sample}
    G0 = {i: _host(g0[i]) for i in sample}
    eta_M = 1.0
    opt = L.LionMuon(params, period=1, eta_muon=eta_M, eta_lion=1e-3, weight_decay=0.0,
                     ns_precision=L.LM_NS_F32_TC)
    opt.step(g0, 0)
    torch.cuda.synchronize()
    W1 = {i: _host(params[i]) for i in sample}
    for i in mats:
        s = 0.2 * math.sqrt(max(shapes[i]))
        o_gpu = (W0[i].astype(np.float64) - W1[i].astype(np.float64)) / (eta_M * s)
        o_ref = O.ns_polynomial(0.1 * G0[i].astype(np.float64), 5, *O.NS_QUINTIC, 1e-7)
        # fp32 W: its rounding adds up to 2^-24 (|W0| + |W1|) / (eta s)
        slack = 2.0 ** -24 * (np.linalg.norm(W0[i]) + np.linalg.norm(W1[i])) / (eta_M * s) / np.linalg.norm(o_ref)
        assert rel_fro(o_gpu, o_ref) <= tol + slack, (shapes[i], rel_fro(o_gpu, o_ref))
    s = 0.2 * math.sqrt(50304)
    o_emb = (W0[emb].astype(np.float64) - W1[emb].astype(np.float64)) / (eta_M * s)
    gh = 0.1 * G0[emb].astype(np.float64)
    sig_g = np.sqrt(np.clip(np.linalg.eigvalsh(gh.T @ gh), 0, None))
    sig_o = np.sqrt(np.clip(np.linalg.eigvalsh(o_emb.T @ o_emb), 0, None))
    want = np.sort(O.ns_scalar_map(sig_g / (np.linalg.norm(sig_g) + 1e-7), 5, *O.NS_QUINTIC))
    slack = 2.0 ** -24 * (np.linalg.norm(W0[emb]) + np.linalg.norm(W1[emb])) / (eta_M * s) / np.linalg.norm(want)
    assert np.linalg.norm(np.sort(sig_o) - want) / np.linalg.norm(want) <= tol + slack
    assert opt.status() == 0
    opt.close()
    del params, g0
    torch.cuda.empty_cache()
