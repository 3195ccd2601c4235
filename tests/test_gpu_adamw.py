"""GPU parity of the AdamW rule for 1-D parameters (LM_VECTOR_ADAMW, the
fallback Section 3 gives biases and norm gains): bit-exact against the
oracle's same-order float32 AdamW step on Lion and Muon steps, bf16 and fp32
parameters, ragged lengths; matrices untouched by the choice; the extra
state, checkpoint/resume of both moments, the learning-rate setter and the
argument errors."""

import numpy as np
import pytest

import oracle as O
from tests.lm_testutil import bits, host_tensor, make_problem, stored_values

pytestmark = pytest.mark.gpu

LR, B1, B2, EPS, WD = 1e-3, 0.8, 0.999, 1e-8, 0.1
SHAPES = [(96, 200), (200,), (37,), (1, 300), (257, 1), (64, 64)]


def _vec(shape):
    return not O.is_matrix(shape)


def _run(W0, grads, dtype, steps, rule, lr_at=None, **cfg):
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    params = [host_tensor(w, dtype).cuda() for w in W0]
    opt = L.LionMuon(params, period=2, vector_rule=rule, **cfg)
    hist = []
    for t in range(steps):
        if lr_at is not None and t == lr_at[0]:
            opt.set_adamw_lr(lr_at[1])
        opt.step([host_tensor(g, dtype).cuda() for g in grads[t]], t)
        torch.cuda.synchronize()
        snap = {"w": [stored_values(p).astype(np.float32) for p in params],
                "m": [stored_values(opt.momentum(i)).astype(np.float32) for i in range(len(params))]}
        if rule == L.LM_VECTOR_ADAMW:
            snap["v"] = {i: stored_values(opt.second_moment(i)).astype(np.float32)
                         for i, p in enumerate(params) if _vec(tuple(p.shape))}
        hist.append(snap)
    flags = opt.status()
    nbytes = opt.state_bytes()
    opt.close()
    return hist, flags, nbytes


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_adamw_vectors_bit_exact_on_lion_and_muon_steps(dtype):
    from paper_2605_19811_gb300 import lionmuon as L
    steps = 6
    W0, grads = make_problem(SHAPES, "student_t", steps)
    hist, flags, _ = _run(W0, grads, dtype, steps, L.LM_VECTOR_ADAMW)
    assert flags == 0
    for i, shp in enumerate(SHAPES):
        if not _vec(shp):
            continue
        w = stored_values(host_tensor(W0[i], dtype)).astype(np.float32)
        m = np.zeros(shp, np.float32)
        v = np.zeros(shp, np.float32)
        for t in range(steps):
            g = stored_values(host_tensor(grads[t][i], dtype)).astype(np.float32)
            w, m, v = O.adamw_step_f32(w, g, m, v, t + 1, LR, B1, B2, EPS, WD, w_dtype=dtype)
            np.testing.assert_array_equal(hist[t]["w"][i].view(np.uint32), w.view(np.uint32))
            np.testing.assert_array_equal(hist[t]["m"][i].view(np.uint32), m.view(np.uint32))
            np.testing.assert_array_equal(hist[t]["v"][i].view(np.uint32), v.view(np.uint32))


def test_matrices_do_not_depend_on_the_vector_rule():
    from paper_2605_19811_gb300 import lionmuon as L
    steps = 4
    W0, grads = make_problem(SHAPES, "student_t", steps)
    ha, _, bytes_a = _run(W0, grads, "bf16", steps, L.LM_VECTOR_ADAMW)
    hl, _, bytes_l = _run(W0, grads, "bf16", steps, L.LM_VECTOR_LION)
    for i, shp in enumerate(SHAPES):
        if _vec(shp):
            continue
        for t in range(steps):
            np.testing.assert_array_equal(ha[t]["w"][i].view(np.uint32), hl[t]["w"][i].view(np.uint32))
    n_all = sum(int(np.prod(s)) for s in SHAPES)
    n_vec = sum(int(np.prod(s)) for s in SHAPES if _vec(s))
    assert bytes_l == 4 * n_all
    assert bytes_a == 4 * (n_all + n_vec)


def test_adamw_learning_rate_setter():
    from paper_2605_19811_gb300 import lionmuon as L
    steps = 4
    shapes = [(300,)]
    W0, grads = make_problem(shapes, "student_t", steps)
    hist, _, _ = _run(W0, grads, "f32", steps, L.LM_VECTOR_ADAMW, lr_at=(2, 5e-4))
    w = W0[0].astype(np.float32)
    m = np.zeros(300, np.float32)
    v = np.zeros(300, np.float32)
    for t in range(steps):
        lr = LR if t < 2 else 5e-4
        g = grads[t][0].astype(np.float32)
        w, m, v = O.adamw_step_f32(w, g, m, v, t + 1, lr, B1, B2, EPS, WD, w_dtype="f32")
    np.testing.assert_array_equal(hist[-1]["w"][0].view(np.uint32), w.view(np.uint32))


def test_resume_from_both_moments_is_bit_identical():
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    steps = 6
    W0, grads = make_problem(SHAPES, "student_t", steps)
    dev = lambda a: host_tensor(a, "bf16").cuda()
    ref = [dev(w) for w in W0]
    opt = L.LionMuon(ref, period=2, vector_rule=L.LM_VECTOR_ADAMW)
    for t in range(3):
        opt.step([dev(g) for g in grads[t]], t)
    torch.cuda.synchronize()
    saved_w = [p.clone() for p in ref]
    saved_m = [opt.momentum(i).clone() for i in range(len(ref))]
    saved_v = {i: opt.second_moment(i).clone() for i, s in enumerate(SHAPES) if _vec(s)}
    for t in range(3, steps):
        opt.step([dev(g) for g in grads[t]], t)
    torch.cuda.synchronize()
    opt.close()

    res = [w.clone() for w in saved_w]
    opt2 = L.LionMuon(res, period=2, vector_rule=L.LM_VECTOR_ADAMW)
    for i in range(len(res)):
        opt2.set_momentum(i, saved_m[i])
    for i, v in saved_v.items():
        opt2.set_second_moment(i, v)
    for t in range(3, steps):
        opt2.step([dev(g) for g in grads[t]], t)
    torch.cuda.synchronize()
    for a, b in zip(ref, res):
        np.testing.assert_array_equal(bits(a), bits(b))
    opt2.close()


def test_adamw_argument_errors():
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    p = [torch.zeros((32, 48), dtype=torch.bfloat16, device="cuda"), torch.zeros(48, device="cuda")]
    with pytest.raises(L.LionMuonError) as e:
        L.LionMuon(p, vector_rule=L.LM_VECTOR_ADAMW, adamw_eps=0.0)
    assert e.value.status == 1
    with pytest.raises(L.LionMuonError):
        L.LionMuon(p, vector_rule=2)
    opt = L.LionMuon(p, vector_rule=L.LM_VECTOR_ADAMW)
    with pytest.raises(L.LionMuonError):
        opt.second_moment(0)                 # a matrix has no second moment
    with pytest.raises(L.LionMuonError):
        opt.set_adamw_lr(float("nan"))
    opt.close()
    opt = L.LionMuon(p)                      # Lion rule: no second moments at all
    with pytest.raises(L.LionMuonError):
        opt.second_moment(1)
    opt.close()
