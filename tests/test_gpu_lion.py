"""GPU parity of the Lion step (Algorithm 1, Lion branch + momentum update):
bit-exact against the same-order float32 oracle, including bf16
round-to-nearest-even, ragged tails, empty tensors and sign ties."""

import numpy as np
import pytest

import oracle as O
from paper_2605_19811_gb300 import synth
from tests.lm_testutil import bits, host_tensor, stored_values

pytestmark = pytest.mark.gpu

SHAPES = [(300, 7), (1,), (5,), (1023,), (64, 64), (17, 33), (0,), (3, 40001), (8,), (129,)]


def _lion_run(dtype, shapes, steps, beta1=0.9, beta2=0.99, eta=0.02, lam=0.1, tie_prefix=16,
              grad_kind="normal"):
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    W0 = synth.init_weights(shapes, seed=3)
    params = [host_tensor(w, dtype).cuda() for w in W0]
    ref_w = [host_tensor(w, dtype).float().numpy() for w in W0]
    ref_m = [np.zeros(s, dtype=np.float32) for s in shapes]
    opt = L.LionMuon(params, beta1=beta1, beta2=beta2, eta_lion=eta, weight_decay=lam, period=0)
    for t in range(steps):
        G = synth.draw_grads(shapes, grad_kind, seed=11, step=t)
        for g in G:
            g.reshape(-1)[:tie_prefix] = 0.0      # with M = 0 at t = 0: G_hat == 0 exactly
        gh = [host_tensor(g, dtype) for g in G]
        opt.step([g.cuda() for g in gh], t)
        for i in range(len(shapes)):
            ref_w[i], ref_m[i] = O.lion_step_f32(ref_w[i], gh[i].float().numpy(), ref_m[i],
                                                 beta1, beta2, eta, lam, w_dtype=dtype)
    torch.cuda.synchronize()
    out = []
    for i in range(len(shapes)):
        out.append((params[i].cpu(), opt.momentum(i).cpu(), ref_w[i], ref_m[i]))
    opt.close()
    return out


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_lion_bit_exact(dtype):
    import torch
    for gw, gm, rw, rm in _lion_run(dtype, SHAPES, steps=4):
        want_w = torch.from_numpy(np.ascontiguousarray(rw)).to(gw.dtype)
        np.testing.assert_array_equal(bits(gw), bits(want_w))
        np.testing.assert_array_equal(bits(gm), np.ascontiguousarray(rm).view(np.uint32))


def test_lion_bit_exact_heavy_tailed_bf16():
    import torch
    shapes = [(768, 2304), (768,), (3072, 768)]
    for gw, gm, rw, rm in _lion_run("bf16", shapes, steps=3, eta=2e-5, grad_kind="student_t"):
        want_w = torch.from_numpy(np.ascontiguousarray(rw)).to(gw.dtype)
        np.testing.assert_array_equal(bits(gw), bits(want_w))
        np.testing.assert_array_equal(bits(gm), np.ascontiguousarray(rm).view(np.uint32))


def test_lion_sign_ties_and_magnitude():
    """Where G_hat == 0 the step is pure decay; elsewhere |dW| = eta (f32)."""
    shapes = [(4096,)]
    (gw, gm, rw, rm), = _lion_run("f32", shapes, steps=1, eta=0.25, lam=0.0, tie_prefix=100)
    W0 = synth.init_weights(shapes, seed=3)[0]
    d = gw.numpy().astype(np.float64) - W0.astype(np.float64)
    assert np.all(d[:100] == 0.0)
    np.testing.assert_allclose(np.abs(d[100:]), 0.25, rtol=1e-6)


def test_lion_nan_propagates():
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    w = torch.zeros(64, device="cuda")
    g = torch.ones(64, device="cuda")
    g[3] = float("nan")
    opt = L.LionMuon([w], eta_lion=0.1, weight_decay=0.0, period=0)
    opt.step([g], 0)
    torch.cuda.synchronize()
    out = w.cpu().numpy()
    assert np.isnan(out[3]) and np.all(out[np.arange(64) != 3] == -0.1)
    opt.close()


def test_lion_large_vector_sampled():
    """A 40M-element bf16 vector (several thousand work chunks): sampled
    elements bit-exact against the same-order oracle."""
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    n = 40_000_003
    gen = torch.Generator().manual_seed(5)
    w = (torch.randn(n, generator=gen) * 0.02).to(torch.bfloat16)
    g = (torch.randn(n, generator=gen) * 1e-3).to(torch.bfloat16)
    m = (torch.randn(n, generator=gen) * 1e-3)
    wd, gd = w.cuda(), g.cuda()
    opt = L.LionMuon([wd], eta_lion=2e-5, weight_decay=0.1, period=0)
    opt.set_momentum(0, m.cuda())
    opt.step([gd], 1)
    torch.cuda.synchronize()
    idx = np.unique(np.concatenate([np.random.default_rng(0).integers(0, n, 200000),
                                    np.arange(n - 64, n)]))
    rw, rm = O.lion_step_f32(w.float().numpy()[idx], g.float().numpy()[idx], m.numpy()[idx],
                             0.9, 0.99, 2e-5, 0.1, w_dtype="bf16")
    got_w = wd.cpu()[idx]
    got_m = opt.momentum(0).cpu().numpy()[idx]
    np.testing.assert_array_equal(bits(got_w), bits(torch.from_numpy(rw).to(torch.bfloat16)))
    np.testing.assert_array_equal(got_m.view(np.uint32), rm.view(np.uint32))
    opt.close()
