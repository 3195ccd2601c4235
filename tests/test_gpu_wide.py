"""GPU tests of the two-block (256 x 512) tile kernel and of programmatic
dependent launch between the Newton-Schulz launches.

A two-block tile issues, per K step, the same N = 256 MMAs over the same K
order as two one-block tiles, and its epilogue applies the same fp32 formula,
so every result must equal the one-block kernel's bit for bit:
msign outputs of wide, tall, square and ragged shapes, whole Muon + Lion steps
(momentum, parameters through the fused parameter write), the stable-rank
schedule's masked launches and split-K Gram tiles.  The two-block results are
also checked against the fp64 oracle recurrence (Section 2's iteration) at
the bf16 tolerance, 2e-2.  LM_NS_TILES chooses the tiles and LM_PDL=0 turns
programmatic launch off; both are read when a state is created or an msign
call starts.  The two-block kernel keeps a X as a separate term of APPLY, so
these tests run the one-block kernel with LM_NS_FOLD=0 as well (the folded
form is checked against the oracle elsewhere)."""

import numpy as np
import pytest

import oracle as O
from paper_2605_19811_gb300 import synth
from tests.lm_testutil import bits, host_tensor, rel_fro, stored_values

pytestmark = pytest.mark.gpu

QUINTIC = O.NS_QUINTIC


@pytest.fixture(autouse=True)
def _unfolded(monkeypatch):
    monkeypatch.setenv("LM_NS_FOLD", "0")


def _msign_bf16(xh, steps=5, coeffs=QUINTIC):
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    x = xh.cuda()
    out = torch.empty(x.shape, dtype=torch.float32, device="cuda")
    L.msign_ns(x, out, steps, *coeffs, eps=1e-7, precision=L.LM_BF16)
    torch.cuda.synchronize()
    return out.cpu()


# s_pad with an even and an odd number of 256 blocks, s_pad not a multiple of
# 256 (the last block half padding), wide and tall, a one-block matrix
@pytest.mark.parametrize("shape", [(640, 1536), (1536, 640), (1280, 1280), (896, 2000), (2000, 896),
                                   (768, 3072), (3072, 768), (1000, 130), (256, 4096)])
def test_wide_msign_bit_identical_and_oracle(shape, monkeypatch):
    xh = host_tensor(synth.draw_matrix(shape, seed=11 + shape[0]), "bf16")
    monkeypatch.setenv("LM_NS_TILES", "narrow")
    narrow = _msign_bf16(xh)
    monkeypatch.setenv("LM_NS_TILES", "wide")
    wide = _msign_bf16(xh)
    np.testing.assert_array_equal(bits(wide), bits(narrow))
    want = O.ns_polynomial(stored_values(xh), 5, *QUINTIC, 1e-7)
    assert rel_fro(stored_values(wide), want) <= 2e-2


@pytest.mark.parametrize("coeffs,steps", [((0.0, 1.0, 0.0), 1), ((0.0, 0.0, 1.0), 1), (QUINTIC, 2)])
def test_wide_msign_each_term(coeffs, steps, monkeypatch):
    """(0,1,0) isolates the Gram and apply products, (0,0,1) the polynomial one."""
    xh = host_tensor(synth.draw_matrix((768, 2048), seed=5), "bf16")
    monkeypatch.setenv("LM_NS_TILES", "wide")
    got = stored_values(_msign_bf16(xh, steps, coeffs))
    want = O.ns_polynomial(stored_values(xh), steps, *coeffs, 1e-7)
    assert rel_fro(got, want) <= 2e-2


def _run_steps(shapes, env, monkeypatch, steps=2, **cfg):
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    for k, v in env.items():
        monkeypatch.setenv(k, v)
    W0 = synth.init_weights(shapes, seed=1)
    params = [host_tensor(w, "bf16").cuda() for w in W0]
    opt = L.LionMuon(params, **cfg)
    for t in range(steps):
        g = [host_tensor(x, "bf16").cuda() for x in synth.draw_grads(shapes, "student_t", seed=0, step=t)]
        opt.step(g, t)
    torch.cuda.synchronize()
    out = [bits(p) for p in params] + [bits(opt.momentum(i)) for i in range(len(params))]
    flags = opt.status()
    opt.close()
    for k in env:
        monkeypatch.delenv(k)
    return out, flags


GPT2L = synth.scaled_set("gpt_2l", layers=2, d=768, vocab=4096)


def test_wide_steps_bit_identical_to_narrow(monkeypatch):
    """Muon step (t = 0, parameter write fused into the last APPLY) and Lion
    step on a 2-layer d = 768 GPT-style set with a 4096 x 768 embedding."""
    a, fa = _run_steps(GPT2L.shapes, {"LM_NS_TILES": "narrow"}, monkeypatch, period=2)
    b, fb = _run_steps(GPT2L.shapes, {"LM_NS_TILES": "wide"}, monkeypatch, period=2)
    assert fa == 0 and fb == 0
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)


def test_pdl_off_bit_identical(monkeypatch):
    a, _ = _run_steps(GPT2L.shapes, {"LM_PDL": "0"}, monkeypatch, steps=3, period=1)
    b, _ = _run_steps(GPT2L.shapes, {}, monkeypatch, steps=3, period=1)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)


def test_wide_masked_steps_bit_identical(monkeypatch):
    """Stable-rank schedule (Appendix G): the masked instantiations."""
    cfg = dict(schedule=1, srank_alpha=0.5)
    a, _ = _run_steps(GPT2L.shapes, {"LM_NS_TILES": "narrow"}, monkeypatch, steps=3, **cfg)
    b, _ = _run_steps(GPT2L.shapes, {"LM_NS_TILES": "wide"}, monkeypatch, steps=3, **cfg)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)


def test_wide_split_gram_tiles(monkeypatch):
    """A 20000-long Gram next to short ones is split along K; a two-block
    tile that qualifies is split per block, with the same parts as before."""
    shapes = [(768, 768), (768, 768), (20000, 768), (768,)]
    a, _ = _run_steps(shapes, {"LM_NS_TILES": "narrow"}, monkeypatch, steps=1, period=1)
    b, _ = _run_steps(shapes, {"LM_NS_TILES": "wide"}, monkeypatch, steps=1, period=1)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)


def test_default_tile_choice_matches_oracle():
    """Eight 1280 x 5120 matrices: with the default choice the APPLY launches
    (800 one-block tiles for 76 CTA pairs) run two-block tiles and the Gram and
    polynomial launches (120 tiles) one-block tiles.  The Muon direction read
    back from the parameters matches the oracle's NS(G_hat)."""
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    shapes = [(1280, 5120)] * 8
    W0 = synth.init_weights(shapes, seed=1)
    params = [host_tensor(w, "bf16").cuda() for w in W0]
    g = [host_tensor(x, "bf16") for x in synth.draw_grads(shapes, "student_t", seed=0, step=0)]
    opt = L.LionMuon(params, period=1, weight_decay=0.0, eta_muon=1.0)
    opt.step([x.cuda() for x in g], 0)
    torch.cuda.synchronize()
    assert opt.status() == 0
    for k in (0, 7):
        w1 = stored_values(params[k])
        d = (stored_values(host_tensor(W0[k], "bf16")) - w1) / (0.2 * np.sqrt(5120))
        gh = 0.1 * stored_values(g[k])     # M_{-1} = 0: G_hat = (1 - beta1) G
        want = O.ns_polynomial(gh, 5, *QUINTIC, 1e-7)
        # W1 is stored in bf16: its rounding moves d by at most 2^-9 |W1| / s per entry
        scale = 0.2 * np.sqrt(5120)
        assert rel_fro(d, want) <= 2e-2 + 2 ** -9 * np.linalg.norm(w1) / (scale * np.linalg.norm(want))
    opt.close()
