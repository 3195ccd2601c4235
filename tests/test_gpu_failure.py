"""Failure detection on the GPU without a fault: a bounded device-side wait
on a barrier that nothing signals gives up, reports LM_FLAG_TIMEOUT through
the status word, and leaves the context usable for further work."""

import time

import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def test_bounded_wait_gives_up_and_context_survives():
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    t0 = time.perf_counter()
    st, flags = L.probe_bounded_wait(20_000_000)       # 20 ms
    dt = time.perf_counter() - t0
    assert st == 7                                       # LM_ERR_TIMEOUT
    assert flags & L.LM_FLAG_TIMEOUT
    assert dt < 5.0
    # the context still runs kernels correctly afterwards
    x = torch.randn(96, 160, device="cuda")
    out = torch.empty_like(x)
    L.msign_ns(x, out, precision=L.LM_F32)
    torch.cuda.synchronize()
    assert bool(torch.isfinite(out).all())


def test_probe_rejects_bad_arguments():
    from paper_2605_19811_gb300 import lionmuon as L
    st, _ = L.probe_bounded_wait(0)
    assert st == 1


def test_step_status_clean_after_normal_work():
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    p = [torch.zeros((256, 384), dtype=torch.bfloat16, device="cuda"), torch.zeros(384, device="cuda")]
    opt = L.LionMuon(p, period=2)
    g = [torch.randn((256, 384), device="cuda").to(torch.bfloat16), torch.randn(384, device="cuda")]
    for t in range(4):
        opt.step(g, t)
    assert opt.status() == 0
    opt.close()


def _gpt2l():
    from paper_2605_19811_gb300 import synth
    return synth.scaled_set("gpt_2l", layers=2, d=768, vocab=4096).shapes


def test_step_stops_after_a_wait_gives_up(monkeypatch):
    """LM_WAIT_LIMIT_NS=1 (read by lm_create) makes the bounded waits of a
    real Muon step give up.  The kernel that gave up raises LM_FLAG_TIMEOUT;
    every kernel after it, in this step and the next, reads the flag at entry
    and does nothing: no matrix is written (the parameter write would be in
    the last NS launch), the next (Lion) step changes nothing, and the step
    returns within about one wait limit instead of one limit per launch."""
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    from paper_2605_19811_gb300 import synth
    from tests.lm_testutil import bits, host_tensor
    shapes = _gpt2l()
    W0 = synth.init_weights(shapes, seed=1)
    params = [host_tensor(w, "bf16").cuda() for w in W0]
    before = [bits(p) for p in params]
    monkeypatch.setenv("LM_WAIT_LIMIT_NS", "1")
    opt = L.LionMuon(params, period=2)
    monkeypatch.delenv("LM_WAIT_LIMIT_NS")
    grads = [[host_tensor(x, "bf16").cuda() for x in synth.draw_grads(shapes, "student_t", seed=0, step=t)]
             for t in range(2)]
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    opt.step(grads[0], 0)            # Muon step
    torch.cuda.synchronize()
    dt = time.perf_counter() - t0
    after_muon = [bits(p) for p in params]
    m_after_muon = [bits(opt.momentum(i)) for i in range(len(params))]
    opt.step(grads[1], 1)            # Lion step: the flag is still set
    torch.cuda.synchronize()
    for i, s in enumerate(shapes):
        if len(s) == 2:              # matrices: never written
            np.testing.assert_array_equal(after_muon[i], before[i])
        np.testing.assert_array_equal(bits(params[i]), after_muon[i])
        np.testing.assert_array_equal(bits(opt.momentum(i)), m_after_muon[i])
    assert opt.status() & L.LM_FLAG_TIMEOUT
    assert dt < 2.0, dt
    opt.close()


def test_state_works_after_flag_cleared():
    """A state with the normal limit, after another state's give-up on the
    same context: its steps run and report no flags."""
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    from paper_2605_19811_gb300 import synth
    from tests.lm_testutil import host_tensor
    shapes = _gpt2l()
    params = [host_tensor(w, "bf16").cuda() for w in synth.init_weights(shapes, seed=1)]
    opt = L.LionMuon(params, period=2)
    for t in range(2):
        opt.step([host_tensor(x, "bf16").cuda() for x in synth.draw_grads(shapes, "student_t", seed=0, step=t)], t)
    torch.cuda.synchronize()
    assert opt.status() == 0
    assert all(bool(torch.isfinite(p.float()).all()) for p in params)
    opt.close()


@pytest.mark.parametrize("precision", [1, 2])   # LM_BF16, LM_NS_F32_TC
def test_msign_reports_timeout(precision, monkeypatch):
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    x = torch.randn(1024, 4096, device="cuda")
    out = torch.empty_like(x)
    monkeypatch.setenv("LM_WAIT_LIMIT_NS", "1")
    with pytest.raises(L.LionMuonError) as ei:
        L.msign_ns(x, out, precision=precision)
    assert ei.value.status == 7                        # LM_ERR_TIMEOUT
    monkeypatch.delenv("LM_WAIT_LIMIT_NS")
    L.msign_ns(x, out, precision=precision)            # the normal limit: no error
    torch.cuda.synchronize()
    assert bool(torch.isfinite(out).all())


def test_noalloc_status_reports_timeout(monkeypatch):
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    x = torch.randn(768, 2048, device="cuda").to(torch.bfloat16)
    out = torch.empty(768, 2048, device="cuda")
    monkeypatch.setenv("LM_WAIT_LIMIT_NS", "1")
    L.msign_ns_noalloc(x, out, precision=L.LM_BF16)
    st, flags = L.msign_ns_noalloc_status()
    assert st == 7 and flags & L.LM_FLAG_TIMEOUT
    monkeypatch.delenv("LM_WAIT_LIMIT_NS")
    L.msign_ns_noalloc(x, out, precision=L.LM_BF16)
    st, flags = L.msign_ns_noalloc_status()
    assert st == 0 and flags == 0
