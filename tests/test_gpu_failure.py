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
