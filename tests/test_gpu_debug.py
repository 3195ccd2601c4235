"""Debug switches read by lm_create from the environment: guard bands around
every workspace part (LM_DEBUG=1) stay intact through steps of every kind and
report an overwrite through LM_FLAG_GUARD; LM_FAULT=oom makes lm_create fail
as a failed allocation would; LM_NS_FORCE_FP32=1 selects the fp32
Newton-Schulz path (bit-identical to asking for it)."""

import numpy as np
import pytest

from tests.lm_testutil import bits, host_tensor, make_problem

pytestmark = pytest.mark.gpu

SHAPES = [(96, 200), (200, 96), (300, 130), (128,)]


def _run(opt_kwargs, steps=4, shapes=SHAPES):
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    W0, grads = make_problem(shapes, "student_t", steps)
    params = [host_tensor(w, "bf16").cuda() for w in W0]
    opt = L.LionMuon(params, **opt_kwargs)
    for t in range(steps):
        opt.step([host_tensor(g, "bf16").cuda() for g in grads[t]], t)
    torch.cuda.synchronize()
    return opt, params


@pytest.mark.parametrize("kwargs", [dict(period=2), dict(period=1, vector_rule=1),
                                    dict(schedule=1, srank_alpha=0.5), dict(period=2, ns_precision=0)])
def test_guard_bands_stay_intact(monkeypatch, kwargs):
    monkeypatch.setenv("LM_DEBUG", "1")
    opt, _ = _run(kwargs)
    assert opt.status() == 0
    opt.close()


def test_guard_band_overwrite_is_reported(monkeypatch):
    """The last parameter's momentum (128 floats, a multiple of the 64-float
    alignment) ends exactly where its guard band begins; writing 16 bytes
    there (inside the state's own allocation) must be reported."""
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    monkeypatch.setenv("LM_DEBUG", "1")
    opt, params = _run(dict(period=2))
    assert opt.status() == 0
    m = opt.momentum(len(params) - 1)
    assert m.numel() == 128
    spill = torch.as_tensor(L._DeviceArray(m.data_ptr() + m.numel() * 4, (4,), "<f4"), device=m.device)
    spill.fill_(1.0)
    torch.cuda.synchronize()
    assert opt.status() & L.LM_FLAG_GUARD
    opt.close()


def test_injected_allocation_failure(monkeypatch):
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    monkeypatch.setenv("LM_FAULT", "oom")
    p = [torch.zeros((32, 48), dtype=torch.bfloat16, device="cuda")]
    with pytest.raises(L.LionMuonError) as e:
        L.LionMuon(p)
    assert e.value.status == 4                    # LM_ERR_OOM
    monkeypatch.delenv("LM_FAULT")
    L.LionMuon(p).close()                          # the next create is unaffected


def test_force_fp32_ns_equals_fp32_request(monkeypatch):
    _, pa = _run(dict(period=2, ns_precision=0))
    monkeypatch.setenv("LM_NS_FORCE_FP32", "1")
    _, pb = _run(dict(period=2, ns_precision=1))
    for a, b in zip(pa, pb):
        np.testing.assert_array_equal(bits(a), bits(b))
