"""Tensor pointers that are not device memory are refused before any work is
enqueued: parameters in host memory at lm_create, page-locked host gradients
at lm_step (a rejected step leaves weights and momentum untouched, and the
next valid step runs), momentum sources, and lm_msign_ns / its no-allocation
variant.  Only page-locked host memory, which the GPU could reach, is ever
passed to a call that launches kernels; plain host memory only goes to
lm_create, which reads no tensor data."""

import ctypes

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2605_19811_gb300 import lionmuon as L

pytestmark = pytest.mark.gpu

INVALID_ARG = 1


def _desc(ptr, rows, cols, dtype=L.LM_F32):
    return L.LmTensor(ctypes.c_void_p(ptr), rows, cols, dtype)


def _create(descs):
    lib = L.load_library()
    cfg = L.default_config()
    h = ctypes.c_void_p()
    arr = (L.LmTensor * len(descs))(*descs)
    st = lib.lm_create(arr, len(descs), ctypes.byref(cfg), None, ctypes.byref(h))
    return st, h


def test_create_refuses_host_parameters():
    host = np.zeros((64, 128), dtype=np.float32)             # plain (unregistered) host memory
    st, h = _create([_desc(host.ctypes.data, 64, 128)])
    assert st == INVALID_ARG and not h.value
    pinned = torch.zeros((64, 128), dtype=torch.float32).pin_memory()
    st, h = _create([_desc(pinned.data_ptr(), 64, 128)])
    assert st == INVALID_ARG and not h.value
    assert b"host" in L.load_library().lm_last_error()


def test_step_refuses_pinned_host_gradients_and_changes_nothing():
    p = [torch.randn(256, 384, device="cuda").to(torch.bfloat16), torch.randn(384, device="cuda")]
    opt = L.LionMuon(p, period=2)
    g_dev = [torch.randn_like(x) * 1e-3 for x in p]
    opt.step(g_dev, 0)
    torch.cuda.synchronize()
    before = [x.clone() for x in p]
    mom_before = [opt.momentum(i).clone() for i in range(2)]
    g_host = [g_dev[0].cpu().pin_memory(), g_dev[1]]
    with pytest.raises(L.LionMuonError) as e:
        opt.step(g_host, 1)
    assert e.value.status == INVALID_ARG
    torch.cuda.synchronize()
    assert all(torch.equal(a, b) for a, b in zip(p, before))
    assert all(torch.equal(opt.momentum(i), mom_before[i]) for i in range(2))
    opt.step(g_dev, 1)                                      # a valid step still runs
    torch.cuda.synchronize()
    assert opt.status() == 0
    assert not torch.equal(p[0], before[0])
    opt.close()


def test_set_momentum_refuses_pinned_host_source():
    p = [torch.zeros(128, 256, device="cuda")]
    opt = L.LionMuon(p)
    src = torch.ones(128, 256).pin_memory()
    with pytest.raises(L.LionMuonError) as e:
        opt.set_momentum(0, src)
    assert e.value.status == INVALID_ARG
    torch.cuda.synchronize()
    assert float(opt.momentum(0).abs().sum()) == 0.0
    opt.close()


@pytest.mark.parametrize("noalloc", [False, True])
def test_msign_refuses_pinned_host_tensors(noalloc):
    x = torch.randn(128, 256).pin_memory()
    out_dev = torch.empty(128, 256, device="cuda")
    x_dev = x.cuda()
    out_host = torch.empty(128, 256).pin_memory()
    call = L.msign_ns_noalloc if noalloc else L.msign_ns
    for a, b in ((x, out_dev), (x_dev, out_host)):
        with pytest.raises(L.LionMuonError) as e:
            call(a, b, precision=L.LM_F32)
        assert e.value.status == INVALID_ARG
    call(x_dev, out_dev, precision=L.LM_F32)                # device tensors still work
    torch.cuda.synchronize()
    assert bool(torch.isfinite(out_dev).all())
