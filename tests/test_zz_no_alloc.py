"""lm_msign_ns_noalloc, the Newton-Schulz entry point for callers that cannot
allocate device memory while they run: a program whose device memory is all
handed out up front by its own allocator, or a latency-critical loop where
cudaMalloc/cudaFree (and cudaFree's device synchronisation) are not
acceptable.  It works in a fixed in-library scratch area instead of
allocating.  Through the C ABI these tests check that calls in a row (a
larger matrix, then smaller ones that reuse what the first left in the
scratch area) match the fp64 oracle recurrence within the NS tolerances
(2e-2 bf16, 1e-5 fp32) and the allocating lm_msign_ns within the same, for
0, 1 and 5 iterations and for an input dtype other than the precision; that
a matrix close to the 64 MiB limit runs and one beyond it is refused; and
that the call's status word reads clean.

The file name sorts last so that a run stopping at its first failure has
already run every other test."""

import ctypes

import numpy as np
import pytest

import oracle as O
from paper_2605_19811_gb300 import synth
from tests.lm_testutil import host_tensor, rel_fro, stored_values

pytestmark = pytest.mark.gpu

QUINTIC = (3.4445, -4.7750, 2.0315)
TOL = {1: 2e-2, 0: 1e-5}   # LM_BF16, LM_F32


def _call(entry, x, precision, steps=5, coeffs=QUINTIC):
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    lib = L.load_library()
    out = torch.empty(x.shape, dtype=torch.float32, device="cuda")
    di, do = L.tensor_desc(x), L.tensor_desc(out)
    fn = getattr(lib, entry)
    st = fn(ctypes.byref(di), ctypes.byref(do), steps, *coeffs, 1e-7, precision,
            ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == 0, (entry, st, lib.lm_last_error())
    torch.cuda.synchronize()
    return stored_values(out)


@pytest.mark.parametrize("precision,in_dtype", [(1, "bf16"), (0, "f32"), (0, "bf16"), (1, "f32")])
@pytest.mark.parametrize("steps", [5, 1, 0])
def test_noalloc_matches_oracle_and_allocating_entry_point(precision, in_dtype, steps):
    from paper_2605_19811_gb300 import lionmuon as L
    # a larger call first, then smaller ones with other padding, so the later
    # calls run on scratch the first one left behind
    for shape, seed in (((640, 1500), 1), ((300, 200), 2), ((1000, 130), 3)):
        xh = host_tensor(synth.draw_matrix(shape, seed=seed), in_dtype)
        x = xh.cuda()
        got = _call("lm_msign_ns_noalloc", x, precision, steps)
        want = O.ns_polynomial(stored_values(xh), steps, *QUINTIC, 1e-7)
        alloc = _call("lm_msign_ns", x, precision, steps)
        assert got.shape == want.shape
        assert np.all(np.isfinite(got))
        assert rel_fro(got, want) <= TOL[precision]
        assert rel_fro(alloc, want) <= TOL[precision]
        assert rel_fro(got, alloc) <= TOL[precision]
        assert L.msign_ns_noalloc_status() == (0, 0)


@pytest.mark.parametrize("precision,in_dtype", [(1, "bf16"), (0, "f32")])
def test_noalloc_cubic_matches_oracle(precision, in_dtype):
    """The classic cubic (c = 0: the tensor-core path runs no polynomial
    launch and APPLY reads A) through both entry points, wide and tall."""
    cubic = (1.5, -0.5, 0.0)
    for shape, seed in (((384, 1100), 6), ((900, 256), 7)):
        xh = host_tensor(synth.draw_matrix(shape, seed=seed), in_dtype)
        x = xh.cuda()
        got = _call("lm_msign_ns_noalloc", x, precision, 8, cubic)
        alloc = _call("lm_msign_ns", x, precision, 8, cubic)
        want = O.ns_polynomial(stored_values(xh), 8, *cubic, 1e-7)
        assert rel_fro(got, want) <= TOL[precision]
        assert rel_fro(alloc, want) <= TOL[precision]


def test_noalloc_near_scratch_limit():
    """2048 x 5120 in bf16 needs (2 * 2048 * 5120 + 2 * 2048^2) * 2 bytes plus
    tables, about 56 MiB: it fits."""
    xh = host_tensor(synth.draw_matrix((2048, 5120), seed=4), "bf16")
    got = _call("lm_msign_ns_noalloc", xh.cuda(), 1)
    want = O.ns_polynomial(stored_values(xh), 5, *QUINTIC, 1e-7)
    assert rel_fro(got, want) <= TOL[1]


def test_noalloc_rejects_matrix_beyond_scratch_limit():
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    lib = L.load_library()
    x = torch.empty((2048, 8192), dtype=torch.bfloat16, device="cuda")
    out = torch.empty_like(x)
    di, do = L.tensor_desc(x), L.tensor_desc(out)
    st = lib.lm_msign_ns_noalloc(ctypes.byref(di), ctypes.byref(do), 5, *QUINTIC, 1e-7, 1,
                                 ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == 6                      # LM_ERR_UNSUPPORTED
    assert b"64 MiB" in lib.lm_last_error()
