"""lm_msign_ns_noalloc, the Newton-Schulz entry point for callers that cannot
allocate device memory while they run (their memory is budgeted up front, or
cudaMalloc/cudaFree are too costly where they call from).  It works in a
fixed in-library scratch area instead of allocating, so these tests check,
through the C ABI, that two calls in a row give the same result as the
allocating lm_msign_ns within the NS tolerances (2e-2 bf16, 1e-5 fp32), and
that a matrix too large for the scratch area is refused.

The file name sorts last so that a run stopping at its first failure has
already run every other test."""

import ctypes

import numpy as np
import pytest

from paper_2605_19811_gb300 import synth
from tests.lm_testutil import host_tensor, rel_fro, stored_values

pytestmark = pytest.mark.gpu

QUINTIC = (3.4445, -4.7750, 2.0315)
TOL = {1: 2e-2, 0: 1e-5}   # LM_BF16, LM_F32


def _call(entry, x, precision, steps=5):
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    lib = L.load_library()
    out = torch.empty(x.shape, dtype=torch.float32, device="cuda")
    di, do = L.tensor_desc(x), L.tensor_desc(out)
    fn = getattr(lib, entry)
    st = fn(ctypes.byref(di), ctypes.byref(do), steps, *QUINTIC, 1e-7, precision,
            ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == 0, (entry, st, lib.lm_last_error())
    torch.cuda.synchronize()
    return stored_values(out)


@pytest.mark.parametrize("precision", [1, 0])
def test_noalloc_matches_allocating_entry_point_two_calls(precision):
    in_dtype = "bf16" if precision == 1 else "f32"
    # a larger call first, then a smaller one with different padding, so the
    # second call runs on scratch the first one left behind
    for shape, seed in (((640, 1500), 1), ((300, 200), 2)):
        x = host_tensor(synth.draw_matrix(shape, seed=seed), in_dtype).cuda()
        want = _call("lm_msign_ns", x, precision)
        got = _call("lm_msign_ns_noalloc", x, precision)
        assert got.shape == want.shape
        assert np.all(np.isfinite(got))
        assert rel_fro(got, want) <= TOL[precision]


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
