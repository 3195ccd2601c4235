"""Python binding of the C ABI in ``include/lionmuon.h`` (ctypes).

Argument marshalling only: every step of the optimizer runs in the CUDA
library.  torch tensors supply device memory and the current CUDA stream.
If the shared library is missing this module raises; there is no fallback.
"""

from __future__ import annotations

import ctypes
import os
from typing import List, Optional, Sequence

from . import build as _build

LM_OK = 0
LM_F32 = 0
LM_BF16 = 1
LM_NS_F32_TC = 2      # ns_precision: fp32 values as three bf16 pieces on the tensor cores
LM_FLAG_NONFINITE = 0x1
LM_FLAG_TIMEOUT = 0x2
LM_FLAG_GUARD = 0x4

STATUS_NAMES = {0: "LM_OK", 1: "LM_ERR_INVALID_ARG", 2: "LM_ERR_DTYPE", 3: "LM_ERR_ALIGN",
                4: "LM_ERR_OOM", 5: "LM_ERR_CUDA", 6: "LM_ERR_UNSUPPORTED", 7: "LM_ERR_TIMEOUT"}

# Every symbol include/lionmuon.h declares.
EXPORTED = ("lm_config_default", "lm_create", "lm_step", "lm_set_lr", "lm_msign_ns",
            "lm_get_momentum", "lm_set_momentum", "lm_get_status", "lm_state_bytes",
            "lm_workspace_bytes", "lm_destroy", "lm_status_string", "lm_last_error",
            "lm_kernel_launch_count", "lm_profile_enable", "lm_profile_read",
            "lm_msign_ns_noalloc", "lm_probe_bounded_wait", "lm_msign_ns_coeffs",
            "lm_set_adamw_lr", "lm_get_second_moment", "lm_set_second_moment", "lm_get_selection",
            "lm_msign_ns_noalloc_status", "lm_shard_owners", "lm_config_size")

KERNEL_FAMILIES = ("lion", "momentum_norm", "ns_gram", "ns_poly", "ns_apply", "finalize", "other", "adamw",
                   "srank")
LM_VECTOR_LION, LM_VECTOR_ADAMW = 0, 1
LM_SCHEDULE_PERIOD, LM_SCHEDULE_STABLE_RANK = 0, 1


class LmTensor(ctypes.Structure):
    _fields_ = [("data", ctypes.c_void_p), ("rows", ctypes.c_int64), ("cols", ctypes.c_int64),
                ("dtype", ctypes.c_int)]


class LmConfig(ctypes.Structure):
    _fields_ = [("beta1", ctypes.c_double), ("beta2", ctypes.c_double),
                ("eta_muon", ctypes.c_double), ("eta_lion", ctypes.c_double),
                ("weight_decay", ctypes.c_double), ("period", ctypes.c_int64),
                ("ns_steps", ctypes.c_int), ("ns_a", ctypes.c_double), ("ns_b", ctypes.c_double),
                ("ns_c", ctypes.c_double), ("ns_eps", ctypes.c_double),
                ("shape_scale", ctypes.c_double), ("ns_precision", ctypes.c_int),
                ("ns_coeffs", ctypes.POINTER(ctypes.c_double)),
                ("vector_rule", ctypes.c_int), ("adamw_lr", ctypes.c_double),
                ("adamw_beta1", ctypes.c_double), ("adamw_beta2", ctypes.c_double),
                ("adamw_eps", ctypes.c_double), ("adamw_weight_decay", ctypes.c_double),
                ("schedule", ctypes.c_int), ("srank_alpha", ctypes.c_double), ("srank_iters", ctypes.c_int),
                ("srank_seed", ctypes.c_uint64), ("shard_rank", ctypes.c_int), ("shard_world", ctypes.c_int)]


class LmProfile(ctypes.Structure):
    _fields_ = [("ms", ctypes.c_double * 9), ("launches", ctypes.c_uint64 * 9)]


class LionMuonError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str):
        self.status = status
        super().__init__(f"{where}: {STATUS_NAMES.get(status, status)}: {detail}")


_LIB = None


def load_library(path: Optional[str] = None) -> ctypes.CDLL:
    """Load liblionmuon.so (built in-tree by ``build.build()``); raises if absent."""
    global _LIB
    if _LIB is not None and path is None:
        return _LIB
    p = path or _build.library_path()
    if not os.path.exists(p):
        raise RuntimeError(f"{p} not found: build the CUDA library first "
                           "(python -c 'import __graft_entry__ as g; g.build()')")
    lib = ctypes.CDLL(p)
    c_void_p, c_int, c_int64, c_double = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_double
    P = ctypes.POINTER
    lib.lm_config_size.argtypes = []
    lib.lm_config_size.restype = ctypes.c_size_t
    if lib.lm_config_size() != ctypes.sizeof(LmConfig):
        raise RuntimeError(f"{p}: lm_config is {lib.lm_config_size()} bytes in the library but "
                           f"{ctypes.sizeof(LmConfig)} in this binding (rebuild the library)")
    lib.lm_config_default.argtypes = [P(LmConfig)]
    lib.lm_config_default.restype = None
    lib.lm_create.argtypes = [P(LmTensor), c_int, P(LmConfig), c_void_p, P(c_void_p)]
    lib.lm_create.restype = c_int
    lib.lm_step.argtypes = [c_void_p, P(LmTensor), c_int, c_int64, c_void_p]
    lib.lm_step.restype = c_int
    lib.lm_set_lr.argtypes = [c_void_p, c_double, c_double]
    lib.lm_set_lr.restype = c_int
    lib.lm_msign_ns.argtypes = [P(LmTensor), P(LmTensor), c_int, c_double, c_double, c_double,
                                c_double, c_int, c_void_p]
    lib.lm_msign_ns.restype = c_int
    lib.lm_msign_ns_coeffs.argtypes = [P(LmTensor), P(LmTensor), c_int, P(c_double), c_double, c_int,
                                       c_void_p]
    lib.lm_msign_ns_coeffs.restype = c_int
    lib.lm_msign_ns_noalloc.argtypes = [P(LmTensor), P(LmTensor), c_int, c_double, c_double, c_double,
                                        c_double, c_int, c_void_p]
    lib.lm_msign_ns_noalloc.restype = c_int
    lib.lm_shard_owners.argtypes = [P(LmTensor), c_int, c_int, P(c_int)]
    lib.lm_shard_owners.restype = c_int
    lib.lm_msign_ns_noalloc_status.argtypes = [P(ctypes.c_uint32), c_void_p]
    lib.lm_msign_ns_noalloc_status.restype = c_int
    lib.lm_get_selection.argtypes = [c_void_p, c_int, P(ctypes.c_ubyte), P(c_double)]
    lib.lm_get_selection.restype = c_int
    lib.lm_set_adamw_lr.argtypes = [c_void_p, c_double]
    lib.lm_set_adamw_lr.restype = c_int
    lib.lm_get_second_moment.argtypes = [c_void_p, c_int, P(LmTensor)]
    lib.lm_get_second_moment.restype = c_int
    lib.lm_set_second_moment.argtypes = [c_void_p, c_int, P(LmTensor), c_void_p]
    lib.lm_set_second_moment.restype = c_int
    lib.lm_get_momentum.argtypes = [c_void_p, c_int, P(LmTensor)]
    lib.lm_get_momentum.restype = c_int
    lib.lm_set_momentum.argtypes = [c_void_p, c_int, P(LmTensor), c_void_p]
    lib.lm_set_momentum.restype = c_int
    lib.lm_get_status.argtypes = [c_void_p, P(ctypes.c_uint32)]
    lib.lm_get_status.restype = c_int
    lib.lm_state_bytes.argtypes = [c_void_p]
    lib.lm_state_bytes.restype = ctypes.c_size_t
    lib.lm_workspace_bytes.argtypes = [c_void_p]
    lib.lm_workspace_bytes.restype = ctypes.c_size_t
    lib.lm_destroy.argtypes = [c_void_p]
    lib.lm_destroy.restype = None
    lib.lm_status_string.argtypes = [c_int]
    lib.lm_status_string.restype = ctypes.c_char_p
    lib.lm_last_error.argtypes = []
    lib.lm_last_error.restype = ctypes.c_char_p
    lib.lm_kernel_launch_count.argtypes = []
    lib.lm_kernel_launch_count.restype = ctypes.c_uint64
    lib.lm_probe_bounded_wait.argtypes = [ctypes.c_uint64, P(ctypes.c_uint32), c_void_p]
    lib.lm_probe_bounded_wait.restype = c_int
    lib.lm_profile_enable.argtypes = [c_void_p, c_int]
    lib.lm_profile_enable.restype = c_int
    lib.lm_profile_read.argtypes = [c_void_p, P(LmProfile), c_int]
    lib.lm_profile_read.restype = c_int
    if path is None:
        _LIB = lib
    return lib


def _check(lib, st: int, where: str):
    if st != LM_OK:
        raise LionMuonError(st, where, lib.lm_last_error().decode())


def _dtype_code(t) -> int:
    import torch
    if t.dtype == torch.bfloat16:
        return LM_BF16
    if t.dtype == torch.float32:
        return LM_F32
    raise TypeError(f"unsupported dtype {t.dtype}")


def tensor_desc(t) -> LmTensor:
    """lm_tensor of a contiguous torch tensor (vectors are 1 x n)."""
    if not t.is_contiguous():
        raise ValueError("tensors must be contiguous")
    if t.dim() == 1:
        rows, cols = 1, t.shape[0]
    elif t.dim() == 2:
        rows, cols = t.shape
    else:
        raise ValueError("tensors must be 1-D or 2-D")
    return LmTensor(ctypes.c_void_p(t.data_ptr()), rows, cols, _dtype_code(t))


def _stream_handle(stream) -> ctypes.c_void_p:
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def default_config() -> LmConfig:
    cfg = LmConfig()
    load_library().lm_config_default(ctypes.byref(cfg))
    return cfg


def kernel_launch_count() -> int:
    return int(load_library().lm_kernel_launch_count())


class _DeviceArray:
    """__cuda_array_interface__ view of library-owned device memory."""

    def __init__(self, ptr: int, shape, typestr: str):
        self.__cuda_array_interface__ = {"shape": tuple(shape), "typestr": typestr,
                                         "data": (ptr, False), "version": 3, "strides": None}


class LionMuon:
    """Optimizer state over a list of torch parameters (the ``lm_state``)."""

    def __init__(self, params: Sequence, stream=None, **cfg):
        """cfg: lm_config fields by name; ns_coeffs may be a sequence of
        (a_k, b_k, c_k) triples, one per NS iteration (ns_steps follows it)."""
        self._lib = load_library()
        self.params = list(params)
        c = default_config()
        table = cfg.pop("ns_coeffs", None)
        for k, v in cfg.items():
            if not hasattr(c, k):
                raise TypeError(f"unknown config field {k!r}")
            setattr(c, k, v)
        keep = None
        if table is not None:
            keep = _coeff_array(table)
            c.ns_steps = len(keep) // 3
            c.ns_coeffs = keep
        self.config = c
        descs = (LmTensor * len(self.params))(*[tensor_desc(p) for p in self.params])
        h = ctypes.c_void_p()
        _check(self._lib, self._lib.lm_create(descs, len(self.params), ctypes.byref(c),
                                              _stream_handle(stream), ctypes.byref(h)), "lm_create")
        self._h = h
        c.ns_coeffs = None   # lm_create copied the table

    def step(self, grads: Sequence, t: int, stream=None) -> None:
        descs = (LmTensor * len(grads))(*[tensor_desc(g) for g in grads])
        _check(self._lib, self._lib.lm_step(self._h, descs, len(grads), int(t), _stream_handle(stream)),
               "lm_step")

    def step_descs(self, descs, n: int, t: int, stream_handle) -> None:
        """lm_step with pre-built descriptors (no per-call marshalling)."""
        _check(self._lib, self._lib.lm_step(self._h, descs, n, int(t), stream_handle), "lm_step")

    def capture_steps(self, grads: Sequence, t0: int = 0) -> list:
        """Capture one step of each phase into torch.cuda.CUDAGraph objects:
        graphs[k] runs step t0 + k, for k < P (P = period; one graph when
        P = 0 or under the stable-rank schedule).  The steps depend on t only
        through t mod P, so with t0 % P == 0 step t replays graphs[t % P].
        The graphs read ``grads`` (write each step's gradients into them
        before its replay) and keep the learning rates of the capture.  The
        AdamW rule for vectors uses t itself and is refused.  Capturing runs
        nothing; each replay runs one step."""
        import torch
        c = self.config
        if c.vector_rule == LM_VECTOR_ADAMW:
            raise ValueError("capture_steps: the AdamW vector rule depends on t (bias correction)")
        period = int(c.period)
        if c.schedule == LM_SCHEDULE_STABLE_RANK or period == 0:
            nphase = 1
        else:
            nphase = period
            if t0 % period != 0:
                raise ValueError("capture_steps: t0 must be a multiple of the period")
        descs = (LmTensor * len(grads))(*[tensor_desc(g) for g in grads])
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        graphs = []
        for k in range(nphase):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=side):
                self.step_descs(descs, len(grads), t0 + k, ctypes.c_void_p(side.cuda_stream))
            graphs.append(g)
        torch.cuda.current_stream().wait_stream(side)
        return graphs

    def set_lr(self, eta_muon: float, eta_lion: float) -> None:
        _check(self._lib, self._lib.lm_set_lr(self._h, eta_muon, eta_lion), "lm_set_lr")

    def momentum(self, i: int):
        """Read-only torch view of parameter i's fp32 momentum buffer."""
        import torch
        v = LmTensor()
        _check(self._lib, self._lib.lm_get_momentum(self._h, i, ctypes.byref(v)), "lm_get_momentum")
        shape = tuple(self.params[i].shape)
        return torch.as_tensor(_DeviceArray(v.data, shape, "<f4"), device=self.params[i].device)

    def selection(self):
        """(took_muon, srank) of the last step, one entry per parameter:
        whether it took the Muon step, and under the stable-rank schedule the
        estimate ||M||_F^2 / sigma_1_hat^2 behind it (NaN otherwise)."""
        n = len(self.params)
        took = (ctypes.c_ubyte * n)()
        est = (ctypes.c_double * n)()
        _check(self._lib, self._lib.lm_get_selection(self._h, n, took, est), "lm_get_selection")
        return [bool(x) for x in took], [float(x) for x in est]

    def set_adamw_lr(self, lr: float) -> None:
        _check(self._lib, self._lib.lm_set_adamw_lr(self._h, lr), "lm_set_adamw_lr")

    def second_moment(self, i: int):
        """Read-only torch view of 1-D parameter i's AdamW second moment."""
        import torch
        v = LmTensor()
        _check(self._lib, self._lib.lm_get_second_moment(self._h, i, ctypes.byref(v)), "lm_get_second_moment")
        shape = tuple(self.params[i].shape)
        return torch.as_tensor(_DeviceArray(v.data, shape, "<f4"), device=self.params[i].device)

    def set_second_moment(self, i: int, src, stream=None) -> None:
        d = tensor_desc(src)
        _check(self._lib, self._lib.lm_set_second_moment(self._h, i, ctypes.byref(d), _stream_handle(stream)),
               "lm_set_second_moment")

    def set_momentum(self, i: int, src, stream=None) -> None:
        d = tensor_desc(src)
        _check(self._lib, self._lib.lm_set_momentum(self._h, i, ctypes.byref(d), _stream_handle(stream)),
               "lm_set_momentum")

    def status(self) -> int:
        f = ctypes.c_uint32()
        _check(self._lib, self._lib.lm_get_status(self._h, ctypes.byref(f)), "lm_get_status")
        return int(f.value)

    def profile(self, on: bool = True) -> None:
        """Time every kernel launch of later steps with CUDA events."""
        _check(self._lib, self._lib.lm_profile_enable(self._h, 1 if on else 0), "lm_profile_enable")

    def profile_read(self, reset: bool = True) -> dict:
        """{family: (total ms, launches)} of the timed launches (synchronises);
        "ns_gemm" sums the three Newton-Schulz phases."""
        p = LmProfile()
        _check(self._lib, self._lib.lm_profile_read(self._h, ctypes.byref(p), 1 if reset else 0),
               "lm_profile_read")
        out = {name: (p.ms[i], int(p.launches[i])) for i, name in enumerate(KERNEL_FAMILIES)}
        out["ns_gemm"] = (sum(out[k][0] for k in ("ns_gram", "ns_poly", "ns_apply")),
                          sum(out[k][1] for k in ("ns_gram", "ns_poly", "ns_apply")))
        return out

    def state_bytes(self) -> int:
        return int(self._lib.lm_state_bytes(self._h))

    def workspace_bytes(self) -> int:
        return int(self._lib.lm_workspace_bytes(self._h))

    def close(self) -> None:
        if getattr(self, "_h", None):
            self._lib.lm_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def msign_ns(x, out, steps: int = 5, a: float = 3.4445, b: float = -4.7750, c: float = 2.0315,
             eps: float = 1e-7, precision: int = LM_BF16, stream=None):
    """out <- NS_steps(x) (Newton-Schulz msign approximation) via lm_msign_ns."""
    lib = load_library()
    di, do = tensor_desc(x), tensor_desc(out)
    _check(lib, lib.lm_msign_ns(ctypes.byref(di), ctypes.byref(do), steps, a, b, c, eps, precision,
                                _stream_handle(stream)), "lm_msign_ns")
    return out


def _coeff_array(table):
    """Flatten (a_k, b_k, c_k) triples into a ctypes double array."""
    flat = [float(x) for tr in table for x in tr]
    if any(len(tr) != 3 for tr in table):
        raise ValueError("every NS coefficient entry must be an (a, b, c) triple")
    return (ctypes.c_double * max(len(flat), 1))(*flat) if flat else None


def msign_ns_coeffs(x, out, coeffs, eps: float = 1e-7, precision: int = LM_BF16, stream=None):
    """out <- NS(x) with iteration-dependent coefficients: coeffs is a
    sequence of (a_k, b_k, c_k) triples, one per iteration (lm_msign_ns_coeffs)."""
    lib = load_library()
    di, do = tensor_desc(x), tensor_desc(out)
    arr = _coeff_array(coeffs)
    _check(lib, lib.lm_msign_ns_coeffs(ctypes.byref(di), ctypes.byref(do), len(coeffs), arr, eps, precision,
                                       _stream_handle(stream)), "lm_msign_ns_coeffs")
    return out


def probe_bounded_wait(limit_ns: int, stream=None):
    """Run the bounded-wait probe; returns (status, device flags)."""
    lib = load_library()
    f = ctypes.c_uint32()
    st = lib.lm_probe_bounded_wait(limit_ns, ctypes.byref(f), _stream_handle(stream))
    return st, int(f.value)


def msign_ns_noalloc(x, out, steps: int = 5, a: float = 3.4445, b: float = -4.7750, c: float = 2.0315,
                     eps: float = 1e-7, precision: int = LM_BF16, stream=None):
    """out <- NS_steps(x) via lm_msign_ns_noalloc (fixed in-library workspace,
    no device allocation; calls must not overlap on the GPU)."""
    lib = load_library()
    di, do = tensor_desc(x), tensor_desc(out)
    _check(lib, lib.lm_msign_ns_noalloc(ctypes.byref(di), ctypes.byref(do), steps, a, b, c, eps,
                                        precision, _stream_handle(stream)), "lm_msign_ns_noalloc")
    return out


def msign_ns_noalloc_status(stream=None):
    """Synchronise the stream of the last lm_msign_ns_noalloc call and return
    (status, device flags) of that call (lm_msign_ns_noalloc_status)."""
    lib = load_library()
    f = ctypes.c_uint32()
    st = lib.lm_msign_ns_noalloc_status(ctypes.byref(f), _stream_handle(stream))
    return st, int(f.value)
