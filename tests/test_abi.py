"""Host-side checks of the C ABI (no GPU needed): the library loads, exports
every symbol the header declares, fills the default config with the paper's
values, and rejects invalid arguments before touching a device."""

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "lionmuon.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2605_19811_gb300 import build, lionmuon
    build.build()
    return lionmuon.load_library()


def declared_symbols():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(lm_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_boundary():
    syms = declared_symbols()
    for s in ("lm_create", "lm_step", "lm_set_lr", "lm_msign_ns", "lm_get_momentum",
              "lm_get_status", "lm_state_bytes", "lm_destroy", "lm_status_string"):
        assert s in syms


def test_library_exports_every_declared_symbol(lib):
    from paper_2605_19811_gb300 import lionmuon
    syms = declared_symbols()
    for s in syms:
        assert hasattr(lib, s), f"{s} declared in lionmuon.h but not exported"
    assert sorted(lionmuon.EXPORTED) == syms


def test_default_config_matches_paper(lib):
    from paper_2605_19811_gb300 import lionmuon as L
    c = L.default_config()
    assert (c.beta1, c.beta2) == (0.9, 0.99)          # Table 5, Lion/LionMuon betas
    assert c.weight_decay == 0.1                      # Table 5
    assert c.ns_steps == 5                            # Table 5, K_NS
    assert c.shape_scale == 0.2                       # Table 5, 0.2 sqrt(max(m, n))
    assert (c.eta_muon, c.eta_lion) == (3e-3, 2e-5)   # Appendix E, LionMuon P=2
    assert c.period == 2
    assert (c.ns_a, c.ns_b, c.ns_c) == (3.4445, -4.7750, 2.0315)


def test_status_strings(lib):
    for code, name in [(0, b"LM_OK"), (1, b"LM_ERR_INVALID_ARG"), (7, b"LM_ERR_TIMEOUT")]:
        assert lib.lm_status_string(code) == name


def _tensor(ptr, rows, cols, dt):
    from paper_2605_19811_gb300.lionmuon import LmTensor
    return LmTensor(ctypes.c_void_p(ptr), rows, cols, dt)


def test_create_rejects_bad_arguments_before_device_use(lib):
    from paper_2605_19811_gb300 import lionmuon as L
    cfg = L.default_config()
    h = ctypes.c_void_p()
    one = (L.LmTensor * 1)(_tensor(4096, 4, 4, L.LM_BF16))
    assert lib.lm_create(one, 0, ctypes.byref(cfg), None, ctypes.byref(h)) == 1
    bad = L.LmConfig.from_buffer_copy(cfg)
    bad.beta1 = 1.0
    assert lib.lm_create(one, 1, ctypes.byref(bad), None, ctypes.byref(h)) == 1
    bad = L.LmConfig.from_buffer_copy(cfg)
    bad.period = -1
    assert lib.lm_create(one, 1, ctypes.byref(bad), None, ctypes.byref(h)) == 1
    for p in (7, 3, -1):          # LM_F32 (0), LM_BF16 (1) and LM_NS_F32_TC (2) are the valid values
        bad = L.LmConfig.from_buffer_copy(cfg)
        bad.ns_precision = p
        assert lib.lm_create(one, 1, ctypes.byref(bad), None, ctypes.byref(h)) == 1
    misaligned = (L.LmTensor * 1)(_tensor(4098, 4, 4, L.LM_BF16))
    assert lib.lm_create(misaligned, 1, ctypes.byref(cfg), None, ctypes.byref(h)) == 3
    null = (L.LmTensor * 1)(_tensor(0, 4, 4, L.LM_BF16))
    assert lib.lm_create(null, 1, ctypes.byref(cfg), None, ctypes.byref(h)) == 1
    baddt = (L.LmTensor * 1)(_tensor(4096, 4, 4, 5))
    assert lib.lm_create(baddt, 1, ctypes.byref(cfg), None, ctypes.byref(h)) == 2
    assert h.value is None
    assert b"" != lib.lm_last_error()


def test_msign_rejects_bad_arguments(lib):
    from paper_2605_19811_gb300 import lionmuon as L
    a = _tensor(4096, 8, 8, L.LM_F32)
    b = _tensor(8192, 8, 9, L.LM_F32)
    assert lib.lm_msign_ns(ctypes.byref(a), ctypes.byref(b), 5, 1, 1, 1, 0, 1, None) == 1
    v = _tensor(4096, 1, 8, L.LM_F32)
    assert lib.lm_msign_ns(ctypes.byref(v), ctypes.byref(v), 5, 1, 1, 1, 0, 1, None) == 1
    assert lib.lm_msign_ns(ctypes.byref(a), ctypes.byref(a), -1, 1, 1, 1, 0, 1, None) == 1
    assert lib.lm_msign_ns(ctypes.byref(a), ctypes.byref(a), 5, 1, 1, 1, 0, 9, None) == 1
    assert lib.lm_msign_ns(ctypes.byref(a), ctypes.byref(a), 5, 1, 1, 1, 0, 3, None) == 1
    # the no-alloc entry point has no three-piece mode
    assert lib.lm_msign_ns_noalloc(ctypes.byref(a), ctypes.byref(a), 5, 1, 1, 1, 0, L.LM_NS_F32_TC, None) == 1


def test_null_handles_are_safe(lib):
    assert lib.lm_state_bytes(None) == 0
    assert lib.lm_workspace_bytes(None) == 0
    lib.lm_destroy(None)
    f = ctypes.c_uint32()
    assert lib.lm_get_status(None, ctypes.byref(f)) == 1
    assert lib.lm_set_lr(None, 1.0, 1.0) == 1


def test_product_path_does_not_import_the_oracle():
    import subprocess
    import sys
    code = ("import sys; import paper_2605_19811_gb300.lionmuon, paper_2605_19811_gb300.synth; "
            "print(any(m == 'oracle' or m.startswith('oracle.') for m in sys.modules))")
    out = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, cwd=ROOT)
    assert out.stdout.strip() == "False", out.stderr
