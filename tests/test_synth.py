"""The seeded synthetic inputs that stand in for the paper's workloads: the
GPT-style parameter sets have the shapes and sizes the measurements are
quoted on (parameter, matrix and vector counts), and the gradient draws have
the stated distributions (Student-t with nu = 3 scaled to std 1e-3; N(0, 1e-6)
with 1% of entries x100; N(0, 1)), checked with statistics that converge on a
sample of a million values, on both the host draw and the device-style draw
(run here with torch on the CPU)."""

import numpy as np
import pytest

from paper_2605_19811_gb300 import synth


def _counts(ps):
    mats = ps.matrices
    vec = sum(int(np.prod(s)) for s in ps.shapes if len(s) == 1)
    return ps.numel, len(mats), vec


@pytest.mark.parametrize("name, numel, nmat, nvec", [
    ("tiny", 655_616, 4, 256),
    ("gpt2_124m", 123_606_528, 49, 38_400),
    ("gpt_355m", 353_601_536, 97, 100_352),
    ("gpt_720m", 772_364_800, 145, 186_880),
    ("stress_7b", 7_784_628_224, 224, 0),
])
def test_parameter_set_sizes(name, numel, nmat, nvec):
    ps = synth.PARAM_SETS[name]
    assert _counts(ps) == (numel, nmat, nvec)


def test_gpt_720m_layer_shapes():
    ps = synth.PARAM_SETS["gpt_720m"]
    mats = ps.matrices
    assert mats[0] == (50304, 1280)
    per_layer = [(1280, 3840), (1280, 1280), (1280, 5120), (5120, 1280)]
    assert mats[1:] == per_layer * 36


def _t3_median_abs(scale):
    scipy_stats = pytest.importorskip("scipy.stats")
    return float(scipy_stats.t.ppf(0.75, 3)) * scale


def test_student_t_gradients_host_draw():
    g = synth.draw_grads([(1000, 1000)], "student_t", seed=0, step=0)[0].astype(np.float64)
    want = _t3_median_abs(1e-3 / np.sqrt(3.0))
    assert abs(np.median(np.abs(g)) / want - 1.0) < 0.01
    assert abs(np.mean(g)) < 5e-6
    # heavy tails: P(|t3| > 10) = 2.13e-3, against 1.5e-23 for N(0, 1) (same scale parameter)
    scipy_stats = pytest.importorskip("scipy.stats")
    frac = np.mean(np.abs(g) > 10 * 1e-3 / np.sqrt(3.0))
    assert abs(frac / (2 * scipy_stats.t.sf(10.0, 3)) - 1.0) < 0.08


def test_student_t_gradients_device_style_draw():
    torch = pytest.importorskip("torch")
    g = synth.device_grads_torch([(1000, 1000)], "student_t", seed=0, device="cpu",
                                 dtype=torch.float32)[0].double().numpy()
    want = _t3_median_abs(1e-3 / np.sqrt(3.0))
    assert abs(np.median(np.abs(g)) / want - 1.0) < 0.01


@pytest.mark.parametrize("draw", ["host", "device"])
def test_outlier_gradients(draw):
    if draw == "host":
        g = synth.draw_grads([(1000, 1000)], "outlier", seed=2, step=0)[0].astype(np.float64)
    else:
        torch = pytest.importorskip("torch")
        g = synth.device_grads_torch([(1000, 1000)], "outlier", seed=2, device="cpu",
                                     dtype=torch.float32)[0].double().numpy()
    # base entries are N(0, 1e-6): beyond 6e-3 with probability 2e-9; the 1%
    # scaled by 100 are N(0, 1e-2): beyond 6e-3 with probability 0.952
    frac = np.mean(np.abs(g) > 6e-3)
    assert abs(frac / (0.01 * 0.95216) - 1.0) < 0.05
    core = g[np.abs(g) < 6e-3]
    assert abs(np.std(core) / 1e-3 - 1.0) < 0.02


def test_normal_gradients_and_weights():
    g = synth.draw_grads([(1000, 1000)], "normal", seed=0, step=0)[0].astype(np.float64)
    assert abs(np.std(g) - 1.0) < 5e-3 and abs(np.mean(g)) < 5e-3
    w = synth.init_weights([(1000, 1000)], seed=1)[0].astype(np.float64)
    assert abs(np.std(w) / 0.02 - 1.0) < 5e-3


def test_draws_are_seeded_and_fresh_per_step_and_tensor():
    a = synth.draw_grads([(64, 64), (64, 64)], "student_t", seed=0, step=3)
    b = synth.draw_grads([(64, 64), (64, 64)], "student_t", seed=0, step=3)
    c = synth.draw_grads([(64, 64), (64, 64)], "student_t", seed=0, step=4)
    assert all(np.array_equal(x, y) for x, y in zip(a, b))
    assert not np.array_equal(a[0], c[0])
    assert not np.array_equal(a[0], a[1])
