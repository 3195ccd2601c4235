"""GPU parity of the Newton-Schulz msign approximation (lm_msign_ns) against
the fp64 oracle recurrence on the same stored input: relative Frobenius error
<= 2e-2 for the bf16 tensor-core path, <= 1e-5 for the fp32 CUDA-core path and
<= 2e-5 for the three-piece tensor-core mode (LM_NS_F32_TC: each fp32 operand
is exactly hi + mid + lo in bf16, the dropped piece products are of order
2^-24 relative, and what remains is the tensor cores' fp32 accumulation, which
loses about a unit of the last place per MMA; with the largest products in an
accumulator of their own it measures 1.3e-6 - 1.8e-5 up to 768 x 50304 and
4096 x 4096, at most 5.8e-6 on the 1280-wide shapes)."""

import numpy as np
import pytest

import oracle as O
from paper_2605_19811_gb300 import synth
from tests.lm_testutil import host_tensor, rel_fro, stored_values

pytestmark = pytest.mark.gpu

TOL = {"bf16": 2e-2, "f32": 1e-5, "f32tc": 2e-5}


def _prec(L, precision):
    return {"bf16": L.LM_BF16, "f32": L.LM_F32, "f32tc": L.LM_NS_F32_TC}[precision]
QUINTIC = O.NS_QUINTIC


def _msign(x_host, precision, steps=5, coeffs=QUINTIC, eps=1e-7, out_dtype="f32"):
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    x = x_host.cuda()
    out = torch.empty(x.shape, dtype={"f32": torch.float32, "bf16": torch.bfloat16}[out_dtype],
                      device="cuda")
    L.msign_ns(x, out, steps, *coeffs, eps=eps, precision=_prec(L, precision))
    torch.cuda.synchronize()
    return stored_values(out)


@pytest.mark.parametrize("precision", ["bf16", "f32", "f32tc"])
@pytest.mark.parametrize("shape", [(128, 256), (256, 128), (300, 700), (700, 300), (64, 64),
                                   (130, 1000), (1000, 130), (257, 257), (2, 3), (40, 9)])
def test_msign_parity_quintic(precision, shape):
    in_dtype = "bf16" if precision == "bf16" else "f32"
    xh = host_tensor(synth.draw_matrix(shape, seed=sum(shape)), in_dtype)
    got = _msign(xh, precision)
    want = O.ns_polynomial(stored_values(xh), 5, *QUINTIC, 1e-7)
    assert got.shape == want.shape
    assert rel_fro(got, want) <= TOL[precision]


@pytest.mark.parametrize("precision", ["bf16", "f32", "f32tc"])
@pytest.mark.parametrize("coeffs,steps", [((0.0, 1.0, 0.0), 1), ((0.0, 0.0, 1.0), 1),
                                          ((1.5, -0.5, 0.0), 8), ((2.0, -1.3, 0.4), 3),
                                          (QUINTIC, 0), (QUINTIC, 1)])
def test_msign_parity_each_term(precision, coeffs, steps):
    """(0,1,0): X X^T X isolates the Gram + apply GEMMs; (0,0,1): A A X
    isolates the polynomial GEMM; steps = 0 is the normalisation alone."""
    shape = (384, 640)
    in_dtype = "bf16" if precision == "bf16" else "f32"
    xh = host_tensor(synth.draw_matrix(shape, seed=7), in_dtype)
    got = _msign(xh, precision, steps=steps, coeffs=coeffs)
    want = O.ns_polynomial(stored_values(xh), steps, *coeffs, 1e-7)
    assert rel_fro(got, want) <= TOL[precision]


@pytest.mark.parametrize("precision", ["bf16", "f32", "f32tc"])
def test_msign_known_svd_closed_form(precision):
    """Input with exactly known SVD: output = U phi^K(sigma/||sigma||) V^T."""
    from tests.test_oracle_pins import known_svd_matrix
    s, l = 64, 256
    sigma = np.linspace(2.0, 0.2, s)
    G, U, V = known_svd_matrix(s, l, sigma, seed=3, tall=False)
    xh = host_tensor(G.astype(np.float32), "f32")
    Gs = stored_values(xh)
    got = _msign(xh, precision)
    phi = O.ns_scalar_map(sigma / (np.linalg.norm(sigma) + 1e-7), 5, *QUINTIC)
    want = U @ np.diag(phi) @ V.T
    assert rel_fro(got, want) <= TOL[precision] + rel_fro(Gs, G) * 10


def test_msign_bf16_output_dtype():
    xh = host_tensor(synth.draw_matrix((200, 500), seed=9), "bf16")
    got = _msign(xh, "bf16", out_dtype="bf16")
    want = O.ns_polynomial(stored_values(xh), 5, *QUINTIC, 1e-7)
    assert rel_fro(got, want) <= 2e-2


def test_msign_cubic_converges_to_svd_msign_fp32():
    r = np.random.default_rng(4)
    s, l = 96, 200
    U, _ = np.linalg.qr(r.standard_normal((s, s)))
    V, _ = np.linalg.qr(r.standard_normal((l, s)))
    G = (U @ np.diag(np.linspace(1.0, 0.5, s)) @ V.T).astype(np.float32)
    xh = host_tensor(G, "f32")
    got = _msign(xh, "f32", steps=40, coeffs=O.NS_CUBIC)
    assert rel_fro(got, O.msign_svd(stored_values(xh))) <= 1e-5


def test_msign_repeat_calls_identical():
    """The workspace is reused through the stream-ordered pool: two calls on
    the same input give the same bits."""
    xh = host_tensor(synth.draw_matrix((300, 520), seed=2), "bf16")
    a = _msign(xh, "bf16")
    b = _msign(xh, "bf16")
    np.testing.assert_array_equal(a, b)


MIXED_TABLE = ((3.0, -3.2, 1.2), (2.0, -1.5, 0.45), (1.875, -1.25, 0.375))
# cubic (c = 0: no polynomial launch, APPLY reads A) and quintic iterations in turn
CUBIC_QUINTIC_TABLE = ((1.5, -0.5, 0.0), QUINTIC, (1.5, -0.5, 0.0), QUINTIC, (1.5, -0.5, 0.0))


def table_tolerance(x, table, precision):
    """NS tolerance for a coefficient table.  bf16: the stated 2e-2, or 1.5
    times the distance that storing the intermediates in bf16 alone puts
    between the oracle's storage-modelled recurrence and its exact one,
    whichever is larger (aggressive first polynomials, the minimax tables
    start near 8.5 x, amplify rounding of small singular values; the
    storage-modelled oracle measures by how much for this input, independently
    of the GPU).  The fp32 modes: the stated tolerance, which holds for the
    constant quintic, times the factor by which the table amplifies fp32-size
    roundings more than the quintic does on the same input (the ratio of the
    two storage-modelled distances in fp32; about 2 for Polar Express), or 1.5
    times the table's own fp32 distance, whichever is larger."""
    if precision == "bf16":
        d = rel_fro(O.ns_polynomial_schedule_storage(x, table, 1e-7, "bf16"), O.ns_polynomial_schedule(x, table, 1e-7))
        return max(TOL[precision], 1.5 * d)
    quintic = [O.NS_QUINTIC] * 5
    d = rel_fro(O.ns_polynomial_schedule_storage(x, table, 1e-7, "f32"), O.ns_polynomial_schedule(x, table, 1e-7))
    dq = rel_fro(O.ns_polynomial_schedule_storage(x, quintic, 1e-7, "f32"),
                 O.ns_polynomial_schedule(x, quintic, 1e-7))
    return max(TOL[precision] * max(1.0, d / dq), 1.5 * d)


def _table(name):
    from paper_2605_19811_gb300 import ns_coeffs as C
    return {"polar_express": C.polar_express(5, 1e-3), "chebyshev_cubic": C.chebyshev_cubic(6, 1e-3),
            "mixed": MIXED_TABLE, "cubic_quintic": CUBIC_QUINTIC_TABLE}[name]


@pytest.mark.parametrize("precision", ["bf16", "f32", "f32tc"])
@pytest.mark.parametrize("name", ["polar_express", "chebyshev_cubic", "mixed", "cubic_quintic"])
@pytest.mark.parametrize("shape", [(256, 768), (768, 256), (300, 130), (64, 64)])
def test_msign_coefficient_table_parity(precision, name, shape):
    """Iteration-dependent coefficients (lm_msign_ns_coeffs) against the
    oracle's NS recurrence with the same table."""
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    table = _table(name)
    in_dtype = "bf16" if precision == "bf16" else "f32"
    xh = host_tensor(synth.draw_matrix(shape, seed=11 + sum(shape)), in_dtype)
    x = xh.cuda()
    out = torch.empty(x.shape, dtype=torch.float32, device="cuda")
    L.msign_ns_coeffs(x, out, table, precision=_prec(L, precision))
    torch.cuda.synchronize()
    want = O.ns_polynomial_schedule(stored_values(xh), table, 1e-7)
    assert rel_fro(stored_values(out), want) <= table_tolerance(stored_values(xh), table, precision)


def test_msign_coefficient_table_argument_errors():
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    x = torch.zeros((32, 48), device="cuda")
    out = torch.empty_like(x)
    with pytest.raises(L.LionMuonError) as e:
        L.msign_ns_coeffs(x, out, [(1.0, float("nan"), 0.0)])
    assert e.value.status == 1
    with pytest.raises(L.LionMuonError):
        L.msign_ns_coeffs(x, out, [(1.0, 0.0, 0.0)] * 65)


@pytest.mark.parametrize("coeffs", [QUINTIC, (1.5, -0.5, 0.0)])
@pytest.mark.parametrize("precision", ["bf16", "f32tc"])
@pytest.mark.parametrize("shape", [(200, 20000), (20000, 200), (768, 50304)])
def test_msign_parity_long_k_split_gram(shape, precision, coeffs):
    """A matrix whose Gram tiles are far longer than a CTA pair's share of
    the launch: the Gram phase splits them along K into parts that add fp32
    partial sums (split-K; in the three-piece mode the finish kernel writes
    the sum as three bf16 planes); the result must match the oracle.  With
    the cubic (c = 0) no polynomial launch runs and APPLY reads the A the
    finish kernel wrote."""
    xh = host_tensor(synth.draw_matrix(shape, seed=5 + shape[0]), "bf16" if precision == "bf16" else "f32")
    got = _msign(xh, precision, coeffs=coeffs)
    want = O.ns_polynomial(stored_values(xh), 5, *coeffs, 1e-7)
    assert rel_fro(got, want) <= TOL[precision]


@pytest.mark.parametrize("shape", [(300, 700), (700, 300), (130, 1000), (512, 2048)])
def test_msign_three_piece_mode_agrees_with_fp32_path(shape):
    """The two fp32 modes (CUDA cores, three-piece tensor cores) give the same
    output within the three-piece tolerance, and both are far closer to the
    exact recurrence than the bf16 tolerance."""
    xh = host_tensor(synth.draw_matrix(shape, seed=3 * shape[0] + shape[1]), "f32")
    a = _msign(xh, "f32")
    b = _msign(xh, "f32tc")
    assert rel_fro(b, a) <= TOL["f32tc"]


def test_msign_three_piece_mode_not_in_noalloc_entry():
    """lm_msign_ns_noalloc serves LM_BF16 and LM_F32 only."""
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    x = torch.zeros((32, 48), device="cuda")
    out = torch.empty_like(x)
    with pytest.raises(L.LionMuonError) as e:
        L.msign_ns_noalloc(x, out, 5, *QUINTIC, precision=L.LM_NS_F32_TC)
    assert e.value.status == 1
