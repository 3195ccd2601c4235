"""Shared helpers for the GPU parity tests: move seeded host inputs to the
device, run the CUDA library through its C ABI, and run the oracle on the very
same stored values."""

import numpy as np

import oracle as O
from paper_2605_19811_gb300 import synth


def torch_dtype(name):
    import torch
    return {"bf16": torch.bfloat16, "f32": torch.float32}[name]


def host_tensor(a: np.ndarray, dtype: str):
    """CPU torch tensor holding ``a`` rounded to the storage dtype."""
    import torch
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch_dtype(dtype))


def stored_values(t) -> np.ndarray:
    """The exact stored values of a (CPU or CUDA) tensor as float64."""
    return t.detach().float().cpu().numpy().astype(np.float64)


def bits(t) -> np.ndarray:
    """Raw bit patterns of a bf16 / fp32 tensor."""
    import torch
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.view(torch.int32).numpy().view(np.uint32)


def rel_fro(a: np.ndarray, b: np.ndarray) -> float:
    den = np.linalg.norm(b)
    return float(np.linalg.norm(a - b) / (den if den > 0 else 1.0))


def oracle_config(**kw) -> O.Config:
    return O.Config(**kw)


def run_trajectory_gpu(W0, grads, dtype, cfg: dict, steps: int):
    """Create a state over device copies of W0, run ``steps`` steps with the
    given per-step host gradients; return (final W list, final M list)."""
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    params = [host_tensor(w, dtype).cuda() for w in W0]
    opt = L.LionMuon(params, **cfg)
    for t in range(steps):
        g = [host_tensor(x, dtype).cuda() for x in grads[t]]
        opt.step(g, t)
    torch.cuda.synchronize()
    Ws = [stored_values(p) for p in params]
    Ms = [stored_values(opt.momentum(i)) for i in range(len(params))]
    flags = opt.status()
    opt.close()
    return Ws, Ms, flags


def run_trajectory_oracle(W0, grads, dtype, cfg: O.Config, steps: int):
    """Storage-modelled oracle run on the same stored input values."""
    P = [stored_values(host_tensor(w, dtype)) for w in W0]
    M = [np.zeros_like(p) for p in P]
    dts = [dtype] * len(P)
    for t in range(steps):
        G = [stored_values(host_tensor(g, dtype)) for g in grads[t]]
        P, M = O.lionmuon_step(P, G, M, t, cfg, param_dtypes=dts)
    return P, M


def make_problem(shapes, grad_kind, steps, wseed=1, gseed=0, w_std=0.02):
    W0 = synth.init_weights(shapes, seed=wseed, std=w_std)
    grads = [synth.draw_grads(shapes, grad_kind, seed=gseed, step=t) for t in range(steps)]
    return W0, grads


def ns_closed_form_rows(G_hat: np.ndarray, steps: int, a: float, b: float, c: float, eps: float = 1e-7,
                        rows=None) -> np.ndarray:
    """NS_steps(G_hat) (Section 2's odd-polynomial iteration with the
    Frobenius pre-normalisation) through its closed form on the SVD, in fp64:
    with X0 = G_hat / (||G_hat||_F + eps) = U diag(s) V^T,
    NS(X0) = U diag(phi^K(s)) V^T = X0 V diag(phi^K(s) / s) V^T, computed
    in the tall orientation (a wide input as its transpose, NS(X^T) =
    NS(X)^T) from the eigen-decomposition of the small Gram X0^T X0.  Returns
    the rows ``rows`` (all if None) of the tall-orientation result, so a large
    matrix can be checked element-wise on a sample of its long dimension.
    Agrees with oracle.ns_polynomial to fp64 rounding (pinned on the CPU)."""
    import oracle as O
    X0 = np.asarray(G_hat, dtype=np.float64)
    X0 = X0 / (np.linalg.norm(X0) + eps)
    Xt = X0 if X0.shape[0] >= X0.shape[1] else X0.T
    lam, V = np.linalg.eigh(Xt.T @ Xt)
    sig = np.sqrt(np.clip(lam, 0.0, None))
    safe = np.where(sig > 0, sig, 1.0)
    f = np.where(sig > 0, O.ns_scalar_map(sig, steps, a, b, c) / safe, 0.0)
    Xr = Xt if rows is None else Xt[rows]
    return ((Xr @ V) * f) @ V.T


def tall(x: np.ndarray) -> np.ndarray:
    """The tall orientation of a matrix (its transpose if it is wide)."""
    return x if x.shape[0] >= x.shape[1] else x.T
