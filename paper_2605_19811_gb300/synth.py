"""Seeded synthetic inputs: parameter-set shapes and random tensors.

This module holds no arithmetic of the optimizer.  It only names the tensor
shapes of the GPT-style parameter sets the step is measured on and draws
seeded random weights and gradients with the stated distributions.  Both the
CUDA path's tests/bench and the CPU oracle take their inputs from here.

Shapes (row-major, "out x in" as a linear layer stores them):

* ``tiny``  : fp32 256x256, 256x1024, 1024x256, 256x256 and one 256-vector.
* ``gpt2_124m`` : per layer (x12, d=768) two LayerNorm vectors, attention QKV
  768x2304, attention out 768x768, two LayerNorm vectors, MLP up 768x3072,
  MLP down 3072x768; a 50304x768 token embedding; a final LayerNorm pair.
* ``gpt_355m`` : the same with 24 layers, d=1024.
* ``gpt_720m`` : the same with 36 layers, d=1280.
* ``stress_7b`` : 32 layers of 4 x (4096x4096), 2 x (4096x14336) and
  1 x (14336x4096) (a 7B-style hidden set, 7.79 G parameters).

Distributions: weights N(0, 0.02^2); gradients N(0,1) (tiny), Student-t with
nu = 3 scaled to standard deviation 1e-3 (GPT sets), or N(0, 1e-3^2) with 1% of
entries multiplied by 100 (stress set).  Vectors are shape ``(n,)``.
"""

from __future__ import annotations

import dataclasses
from typing import List, Sequence, Tuple

import numpy as np

VOCAB = 50304


@dataclasses.dataclass(frozen=True)
class ParamSet:
    name: str
    shapes: Tuple[Tuple[int, ...], ...]
    dtype: str            # 'bf16' or 'f32' (storage dtype of W and G)
    grad_kind: str        # 'normal', 'student_t' or 'outlier'

    @property
    def numel(self) -> int:
        return int(sum(int(np.prod(s)) for s in self.shapes))

    @property
    def matrices(self) -> List[Tuple[int, int]]:
        return [s for s in self.shapes if len(s) == 2 and s[0] > 1 and s[1] > 1]


def _gpt(name: str, layers: int, d: int) -> ParamSet:
    shapes: List[Tuple[int, ...]] = [(VOCAB, d)]
    for _ in range(layers):
        shapes += [(d,), (d,), (d, 3 * d), (d, d), (d,), (d,), (d, 4 * d), (4 * d, d)]
    shapes += [(d,), (d,)]
    return ParamSet(name, tuple(shapes), "bf16", "student_t")


def _stress() -> ParamSet:
    shapes: List[Tuple[int, ...]] = []
    for _ in range(32):
        shapes += [(4096, 4096)] * 4 + [(4096, 14336)] * 2 + [(14336, 4096)]
    return ParamSet("stress_7b", tuple(shapes), "bf16", "outlier")


def _layers_only(name: str, layers: int, d: int) -> ParamSet:
    shapes: List[Tuple[int, ...]] = []
    for _ in range(layers):
        shapes += [(d, 3 * d), (d, d), (d, 4 * d), (4 * d, d)]
    return ParamSet(name, tuple(shapes), "bf16", "student_t")


PARAM_SETS = {
    "tiny": ParamSet("tiny", ((256, 256), (256, 1024), (1024, 256), (256, 256), (256,)),
                     "f32", "normal"),
    "gpt2_124m": _gpt("gpt2_124m", 12, 768),
    "gpt_355m": _gpt("gpt_355m", 24, 1024),
    "gpt_720m": _gpt("gpt_720m", 36, 1280),
    "stress_7b": _stress(),
    # four hidden layers of the 720M-shaped set (no embedding, no vectors):
    # a small case with the same matrix shapes, for profiling captures
    "gpt_720m_4layers": _layers_only("gpt_720m_4layers", 4, 1280),
}


def scaled_set(name: str, layers: int, d: int, vocab: int, dtype: str = "bf16",
               grad_kind: str = "student_t") -> ParamSet:
    """A GPT-style set with the same per-layer structure as the named sets but
    chosen sizes (for tests that must finish quickly on the CPU)."""
    shapes: List[Tuple[int, ...]] = [(vocab, d)]
    for _ in range(layers):
        shapes += [(d,), (d,), (d, 3 * d), (d, d), (d,), (d,), (d, 4 * d), (4 * d, d)]
    shapes += [(d,), (d,)]
    return ParamSet(name, tuple(shapes), dtype, grad_kind)


def _rng(*seed_words: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence(list(seed_words))))


def init_weights(shapes: Sequence[Tuple[int, ...]], seed: int = 1, std: float = 0.02) -> List[np.ndarray]:
    """W_0 ~ N(0, std^2), float32, one independent stream per tensor."""
    return [(_rng(seed, i).standard_normal(size=s, dtype=np.float32) * np.float32(std))
            for i, s in enumerate(shapes)]


def draw_grads(shapes: Sequence[Tuple[int, ...]], kind: str, seed: int = 0, step: int = 0) -> List[np.ndarray]:
    """Gradients for step ``step``, float32, fresh per step and per tensor."""
    out = []
    for i, s in enumerate(shapes):
        r = _rng(seed, step, i)
        if kind == "normal":
            g = r.standard_normal(size=s, dtype=np.float32)
        elif kind == "student_t":
            # Student-t, nu = 3 (variance 3), scaled to std 1e-3.
            g = (r.standard_t(3.0, size=s) * (1e-3 / np.sqrt(3.0))).astype(np.float32)
        elif kind == "outlier":
            g = r.standard_normal(size=s, dtype=np.float32) * np.float32(1e-3)
            mask = r.random(size=s) < 0.01
            g = np.where(mask, g * np.float32(100.0), g).astype(np.float32)
        else:
            raise ValueError(f"unknown gradient kind {kind!r}")
        out.append(g)
    return out


def draw_matrix(shape: Tuple[int, int], seed: int, kind: str = "normal") -> np.ndarray:
    """One float32 matrix for Newton-Schulz tests."""
    return draw_grads([shape], kind, seed=seed, step=0)[0]


def device_grads_torch(shapes, kind: str, seed: int, device, dtype):
    """Large gradient sets drawn on the device with torch's generator (same
    distributions as ``draw_grads``, different random stream).  Used where a
    host draw of hundreds of millions of values would dominate run time."""
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    out = []
    for s in shapes:
        if kind == "normal":
            g = torch.randn(s, generator=gen, device=device, dtype=torch.float32)
        elif kind == "student_t":
            z = torch.randn(s, generator=gen, device=device, dtype=torch.float32)
            chi = torch.zeros(s, device=device, dtype=torch.float32)
            for _ in range(3):
                e = torch.randn(s, generator=gen, device=device, dtype=torch.float32)
                chi.addcmul_(e, e)
            g = z * torch.rsqrt(chi / 3.0) * (1e-3 / 3.0 ** 0.5)
            del z, chi
        elif kind == "outlier":
            g = torch.randn(s, generator=gen, device=device, dtype=torch.float32) * 1e-3
            mask = torch.rand(s, generator=gen, device=device) < 0.01
            g = torch.where(mask, g * 100.0, g)
        else:
            raise ValueError(f"unknown gradient kind {kind!r}")
        out.append(g.to(dtype))
    return out


def device_weights_torch(shapes, seed: int, device, dtype, std: float = 0.02):
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    return [(torch.randn(s, generator=gen, device=device, dtype=torch.float32) * std).to(dtype)
            for s in shapes]
