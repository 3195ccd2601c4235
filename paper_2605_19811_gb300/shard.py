"""Layer-sharded Muon across ranks (Section 5.4: a Muon step needs each
matrix whole, a Lion step is element-wise).

Every rank holds all parameters, the already-reduced gradients and the
momentum, and runs the same ``lm_step``.  Each matrix has one owner rank
(``owners``, computed by the library's ``lm_shard_owners``): on a Muon step
a rank runs the momentum, Newton-Schulz and parameter write only for the
matrices it owns, and the momentum update alone for the others
(``lm_config.shard_rank`` / ``shard_world``).  ``exchange`` then copies each
matrix from its owner to every other rank, on Muon steps only; Lion steps
and 1-D parameters exchange nothing.  The Newton-Schulz work of a Muon step
is divided among the ranks, and the exchange moves the bf16 matrices once.

This module is plumbing over ``torch.distributed`` (NCCL on GPUs, gloo on
CPUs); the arithmetic stays in the library."""

from __future__ import annotations

import ctypes
from typing import List, Optional, Sequence

from . import lionmuon as _L


def _shape_desc(shape, dtype_code: int) -> _L.LmTensor:
    if len(shape) == 1:
        rows, cols = 1, int(shape[0])
    elif len(shape) == 2:
        rows, cols = int(shape[0]), int(shape[1])
    else:
        raise ValueError("parameters must be 1-D or 2-D")
    return _L.LmTensor(ctypes.c_void_p(0), rows, cols, dtype_code)


def owners(shapes: Sequence, world: int) -> List[int]:
    """Owner rank of each parameter (shapes: tuples, or tensors), -1 for 1-D
    parameters; the same on every rank.  No device access."""
    lib = _L.load_library()
    shp = [tuple(s.shape) if hasattr(s, "shape") else tuple(s) for s in shapes]
    n = len(shp)
    descs = (_L.LmTensor * n)(*[_shape_desc(s, _L.LM_BF16) for s in shp])
    out = (ctypes.c_int * n)()
    _L._check(lib, lib.lm_shard_owners(descs, n, int(world), out), "lm_shard_owners")
    return [int(x) for x in out]


class Exchange:
    """The copies of one layer-sharded Muon step: rank r broadcasts the
    matrices it owns.  Where a rank's matrices are adjacent in memory (the
    layout ``owner_order`` gives) they go as one contiguous broadcast, so the
    exchange is one collective per rank; otherwise one per matrix."""

    def __init__(self, params: Sequence, owner: Sequence[int], group=None):
        import torch
        self.group = group
        self.items = []          # (tensor to broadcast, owner rank)
        spans = [(t.data_ptr(), t.data_ptr() + t.numel() * t.element_size()) for t in params]
        by_owner = {}
        for i, o in enumerate(owner):
            if o >= 0:
                by_owner.setdefault(o, []).append(i)
        for o in sorted(by_owner):
            ids = sorted(by_owner[o], key=lambda i: spans[i][0])
            ps = [params[i] for i in ids]
            lo, hi = spans[ids[0]][0], spans[ids[-1]][1]
            # one broadcast over the rank's whole range: the tensors are
            # contiguous, of one dtype and storage, apart by alignment padding
            # only, and no other parameter lies in the range
            one = (len(ps) > 1 and all(t.is_contiguous() and t.dtype == ps[0].dtype for t in ps) and
                   all(t.untyped_storage().data_ptr() == ps[0].untyped_storage().data_ptr() for t in ps) and
                   all(0 <= spans[b][0] - spans[a][1] < 256 for a, b in zip(ids, ids[1:])) and
                   not any(lo <= spans[j][0] < hi for j in range(len(params)) if j not in set(ids)))
            if one:
                es = ps[0].element_size()
                flat = torch.empty(0, dtype=ps[0].dtype, device=ps[0].device).set_(
                    ps[0].untyped_storage(), ps[0].storage_offset(), ((hi - lo) // es,), (1,))
                self.items.append((flat, o))
            else:
                self.items.extend((t, o) for t in ps)
        self.bytes_per_owner = {}
        for t, o in self.items:
            self.bytes_per_owner[o] = self.bytes_per_owner.get(o, 0) + t.numel() * t.element_size()

    def received_bytes(self, rank: int) -> int:
        """Bytes rank ``rank`` receives per Muon step (the matrices others own)."""
        return sum(b for o, b in self.bytes_per_owner.items() if o != rank)

    def run(self) -> None:
        """Broadcast every matrix from its owner (blocking until done)."""
        import torch.distributed as dist
        works = []
        for t, o in self.items:
            src = dist.get_global_rank(self.group, o) if self.group is not None else o
            works.append(dist.broadcast(t, src=src, group=self.group, async_op=True))
        for w in works:
            w.wait()


def exchange(params: Sequence, owner: Sequence[int], group=None) -> None:
    """One-off form of ``Exchange(params, owner, group).run()``."""
    Exchange(params, owner, group).run()


def owner_order(shapes: Sequence, owner: Sequence[int]) -> List[int]:
    """Parameter indices ordered for allocation so that each rank's matrices
    are adjacent (rank 0's first, then rank 1's, ...; 1-D parameters last)."""
    idx = list(range(len(shapes)))
    return sorted(idx, key=lambda i: (owner[i] if owner[i] >= 0 else 1 << 30, i))


def is_muon_step(t: int, period: int) -> bool:
    """Algorithm 1's dispatch: a Muon step iff period != 0 and t mod period == 0."""
    return period != 0 and t % period == 0


def step(opt: "_L.LionMuon", grads: Sequence, t: int, ex: Optional[Exchange], period: int, stream=None) -> None:
    """One layer-sharded LionMuon step: ``lm_step`` on this rank, then on a
    Muon step the exchange.  The collectives are ordered after the work on
    torch's current stream; a step run on another stream is joined to it
    first."""
    import torch
    opt.step(grads, t, stream)
    if ex is not None and is_muon_step(t, period):
        if stream is not None:
            torch.cuda.current_stream().wait_stream(stream)
        ex.run()
