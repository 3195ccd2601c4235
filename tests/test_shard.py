"""Layer-sharded Muon (Section 5.4: a Muon step needs the whole matrix, a
Lion step is element-wise) on the CPU: the owner partition of the library
(lm_shard_owners, host code, no GPU) and the exchange protocol over gloo with
two ranks.

The partition: every matrix has exactly one owner, 1-D parameters none, the
same inputs give the same owners, and the largest-first greedy split keeps
the most loaded rank within 4/3 of the best split (Graham's bound for
longest-processing-time scheduling), checked against brute force on small
sets.  The protocol: two gloo ranks, each standing in for the library with
the oracle (Algorithm 1 for the matrices it owns, the momentum update alone
for the others, the Lion step for vectors), then the exchange, end with
weights and momentum equal bit for bit to a one-rank run of the oracle."""

import itertools
import os
import socket
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _cost(shape):
    s, l = min(shape), max(shape)
    return 3.0 * s * s * l + s ** 3


def test_owners_cover_every_matrix_once():
    from paper_2605_19811_gb300 import shard, synth
    shapes = synth.PARAM_SETS["gpt_720m"].shapes
    for world in (1, 2, 3, 4, 8):
        own = shard.owners(shapes, world)
        assert own == shard.owners(shapes, world)                # deterministic
        for s, o in zip(shapes, own):
            if len(s) == 2 and min(s) > 1:
                assert 0 <= o < world
            else:
                assert o == -1
        loads = [0.0] * world
        for s, o in zip(shapes, own):
            if o >= 0:
                loads[o] += _cost(s)
        biggest = max(_cost(s) for s, o in zip(shapes, own) if o >= 0)
        assert max(loads) - min(loads) <= biggest                 # greedy: within one matrix
        if world == 1:
            assert set(o for o in own if o >= 0) == {0}


@pytest.mark.parametrize("seed", range(6))
def test_owner_split_within_graham_bound(seed):
    """Brute force over all assignments of up to 8 matrices to 2 or 3 ranks."""
    from paper_2605_19811_gb300 import shard
    rng = np.random.default_rng(seed)
    n = int(rng.integers(4, 9))
    world = 2 + seed % 2
    shapes = [(int(rng.integers(2, 40)) * 32, int(rng.integers(2, 40)) * 32) for _ in range(n)] + [(1, 64)]
    own = shard.owners(shapes, world)
    costs = [_cost(s) for s in shapes[:-1]]
    got = max(sum(c for c, o in zip(costs, own) if o == r) for r in range(world))
    best = min(max(sum(c for c, a in zip(costs, asg) if a == r) for r in range(world))
               for asg in itertools.product(range(world), repeat=n))
    assert got <= (4.0 / 3.0 - 1.0 / (3 * world)) * best + 1e-6 * best
    assert own[-1] == -1


def test_owners_reject_bad_world():
    from paper_2605_19811_gb300 import lionmuon as L
    from paper_2605_19811_gb300 import shard
    for w in (0, 5000):
        with pytest.raises(L.LionMuonError):
            shard.owners([(4, 4)], w)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


SHAPES = [(64, 96), (96, 64), (128, 128), (32, 256), (256, 32), (48, 48), (96,), (1, 40)]


def _problem():
    sys.path.insert(0, ROOT)
    from paper_2605_19811_gb300 import synth
    W0 = synth.init_weights(SHAPES, seed=1)
    grads = [synth.draw_grads(SHAPES, "student_t", seed=0, step=t) for t in range(4)]
    return [np.asarray(w, np.float64) for w in W0], [[np.asarray(g, np.float64) for g in gs] for gs in grads]


def _worker(rank, world, port, q, flat):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import torch
    import torch.distributed as dist
    import oracle as O
    from paper_2605_19811_gb300 import shard
    dist.init_process_group("gloo", rank=rank, world_size=world)
    W0, grads = _problem()
    own = shard.owners(SHAPES, world)
    cfg = O.Config(period=2, eta_muon=3e-3, eta_lion=2e-5)
    if flat:
        # parameters as views of one buffer, each rank's matrices adjacent
        order = shard.owner_order(SHAPES, own)
        sizes = [int(np.prod(s)) for s in SHAPES]
        buf = torch.zeros(sum(sizes) + 64 * len(SHAPES), dtype=torch.float64)
        params, off = [None] * len(SHAPES), 0
        for i in order:
            params[i] = buf[off:off + sizes[i]].view(SHAPES[i])
            off += sizes[i]
    else:
        params = [torch.zeros(s, dtype=torch.float64) for s in SHAPES]
    for p, w in zip(params, W0):
        p.copy_(torch.from_numpy(w))
    ex = shard.Exchange(params, own)
    M = [np.zeros(s) for s in SHAPES]
    for t in range(4):
        for i, (p, g) in enumerate(zip(params, grads[t])):
            w = p.numpy().copy()
            if len(SHAPES[i]) == 2 and min(SHAPES[i]) > 1 and O.is_muon_step(t, cfg.period) and own[i] != rank:
                M[i] = O.momentum_update(M[i], g, cfg.beta2)        # another rank owns it
            else:
                w, M[i] = O.lionmuon_param_step(w, g, M[i], t, cfg)
                p.copy_(torch.from_numpy(w))
        if shard.is_muon_step(t, cfg.period):
            ex.run()
    q.put((rank, [p.numpy().copy() for p in params], M, len(ex.items)))
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.parametrize("flat", [False, True])
def test_two_ranks_match_one_rank(flat):
    import torch.multiprocessing as mp
    import oracle as O
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q, flat)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted((q.get(timeout=180) for _ in procs), key=lambda x: x[0])
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    W0, grads = _problem()
    cfg = O.Config(period=2, eta_muon=3e-3, eta_lion=2e-5)
    W, M = [w.copy() for w in W0], [np.zeros(s) for s in SHAPES]
    for t in range(4):
        for i in range(len(SHAPES)):
            W[i], M[i] = O.lionmuon_param_step(W[i], grads[t][i], M[i], t, cfg)
    for rank, Wr, Mr, nitems in out:
        for a, b in zip(Wr, W):
            np.testing.assert_array_equal(a, b)
        for a, b in zip(Mr, M):
            np.testing.assert_array_equal(a, b)
        if flat:
            assert nitems == 2          # one broadcast per owner rank
