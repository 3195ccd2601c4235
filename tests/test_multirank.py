"""Host-side logic of the multi-rank bench harness with gloo on the CPU
(world size 2): the max-over-ranks timing reduction, and the reference arm
printing only on rank 0.  (The layer-sharded exchange itself is covered by
test_shard.py.)"""

import io
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    got = bench.max_over_ranks(1.5 + rank, world, "cpu")
    # the reference arm runs and prints on rank 0 only
    bench.oracle_times = lambda name, period, which=None, table=None: (0.0, {})
    bench.oracle_estimate = lambda name, period, lion, times: 42.0

    class A:
        gpus, steps, warmup, set, period, ns_table = world, 1, 0, "gpt2_124m", 2, "quintic"
    buf = io.StringIO()
    with redirect_stdout(buf):
        rc = bench.run_reference(A)
    dist.barrier()
    dist.destroy_process_group()
    q.put((rank, got, rc, buf.getvalue()))


def test_max_over_ranks_and_rank0_printing():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, m0, rc0, s0), (r1, m1, rc1, s1) = out
    assert m0 == m1 == 2.5
    assert rc0 == rc1 == 0
    assert '"impl": "reference"' in s0 and '"value": 42.0' in s0
    assert s1 == ""
