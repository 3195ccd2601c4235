"""Layer-sharded Muon (Section 5.4) through the C ABI on one GPU: the ranks
are emulated by one optimizer state per rank, each over its own copy of the
parameters (nothing waits on another state), and the exchange of a Muon step
is a device copy of every matrix from its owner's copy to the others'.

With every matrix's Newton-Schulz tiles cut the same way in the sharded and
the single states (no split-K Gram tiles), the combined result equals a
single state's bit for bit: each rank's own matrices (Muon branch), its
momentum of the others' matrices (the momentum update alone), the Lion steps
and the vectors.  On a set where the Gram tiles of a rank are split along K
differently (the split depends on the launch's load), the momentum and the
vectors are still bit-identical and the matrices agree to the bf16 rounding
of fp32 sums taken in another order."""

import numpy as np
import pytest

from paper_2605_19811_gb300 import synth
from tests.lm_testutil import bits, host_tensor, rel_fro, stored_values

pytestmark = pytest.mark.gpu


def _run(shapes, world, steps, period=2):
    """Final (params, momenta) per emulated rank; world = 1 is the plain state."""
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    from paper_2605_19811_gb300 import shard
    W0 = synth.init_weights(shapes, seed=1)
    own = shard.owners(shapes, world) if world > 1 else [0 if len(s) == 2 else -1 for s in shapes]
    copies = [[host_tensor(w, "bf16").cuda() for w in W0] for _ in range(world)]
    opts = [L.LionMuon(copies[r], period=period, shard_rank=r, shard_world=world) for r in range(world)]
    for t in range(steps):
        g = [host_tensor(x, "bf16").cuda() for x in synth.draw_grads(shapes, "student_t", seed=0, step=t)]
        for o in opts:
            o.step(g, t)
        if world > 1 and shard.is_muon_step(t, period):
            for i, o in enumerate(own):
                if o >= 0:
                    for r in range(world):
                        if r != o:
                            copies[r][i].copy_(copies[o][i])
    torch.cuda.synchronize()
    out = []
    for r, o in enumerate(opts):
        assert o.status() == 0
        out.append(([p.clone() for p in copies[r]], [o.momentum(i).clone() for i in range(len(shapes))],
                    o.workspace_bytes()))
        o.close()
    return out, own


@pytest.mark.parametrize("world", [2, 4])
def test_sharded_states_equal_single_state(world):
    # at least 38 Gram tiles of 16 K blocks per launch (four 1024 x 1024
    # matrices per rank): no launch splits a Gram tile along K
    shapes = [(1024, 1024)] * 16 + [(1024,), (1, 1024)]
    single, _ = _run(shapes, 1, steps=3)
    (W1, M1, ws1), = single
    ranks, own = _run(shapes, world, steps=3)
    assert sorted(set(o for o in own if o >= 0)) == list(range(world))
    for W, M, ws in ranks:
        assert ws < ws1           # the NS workspace holds this rank's matrices only
        for a, b in zip(W, W1):
            np.testing.assert_array_equal(bits(a), bits(b))
        for a, b in zip(M, M1):
            np.testing.assert_array_equal(bits(a), bits(b))


def test_sharded_gpt_set_matches_single_state():
    shapes = synth.scaled_set("gpt_2l", layers=2, d=768, vocab=4096).shapes
    single, _ = _run(shapes, 1, steps=2)
    (W1, M1, _), = single
    ranks, own = _run(shapes, 3, steps=2)
    for W, M, _ in ranks:
        for i, (a, b) in enumerate(zip(W, W1)):
            if len(shapes[i]) == 2 and min(shapes[i]) > 1:
                assert rel_fro(stored_values(a), stored_values(b)) <= 2e-3
            else:
                np.testing.assert_array_equal(bits(a), bits(b))
        for a, b in zip(M, M1):
            np.testing.assert_array_equal(bits(a), bits(b))


def test_shard_config_checks():
    import torch
    from paper_2605_19811_gb300 import lionmuon as L
    p = [torch.zeros((64, 64), dtype=torch.bfloat16, device="cuda")]
    with pytest.raises(L.LionMuonError):
        L.LionMuon(p, shard_rank=2, shard_world=2)
    with pytest.raises(L.LionMuonError) as ei:
        L.LionMuon(p, shard_rank=0, shard_world=2, schedule=L.LM_SCHEDULE_STABLE_RANK)
    assert ei.value.status == 6
    o = L.LionMuon(p, shard_rank=1, shard_world=2)   # owns nothing: Muon steps update momentum only
    g = [torch.ones((64, 64), dtype=torch.bfloat16, device="cuda")]
    o.step(g, 0)
    torch.cuda.synchronize()
    assert o.status() == 0
    assert bool((p[0] == 0).all())
    assert float(o.momentum(0)[0, 0]) == pytest.approx(0.01, rel=1e-6)   # (1 - beta2) g
    o.close()
