"""lm_step captured into CUDA graphs: replaying one graph per step phase
(t mod P) gives the same trajectory as calling lm_step eagerly, for the
periodic schedule of Algorithm 1 (Muon on t % P == 0, Lion otherwise) and for
the stable-rank schedule of Appendix G, whose power-iteration launches run on
side streams forked from and joined to the capturing stream (an unjoined
fork would make the capture fail).  Also: eager steps after a replay use
their own gradients (the pointer table is re-uploaded after a capture), and
the AdamW rule, which uses t itself, is refused."""

import pytest

torch = pytest.importorskip("torch")

from paper_2605_19811_gb300 import lionmuon as L
from paper_2605_19811_gb300 import synth

pytestmark = pytest.mark.gpu

# rows of 256-1024, 1280 and 3072 columns: three power-iteration launches per
# pass under the stable-rank schedule, so its side streams take part
SHAPES = [(256, 768), (768, 256), (512, 512), (384, 1280), (256, 3072), (1024,)]


def _setup(seed=1):
    dev = torch.device("cuda", 0)
    params = synth.device_weights_torch(SHAPES, seed, dev, torch.bfloat16)
    grads = [synth.device_grads_torch(SHAPES, "student_t", 100 + t, dev, torch.bfloat16) for t in range(6)]
    return dev, params, grads


def _same_state(pa, pb, oa, ob):
    for i, (a, b) in enumerate(zip(pa, pb)):
        # momentum: the same fp32 EMA on both sides
        assert torch.equal(oa.momentum(i), ob.momentum(i)), i
        # parameters: identical kernels; the Frobenius norm is summed with
        # atomics, so allow rounding-level differences
        d = (a.float() - b.float()).norm() / a.float().norm().clamp_min(1e-30)
        assert d.item() <= 1e-6, (i, d.item())


@pytest.mark.parametrize("period", [2, 3])
def test_graph_replay_matches_eager_periodic(period):
    dev, params, grads = _setup()
    pa = [p.clone() for p in params]
    pb = [p.clone() for p in params]
    oa = L.LionMuon(pa, period=period)
    ob = L.LionMuon(pb, period=period)
    gbuf = [torch.empty_like(g) for g in grads[0]]
    graphs = ob.capture_steps(gbuf, 0)
    assert len(graphs) == period
    for t in range(6):
        oa.step(grads[t], t)
        for dst, src in zip(gbuf, grads[t]):
            dst.copy_(src)
        graphs[t % period].replay()
    torch.cuda.synchronize()
    assert oa.status() == 0 and ob.status() == 0
    _same_state(pa, pb, oa, ob)
    oa.close(); ob.close()


def test_graph_replay_matches_eager_stable_rank():
    dev, params, grads = _setup(seed=3)
    pa = [p.clone() for p in params]
    pb = [p.clone() for p in params]
    kw = dict(schedule=L.LM_SCHEDULE_STABLE_RANK, srank_alpha=0.01)
    oa = L.LionMuon(pa, **kw)
    ob = L.LionMuon(pb, **kw)
    gbuf = [torch.empty_like(g) for g in grads[0]]
    graphs = ob.capture_steps(gbuf, 0)
    assert len(graphs) == 1
    for t in range(4):
        oa.step(grads[t], t)
        for dst, src in zip(gbuf, grads[t]):
            dst.copy_(src)
        graphs[0].replay()
        torch.cuda.synchronize()
        assert oa.selection()[0] == ob.selection()[0], t
    assert oa.status() == 0 and ob.status() == 0
    _same_state(pa, pb, oa, ob)
    oa.close(); ob.close()


def test_eager_step_after_replay_uses_its_own_gradients():
    """Eager steps and replays interleaved: an eager step reuses the buffer of
    the eager step before it, with a replay (which rewrites the device's
    gradient-pointer table) in between."""
    dev, params, grads = _setup(seed=5)
    pa = [p.clone() for p in params]
    pb = [p.clone() for p in params]
    oa = L.LionMuon(pa, period=2)
    ob = L.LionMuon(pb, period=2)
    gbuf = [torch.empty_like(g) for g in grads[0]]
    ebuf = [torch.empty_like(g) for g in grads[0]]
    graphs = ob.capture_steps(gbuf, 0)
    for t in range(4):
        oa.step(grads[t], t)
        if t % 2 == 0:      # eager, always from ebuf
            for dst, src in zip(ebuf, grads[t]):
                dst.copy_(src)
            ob.step(ebuf, t)
        else:               # replay, from gbuf
            for dst, src in zip(gbuf, grads[t]):
                dst.copy_(src)
            graphs[1].replay()
    torch.cuda.synchronize()
    assert oa.status() == 0 and ob.status() == 0
    _same_state(pa, pb, oa, ob)
    oa.close(); ob.close()


def test_capture_refuses_adamw_and_misaligned_start():
    dev, params, grads = _setup()
    o = L.LionMuon([p.clone() for p in params], vector_rule=L.LM_VECTOR_ADAMW)
    with pytest.raises(ValueError):
        o.capture_steps(grads[0], 0)
    o.close()
    o = L.LionMuon([p.clone() for p in params], period=2)
    with pytest.raises(ValueError):
        o.capture_steps(grads[0], 1)
    o.close()


def test_capture_with_profiling_on_records_no_events():
    """Profiling left on during a capture: the captured launches are not
    timed, and eager steps afterwards are."""
    dev, params, grads = _setup(seed=7)
    o = L.LionMuon([p.clone() for p in params], period=2)
    o.profile(True)
    graphs = o.capture_steps(grads[0], 0)
    graphs[0].replay()
    graphs[1].replay()
    torch.cuda.synchronize()
    prof = o.profile_read()
    assert all(v[1] == 0 for v in prof.values()), prof
    o.step(grads[1], 2)
    prof = o.profile_read()
    assert prof["ns_gemm"][1] > 0 and prof["lion"][1] > 0
    assert o.status() == 0
    o.close()
