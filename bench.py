#!/usr/bin/env python
"""Benchmark of the LionMuon optimizer step on one GB300 per rank.

A step is one lm_step over the whole parameter set (a Muon step when
t mod P == 0, otherwise a Lion step).  The headline value is the
period-averaged optimizer time per step (P = 2 by default) on the 720M-shaped
GPT parameter set, inputs resident in HBM, timed with CUDA events over whole
periods.  Prints one JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Under torchrun the N ranks share one parameter set by layer sharding
(Section 5.4): every rank holds all parameters, gradients and momentum and
runs the same step, each matrix's Muon update (momentum, Newton-Schulz,
parameter write) runs on its owner rank only, and after every Muon step each
rank broadcasts the matrices it owns (NCCL, inside the timed region).  The
work per step is fixed as N grows (strong scaling); the time is the max over
ranks.  ``--impl reference`` times the CPU oracle on bounded samples of the
same workload instead (rank 0 only).
"""

from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = ("period-averaged optimizer ms/step (P=2) per param set; Lion HBM GB/s; "
          "NS tensor-pipe %")
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=8)
    ap.add_argument("--warmup", type=int, default=4)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--set", default="gpt_720m")
    ap.add_argument("--period", type=int, default=2)
    ap.add_argument("--precision", choices=["bf16", "f32", "f32tc"], default="bf16",
                    help="NS precision: bf16 tensor cores, fp32 CUDA cores, or fp32 values as three "
                         "bf16 pieces on the tensor cores")
    ap.add_argument("--schedule", choices=["period", "srank"], default="period",
                    help="period: Algorithm 1's fixed P; srank: Appendix G's stable-rank selection")
    ap.add_argument("--srank-alpha", type=float, default=0.01)
    ap.add_argument("--srank-iters", type=int, default=5)
    ap.add_argument("--vector-rule", choices=["lion", "adamw"], default="lion",
                    help="1-D parameters: the Lion step, or the AdamW fallback of Section 3")
    ap.add_argument("--ns-table", choices=["quintic", "polar_express", "chebyshev3"], default="quintic",
                    help="Newton-Schulz coefficients: the constant quintic, or a per-iteration minimax table "
                         "(degree 5 Polar Express, degree 3 Chebyshev-type)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-graph", action="store_true",
                    help="skip timing the same steps replayed from CUDA graphs")
    ap.add_argument("--cublas-context", action="store_true",
                    help="also time the same NS iterations in torch.bmm/baddbmm (cuBLAS) for context")
    ap.add_argument("--no-cpu", action="store_true")
    return ap.parse_args()


# ---------------------------------------------------------------------------
# workload description (shared by both arms)
# ---------------------------------------------------------------------------

def workload(name):
    from paper_2605_19811_gb300 import synth
    ps = synth.PARAM_SETS[name]
    shapes = [tuple(s) for s in ps.shapes]
    mats = [s for s in shapes if len(s) == 2 and s[0] > 1 and s[1] > 1]
    numel = sum(int(math.prod(s)) for s in shapes)
    mat_elems = sum(a * b for a, b in mats)
    return ps, shapes, mats, numel, mat_elems


def ns_flops_sym(mats, steps=5, poly_steps=None):
    """Algorithmic FLOPs of NS_K per Muon step, symmetric products counted
    once: per iteration 3 s^2 l + s^3 per matrix (s = min, l = max), the s^3
    of A A only in the poly_steps iterations whose c is not 0 (all of them
    if None)."""
    poly_steps = steps if poly_steps is None else poly_steps
    tot = 0.0
    for a, b in mats:
        s, l = min(a, b), max(a, b)
        tot += steps * 3.0 * s * s * l + poly_steps * 1.0 * s ** 3
    return tot


def ns_table(name):
    """(table or None, iterations with c != 0) for --ns-table."""
    from paper_2605_19811_gb300 import ns_coeffs
    if name == "quintic":
        return None, 5
    table = {"polar_express": ns_coeffs.polar_express, "chebyshev3": ns_coeffs.chebyshev_cubic}[name](5)
    return table, sum(1 for t in table if t[2] != 0.0)


def cublas_ns_context(mats, dev, reps=5):
    """Context only, not the library's path: the same five NS iterations in
    torch.bmm / torch.baddbmm (cuBLAS) on the set's matrices (wide
    orientation, batched per shape), bf16 operands: A = X X^T, B = b A + c A A,
    X = a X + B X, with the symmetric products computed in full.  Returns ms
    per Muon step's NS (CUDA events, after warm-up)."""
    import torch
    a, b, c = 3.4445, -4.7750, 2.0315
    groups = {}
    for m, n in mats:
        key = (min(m, n), max(m, n))
        groups[key] = groups.get(key, 0) + 1
    bufs = []
    for (sm, lg), cnt in groups.items():
        x = torch.randn(cnt, sm, lg, device=dev, dtype=torch.bfloat16) / math.sqrt(sm * lg)
        bufs.append([x, torch.empty_like(x), torch.empty(cnt, sm, sm, device=dev, dtype=torch.bfloat16),
                     torch.empty(cnt, sm, sm, device=dev, dtype=torch.bfloat16)])

    def ns():
        for buf in bufs:
            for _ in range(5):
                x, y, A, B = buf
                torch.bmm(x, x.transpose(1, 2), out=A)
                torch.baddbmm(A, A, A, beta=b, alpha=c, out=B)
                torch.baddbmm(x, B, x, beta=a, alpha=1.0, out=y)
                buf[0], buf[1] = y, x
    for _ in range(2):
        ns()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        ns()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    del bufs
    torch.cuda.empty_cache()
    return ms


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured (MEASURED_PEAKS.json)"
    return dict(FALLBACK_PEAKS), "fallback"


def kernel_traffic(kernel: str):
    """DRAM bytes per launch of ``kernel`` from the committed ncu summary, if
    the kernel source still matches the hash recorded with it."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.txt")
    if not os.path.exists(path):
        return None
    for line in open(path):
        parts = line.split()
        if len(parts) >= 4 and parts[0] == kernel and not line.startswith("#"):
            src = os.path.join(ROOT, "paper_2605_19811_gb300", "csrc", parts[1])
            if not os.path.exists(src):
                return None
            h = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
            if h != parts[2]:
                return None
            return float(parts[3])
    return None


class ClockSampler:
    """nvidia-smi clock/throttle samples while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-f", self.path], stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        rows = []
        try:
            for line in open(self.path):
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
            os.unlink(self.path)
        except Exception:
            return None
        if not rows:
            return None
        def num(x):
            try:
                return float(x)
            except ValueError:
                return float("nan")
        sm = [num(r[1]) for r in rows]
        mx = [num(r[2]) for r in rows]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if "Active" in r[5 + i] and "Not" not in r[5 + i]})
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": reasons,
                "samples": len(rows), "power_w_max": max(num(r[3]) for r in rows)}


# ---------------------------------------------------------------------------
# CPU oracle timing (cpu_baseline leg and --impl reference)
# ---------------------------------------------------------------------------

def oracle_times(name, period, which=None, table=None):
    """Time the oracle: a Lion step on a 4 M-element vector sample, and a full
    fp64 Muon step (momentum, K_NS = 5 NS iterations, parameter update) of one
    matrix of each shape in ``which`` (every distinct matrix shape of the set,
    embedding included, if None).  Returns (Lion seconds per element,
    {shape: Muon-step seconds})."""
    import numpy as np
    import oracle as O
    _, _, mats, _, _ = workload(name)
    cfg = O.Config(period=period, ns_coeffs=table)
    rng = np.random.default_rng(0)
    n = 4_000_000
    W = rng.standard_normal(n) * 0.02
    G = rng.standard_normal(n) * 1e-3
    M = rng.standard_normal(n) * 1e-3
    t0 = time.perf_counter()
    O.lionmuon_param_step(W, G, M, 1, cfg)
    lion_per_elem = (time.perf_counter() - t0) / n
    del W, G, M
    times = {}
    for a, b in (sorted(set(mats)) if which is None else which):
        Wm = rng.standard_normal((a, b)) * 0.02
        Gm = rng.standard_normal((a, b)) * 1e-3
        Mm = np.zeros((a, b))
        t1 = time.perf_counter()
        O.lionmuon_param_step(Wm, Gm, Mm, 0, cfg)
        times[(a, b)] = time.perf_counter() - t1
        del Wm, Gm, Mm
    return lion_per_elem, times


def oracle_estimate(name, period, lion_per_elem, times):
    """Period-averaged ms/step of the whole set from sampled oracle times: each
    shape's Muon-step time once per matrix of that shape, the Lion time once
    per element (vectors take the Lion step on Muon steps too)."""
    _, _, mats, numel, mat_elems = workload(name)
    t_muon = lion_per_elem * (numel - mat_elems) + sum(times[tuple(m)] for m in mats)
    t_lion = lion_per_elem * numel
    return 1e3 * ((t_muon + (period - 1) * t_lion) / period if period > 0 else t_lion)


def oracle_sample(name, period, table=None):
    """(ms_per_step, description) of the oracle on the bounded sample of
    oracle_times over every matrix shape."""
    lion, times = oracle_times(name, period, table=table)
    _, _, mats, _, _ = workload(name)
    return oracle_estimate(name, period, lion, times), shape_counts(mats, times)


def shape_counts(mats, times):
    """'rows x cols (x count)' for each sampled shape."""
    counts = {}
    for m in mats:
        counts[tuple(m)] = counts.get(tuple(m), 0) + 1
    return ", ".join(f"{a}x{b} (x{counts[(a, b)]})" for a, b in sorted(times))


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


# ---------------------------------------------------------------------------
# the two arms
# ---------------------------------------------------------------------------

def max_over_ranks(value: float, world: int, device) -> float:
    """Max of a per-rank scalar over all ranks (the timing rule for N > 1)."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def run_reference(args):
    """The oracle timed on the host cores: all matrix shapes once (before the
    warm-up steps), then per step the Lion sample and one shape's Muon step in
    turn, so that the whole run stays within a few minutes; a step's value is
    the estimate from the latest time of every shape."""
    rank, world, local = dist_env()
    if rank != 0:
        return 0
    ps, shapes, mats, numel, mat_elems = workload(args.set)
    table, _ = ns_table(args.ns_table)
    lion, times = oracle_times(args.set, args.period, table=table)
    value = oracle_estimate(args.set, args.period, lion, times)
    desc = shape_counts(mats, times)
    order = sorted(times)
    vals = []
    for i in range(args.warmup + args.steps):
        which = [order[i % len(order)]] if order else []
        lion, t1 = oracle_times(args.set, args.period, which=which, table=table)
        times.update(t1)
        v = oracle_estimate(args.set, args.period, lion, times)
        if i >= args.warmup:
            vals.append(v)
    value = statistics.median(vals) if vals else value
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "ms/step",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": value, "higher_is_better": False, "scaling": "weak", "vs_baseline": None,
        "dtype": "f64", "data": "synthetic",
        "config": {"workload": args.set, "params": numel, "matrices": len(mats), "period": args.period,
                   "ns_steps": 5},
        "cpu_baseline": {"value": value, "unit": "ms/step", "cores": cpu_cores(), "kind": "oracle",
                         "sample": ("fp64 oracle: a full Muon step of one matrix of every shape "
                                    f"({desc}), timed once, then per step a 4M-element Lion step and "
                                    "one shape's Muon step in turn; each shape's latest time counted "
                                    "once per matrix of that shape, the Lion time per element "
                                    "(extrapolated)")},
        "e2e": {"value": value, "unit": "ms/step", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def run_ours(args):
    import torch
    import torch.distributed as dist
    from paper_2605_19811_gb300 import build as B
    from paper_2605_19811_gb300 import lionmuon as L
    from paper_2605_19811_gb300 import shard
    from paper_2605_19811_gb300 import synth

    rank, world, local = dist_env()
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if not os.path.exists(B.library_path()):
        B.build()
    L.load_library()

    ps, shapes, mats, numel, mat_elems = workload(args.set)
    P = args.period
    srank = args.schedule == "srank"
    sharded = world > 1
    if sharded and srank:
        raise SystemExit("the stable-rank schedule is not layer-sharded; run it on one GPU")
    owner = shard.owners(shapes, world) if sharded else [0 if len(s) == 2 and min(s) > 1 else -1 for s in shapes]
    own_mats = [s for s, o in zip(shapes, owner) if o == rank]
    # Parameters and gradients live in two flat device buffers (views per
    # tensor, 256-byte aligned) so that the end-to-end leg moves each with one
    # copy; sharded, each rank's matrices are adjacent, so that the exchange
    # is one broadcast per rank.
    elt = 2
    offs, cur = [0] * len(shapes), 0
    for i in (shard.owner_order(shapes, owner) if sharded else range(len(shapes))):
        offs[i] = cur
        cur += (int(math.prod(shapes[i])) * elt + 255) // 256 * 256
    flat_bytes = cur
    wflat = torch.empty(flat_bytes // 2, dtype=torch.bfloat16, device=dev)
    gflat = torch.empty(flat_bytes // 2, dtype=torch.bfloat16, device=dev)
    def views(flat):
        return [flat[o // 2: o // 2 + int(math.prod(s))].view(s) for o, s in zip(offs, shapes)]
    params, grads = views(wflat), views(gflat)
    # the same parameters and (already reduced) gradients on every rank
    for p, w in zip(params, synth.device_weights_torch(shapes, seed=1, device=dev, dtype=torch.bfloat16)):
        p.copy_(w)
    for g, x in zip(grads, synth.device_grads_torch(shapes, ps.grad_kind, seed=100, device=dev,
                                                     dtype=torch.bfloat16)):
        g.copy_(x)
    torch.cuda.synchronize()

    prec = {"bf16": L.LM_BF16, "f32": L.LM_F32, "f32tc": L.LM_NS_F32_TC}[args.precision]
    extra = {"vector_rule": L.LM_VECTOR_ADAMW} if args.vector_rule == "adamw" else {}
    if sharded:
        extra.update(shard_rank=rank, shard_world=world)
    table, poly_steps = ns_table(args.ns_table)
    if table is not None:
        extra["ns_coeffs"] = table
    if srank:
        opt = L.LionMuon(params, period=P, ns_precision=prec, schedule=L.LM_SCHEDULE_STABLE_RANK,
                         srank_alpha=args.srank_alpha, srank_iters=args.srank_iters, **extra)
    else:
        opt = L.LionMuon(params, period=P, ns_precision=prec, **extra)
    n = len(params)
    gdesc = (L.LmTensor * n)(*[L.tensor_desc(g) for g in grads])
    stream = torch.cuda.current_stream()
    sh = ctypes.c_void_p(stream.cuda_stream)
    ex = shard.Exchange(params, owner) if sharded else None

    def barrier():
        if world > 1:
            dist.barrier()

    def step(descs, t, handle):
        """One step; sharded, a Muon step ends with the exchange (NCCL waits
        for the step's work on torch's current stream, which it runs on)."""
        opt.step_descs(descs, n, t, handle)
        if ex is not None and shard.is_muon_step(t, P):
            ex.run()

    t = 0
    for _ in range(args.warmup):
        step(gdesc, t, sh)
        t += 1
    base = ((t + P - 1) // P) * P if P > 0 and not srank else t
    torch.cuda.synchronize()
    barrier()

    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    launches0 = L.kernel_launch_count()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    barrier()
    ev0.record(stream)
    for i in range(args.steps):
        step(gdesc, base + i, sh)
    ev1.record(stream)
    torch.cuda.synchronize()
    barrier()
    launches = L.kernel_launch_count() - launches0
    ms_total = max_over_ranks(ev0.elapsed_time(ev1), world, dev)
    ms_per_step = ms_total / args.steps
    value = ms_per_step          # one parameter set, whatever N

    # The same K steps again, from the same phase, with the library's
    # per-launch events on: the per-kernel split and the rooflines come from
    # this pass, so that its events stay out of the timed region above.
    base_p = base + (((args.steps + P - 1) // P) * P if P > 0 and not srank else args.steps)
    opt.profile(True)
    for i in range(args.steps):
        step(gdesc, base_p + i, sh)
    torch.cuda.synchronize()
    prof = opt.profile_read()
    opt.profile(False)
    base_g = base_p + (base_p - base)   # next aligned start, for the graph capture

    # ---- the same steps replayed from CUDA graphs, one per step phase ----
    # (t enters the Lion/Muon rules only mod P; AdamW's bias correction uses
    # t itself, so that rule is not captured)
    graph = None
    if not args.no_graph and args.vector_rule != "adamw" and not sharded:
        graphs = opt.capture_steps(grads, base_g)
        nph = len(graphs)
        for i in range(2 * nph):
            graphs[i % nph].replay()
        torch.cuda.synchronize()
        barrier()
        g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        g0.record(stream)
        for i in range(args.steps):
            graphs[i % nph].replay()
        g1.record(stream)
        torch.cuda.synchronize()
        barrier()
        g_ms = max_over_ranks(g0.elapsed_time(g1), world, dev) / args.steps
        graph = {"ms_per_step": g_ms,
                 "what": "the same K steps replayed from CUDA graphs of lm_step (one per phase t mod P), "
                         "captured once; inputs resident in HBM as for value"}
        del graphs

    # ---- end to end through the public API with host buffers ----
    # Every step copies its gradients in from pinned host memory and reads
    # the updated parameters back.  The copies are pipelined across steps:
    # the gradients of step t+1 go into a free device buffer (three in a
    # ring, so that the copy also overlaps a long Muon step followed by a
    # short Lion step) while earlier steps run; after step t a
    # device-to-device copy snapshots the parameters (W is updated in place
    # by step t+1), and the snapshot is read back to the host while step t+1
    # runs.  Warm-up steps run through the same pipeline before the timed
    # region, as in a training loop that reuses its buffers.  Sharded, a
    # Muon step's exchange is enqueued on the compute stream after the step
    # and before the snapshot, so the parameters read back are the exchanged
    # ones.
    e2e = None
    if not args.no_e2e:
        g_host = torch.empty(flat_bytes // 2, dtype=torch.bfloat16, pin_memory=True)
        w_host = torch.empty(flat_bytes // 2, dtype=torch.bfloat16, pin_memory=True)
        g_host.copy_(gflat)
        NG = 3
        gbufs = [gflat] + [torch.empty_like(gflat) for _ in range(NG - 1)]
        gdescs = [gdesc] + [(L.LmTensor * n)(*[L.tensor_desc(g) for g in views(gb)]) for gb in gbufs[1:]]
        snaps = (torch.empty_like(wflat), torch.empty_like(wflat))
        # three non-default streams: the legacy default stream would serialise them
        s_cmp, s_h2d, s_d2h = (torch.cuda.Stream(device=dev) for _ in range(3))
        sh_cmp = ctypes.c_void_p(s_cmp.cuda_stream)
        ev_in = [torch.cuda.Event() for _ in range(NG)]     # gradients of a buffer are in
        ev_used = [torch.cuda.Event() for _ in range(NG)]   # the step reading a buffer is done
        ev_snap = [torch.cuda.Event() for _ in range(2)]    # parameters copied into a snapshot
        ev_out = [torch.cuda.Event() for _ in range(2)]     # a snapshot read back to the host
        def pipelined(nsteps, t0):
            """nsteps pipelined steps from step t0; returns the (start, end) events on s_cmp."""
            ev_a, ev_b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            ev_a.record(s_cmp)
            s_h2d.wait_event(ev_a)
            with torch.cuda.stream(s_h2d):
                gbufs[0].copy_(g_host, non_blocking=True)
                ev_in[0].record(s_h2d)
            for i in range(nsteps):
                b, sb = i % NG, i & 1
                if i + 1 < nsteps:          # next step's gradients, once their buffer is free
                    nb = (i + 1) % NG
                    if i + 1 >= NG:
                        s_h2d.wait_event(ev_used[nb])
                    with torch.cuda.stream(s_h2d):
                        gbufs[nb].copy_(g_host, non_blocking=True)
                        ev_in[nb].record(s_h2d)
                s_cmp.wait_event(ev_in[b])
                opt.step_descs(gdescs[b], n, t0 + i, sh_cmp)
                if ex is not None and shard.is_muon_step(t0 + i, P):
                    with torch.cuda.stream(s_cmp):
                        ex.run()
                ev_used[b].record(s_cmp)
                if i >= 2:                  # the snapshot buffer's previous read-back is done
                    s_cmp.wait_event(ev_out[sb])
                with torch.cuda.stream(s_cmp):
                    snaps[sb].copy_(wflat, non_blocking=True)
                    ev_snap[sb].record(s_cmp)
                s_d2h.wait_event(ev_snap[sb])
                with torch.cuda.stream(s_d2h):
                    w_host.copy_(snaps[sb], non_blocking=True)
                    ev_out[sb].record(s_d2h)
            s_cmp.wait_event(ev_out[(nsteps - 1) & 1])
            ev_b.record(s_cmp)
            return ev_a, ev_b

        # untimed warm-up passes of the same pipeline (copies in both directions
        # at once, streams, events), then the timed steps; whole periods from a
        # Muon step in both
        t_e2e = base + args.steps
        nwarm = max(2, ((args.warmup + P - 1) // P) * P if P > 0 and not srank else args.warmup)
        pipelined(nwarm, t_e2e)
        t_e2e += nwarm
        torch.cuda.synchronize()
        barrier()
        e0, e1 = pipelined(args.steps, t_e2e)
        torch.cuda.synchronize()
        barrier()
        e_ms = max_over_ranks(e0.elapsed_time(e1), world, dev)
        e2e = {"value": e_ms / args.steps, "unit": "ms/step", "h2d_bytes_per_step": flat_bytes,
               "d2h_bytes_per_step": flat_bytes,
               "what": "pinned-host gradients copied in and updated parameters copied out every step, "
                       "through lm_step; the gradient copies and the read-back of a device snapshot of "
                       "the parameters overlap the steps (three gradient and two snapshot buffers); "
                       "the same pipeline runs untimed warm-up steps first"
                       + ("; layer-sharded: each rank copies the full gradient set in and reads the exchanged "
                          "parameters back, the NCCL exchange of each Muon step inside the timed region"
                          if sharded else "")}
    clk = clocks.stop()
    flags = opt.status()
    took_last = opt.selection()[0] if srank else None
    context = None
    if args.cublas_context and rank == 0:
        dense = sum(5 * (4.0 * min(m, n) ** 2 * max(m, n) + 2.0 * min(m, n) ** 3) for m, n in mats)
        cms = cublas_ns_context(mats, dev)
        context = {"what": "the same 5 NS iterations in torch.bmm/baddbmm (cuBLAS, bf16), full symmetric products, "
                           "for context only (not the library's path)",
                   "cublas_ms_per_muon_step": cms, "cublas_dense_tflops": dense / (cms / 1e3) / 1e12}

    # ---- roofline of the dominant kernel family ----
    peaks, peak_src = load_peaks()
    n_muon = 0 if srank else sum(1 for i in range(args.steps) if P > 0 and (base + i) % P == 0)
    n_lion = args.steps - n_muon
    ns_ms, ns_launches = prof["ns_gemm"]
    lion_ms, lion_launches = prof["lion"]
    ns_mats = own_mats if sharded else mats      # sharded: this rank's Newton-Schulz work
    traffic_ok = args.set == "gpt_720m" and not sharded and not srank and args.ns_table == "quintic"
    fl = ns_flops_sym(ns_mats, 5, poly_steps) * n_muon
    # The burst peak applies to a kernel timed in a short region, the
    # sustained one (the power cap's) to one inside a seconds-long loop.
    pk_burst = peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])
    pk_sust = peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"])
    long_region = ms_total >= 1000.0
    pk_bf16 = pk_sust if long_region else pk_burst
    bf16_kind = (f"bf16 {'sustained' if long_region else 'burst'} ({ms_total / 1e3:.2f} s timed region), "
                 f"{peak_src}")
    roof = None
    if ns_ms > 0 and n_muon > 0:
        achieved = fl / (ns_ms / 1e3) / 1e12
        flops_note = ("symmetric count 3 s^2 l + s^3 per matrix per NS iteration"
                      + (f" (s^3 in the {poly_steps} iterations with c != 0)" if poly_steps != 5 else ""))
        if args.precision == "bf16":
            pk = pk_bf16
            bound, kernel, peak_kind = "tensor", "ns_tc_kernel", bf16_kind
        elif args.precision == "f32tc":
            # six bf16 piece products per fp32 product, on the bf16 tensor pipe
            achieved *= 6
            fl *= 6
            pk = pk_bf16
            bound, kernel, peak_kind = "tensor", "ns_tc_kernel", bf16_kind
            flops_note = "6 x the symmetric count 3 s^2 l + s^3 (six bf16 piece products per fp32 product)"
        else:
            # fp32 FMA on the CUDA cores: SMs x 128 lanes x 2 FLOP x the maximum SM clock
            sms = torch.cuda.get_device_properties(dev).multi_processor_count
            mhz = (clk or {}).get("sm_max_mhz") or 2070.0
            pk = sms * 128 * 2 * mhz * 1e6 / 1e12
            bound, kernel = "alu", "ns_simt_kernel"
            peak_kind = f"fp32 FMA, derived: {sms} SMs x 128 lanes x 2 FLOP x {mhz:.0f} MHz"
        # the recorded traffic is that of the 720M set's bf16 launches on one GPU
        traffic = kernel_traffic(kernel) if traffic_ok and args.precision == "bf16" else None
        dense = sum(5 * 4.0 * min(m, n) ** 2 * max(m, n) + poly_steps * 2.0 * min(m, n) ** 3
                    for m, n in ns_mats) * n_muon
        # per phase: GRAM s^2 l, POLY s^3 (the symmetric products once), APPLY 2 s^2 l per iteration
        ph_fl = {"ns_gram": sum(min(a, b) ** 2 * max(a, b) for a, b in ns_mats),
                 "ns_poly": sum(min(a, b) ** 3 for a, b in ns_mats),
                 "ns_apply": sum(2.0 * min(a, b) ** 2 * max(a, b) for a, b in ns_mats)}
        mult = 6 if args.precision == "f32tc" else 1
        phases = {}
        for k, f1 in ph_fl.items():
            ms_k, n_k = prof[k]
            if ms_k > 0:
                tf = mult * (poly_steps if k == "ns_poly" else 5) * f1 * n_muon / (ms_k / 1e3) / 1e12
                phases[k] = {"ms_per_launch": ms_k / max(n_k, 1), "tflops": tf,
                             **({"frac": tf / pk} if bound == "tensor" else {})}
        roof = {"bound": bound, "achieved": achieved, "peak": pk, "unit": "TFLOP/s",
                "frac": achieved / pk, "traffic": traffic, "kernel": kernel,
                **({"frac_of_sustained": achieved / pk_sust, "frac_of_burst": achieved / pk_burst}
                   if bound == "tensor" else {}),
                "phases": phases,
                # the same time over the dense count 4 s^2 l + 2 s^3 (both symmetric products in full)
                "dense_equivalent_tflops": dense / (ns_ms / 1e3) / 1e12,
                "per_launch_ms": ns_ms / max(ns_launches, 1),
                "per_launch_tflop": fl / max(ns_launches, 1) / 1e12,
                "peak_kind": peak_kind,
                "flops": flops_note}
    lion_roof = None
    if lion_ms > 0:
        # Lion-step launches over all params: 14 B/param (bf16 W,G r/w W, fp32 M r/w)
        bytes_moved = 14.0 * numel * n_lion + 14.0 * (numel - mat_elems) * n_muon
        gbs = bytes_moved / (lion_ms / 1e3) / 1e9
        pk = peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"])
        lion_roof = {"bound": "hbm", "achieved": gbs, "peak": pk, "unit": "GB/s", "frac": gbs / pk,
                     "traffic": kernel_traffic("lion_kernel") if traffic_ok else None, "kernel": "lion_kernel",
                     # per full-set launch (one per Lion step); the vector-only launches of the
                     # Muon steps (0.02% of the parameters) are inside the sum
                     "per_launch_ms": lion_ms / max(n_lion, 1),
                     "frac_of_8tbs": gbs / 8000.0, "peak_kind": f"HBM copy, {peak_src}"}
    srank_roof = None
    if srank and prof["srank"][0] > 0:
        # every pass reads each fp32 momentum matrix once: 4 B per matrix element
        sr_ms = prof["srank"][0]
        gbs = 4.0 * mat_elems * args.srank_iters * args.steps / (sr_ms / 1e3) / 1e9
        pk = peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"])
        srank_roof = {"bound": "hbm", "achieved": gbs, "peak": pk, "unit": "GB/s", "frac": gbs / pk,
                      "traffic": None, "kernel": "srank_ring_kernel",
                      "per_step_ms": sr_ms / args.steps, "peak_kind": f"HBM copy, {peak_src}",
                      "bytes": "4 B x matrix elements x passes (plus resets and the decision)"}
    fam_ms = {k: v[0] / args.steps for k, v in prof.items() if k != "ns_gemm"}
    if context is not None and n_muon > 0:
        context["library_ns_ms_per_muon_step"] = ns_ms / n_muon

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        v, desc = oracle_sample(args.set, P, table)
        cpu = {"value": v, "unit": "ms/step", "cores": cpu_cores(), "kind": "oracle",
               "sample": ("fp64 oracle on a 4M-element Lion step and a full Muon step of one matrix of "
                          f"every shape, {desc}; each shape's time counted once per matrix of that shape, "
                          "the Lion time per element (extrapolated)")}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "ms/step", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
            "higher_is_better": False, "scaling": "strong", "vs_baseline": None,
            "dtype": {"bf16": "bf16", "f32": "f32", "f32tc": "f32 (3 x bf16 pieces)"}[args.precision],
            "data": "synthetic",
            "config": {"workload": args.set, "params": numel, "matrices": len(mats),
                       "period": None if srank else P, "ns_steps": 5, "ns_precision": args.precision,
                       **({"ns_table": args.ns_table} if args.ns_table != "quintic" else {}),
                       **({"vector_rule": "adamw"} if args.vector_rule == "adamw" else {}),
                       **({"schedule": "stable_rank", "srank_alpha": args.srank_alpha,
                           "srank_iters": args.srank_iters,
                           "muon_matrices_last_step": sum(1 for i, s in enumerate(shapes)
                                                          if len(s) == 2 and took_last[i])} if srank else {}),
                       "grads": f"{ps.grad_kind}, drawn on device, same gradients every step",
                       "l2": "inputs larger than L2 (14 B/param x %.0f M params streamed per Lion step)" % (numel / 1e6),
                       "timed_steps": f"t = {base} .. {base + args.steps - 1}" +
                                      ("" if srank else " (whole periods from a Muon step)"),
                       "parallelism": (f"layer-sharded Muon over {world} GPUs (each matrix's Muon update on "
                                       "its owner, owners' matrices broadcast after each Muon step; Lion "
                                       "steps on every GPU)") if sharded else "one GPU"},
            **({"exchange": {"bytes_received_per_muon_step_rank0": ex.received_bytes(0),
                             "broadcasts_per_muon_step": len(ex.items),
                             "ns_tflop_per_muon_step_rank0": ns_flops_sym(own_mats, 5, poly_steps) / 1e12,
                             "ns_tflop_per_muon_step_total": ns_flops_sym(mats, 5, poly_steps) / 1e12}} if sharded else {}),
            "roofline": srank_roof if srank else roof, "roofline_lion": lion_roof,
            **({"roofline_ns": roof} if srank else {}),
            "kernel_ms_per_step": fam_ms,
            "cpu_baseline": cpu, "e2e": e2e, "graph": graph, "gpu_launches": launches, "clocks": clk,
            "device_flags": flags,
            **({"context_cublas": context} if context else {}),
        }
        print(json.dumps(line), flush=True)
    opt.close()
    if world > 1:
        dist.destroy_process_group()
    return 0


def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
