"""Benchmark of the LookME lookup + sparse injection on GB300.

A step is one lookme_lookup_inject call (level-1 routing, bucketing, level-2
scoring with top-k and softmax, token selection, gather and residual add; the
same results as lookme_lookup + lookme_inject) over one batch of seeded
synthetic tokens: the single-image workload
(1,024 tokens, d_k 256, 1,024 scenes x 256 primitives, d_v 2,048, bf16, top-8,
keep 25%) unless --workload says otherwise.

  value      tokens/s over K device-timed steps, inputs resident in HBM.  When
             the table is small enough to hold several copies (single image:
             16 replicas, 18 GiB), step i runs on replica i % R and the steps
             rotate over S streams (single image: 16), so S batches are in
             flight (some batches' routing, bucketing and injection beside
             others' level 2), with the routing and bucketing grids sized for
             16 SMs and level 2 on 56 CTAs (lookme_set_grids); the steps are
             replayed as CUDA graphs of 64 steps between one pair of events,
             and R - 1 other steps pass between two uses of a replica, so its
             data is out of L2 (inputs larger than L2, no flush).
             Otherwise one step per graph replay with L2 flushed by writing
             then reading 512 MiB before every step, outside its events.
             Reported beside it: the latency of one call at a time (L2
             flushed, one graph replay) and the eager time.
  e2e        the same through host buffers: pinned-host queries and hidden
             states copied in and the updated hidden states copied out, inside
             the timed region, every step (replayed from the same kind of CUDA
             graphs as value when the steps are replicated)
  roofline   the level-2 scoring kernel (the dominant one): algorithmic bytes
             per launch / its mean event-timed duration, against the measured
             HBM copy bandwidth
  cpu_baseline  the CPU oracle on a bounded sample of the same workload

--impl reference times the CPU oracle itself as the reference arm.
Multi-GPU (torchrun): independent replicas, one per GPU (weak scaling).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "visual tokens/sec looked-up+injected at 1 GB300; fraction of GEMM/HBM roofline"
UNIT = "tokens/s"
FLUSH_BYTES = 512 << 20


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="lookme", choices=["lookme", "reference"])
    ap.add_argument("--workload", default="single_image")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--path", default="keys", choices=("keys",) + PATHS,
                    help="keys: the two-level lookup + injection (the default step); the others time one of the "
                         "paper-exact pieces on the single-image sizes")
    ap.add_argument("--replicas", type=int, default=0,
                    help="table replicas the timed steps rotate through (0: as many as keep L2 cold; "
                         "1: one table, L2 flushed before every step, e.g. for small profiler captures)")
    ap.add_argument("--streams", type=int, default=0,
                    help="streams the replicated steps rotate over (0: the plan's; must divide --replicas)")
    ap.add_argument("--small-grid", type=int, default=-1,
                    help="SMs the routing and bucketing grids are sized for in the replicated steps "
                         "(-1: 16 with four or more streams, else all; 0: all)")
    ap.add_argument("--level2-ctas", type=int, default=-1,
                    help="CTAs of level 2 in the replicated steps (-1: 56 with four or more streams, else one "
                         "per SM; 0: one per SM)")
    ap.add_argument("--value-width", type=int, default=0,
                    help="value row width d_v in place of the workload's (0: the workload's own); for ncu captures "
                         "of level 2, which streams keys only, within a few GB of device memory")
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="target CPU time of the oracle baseline")
    return ap.parse_args()


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


# The sources each profiled kernel is built from (the hash ties an ncu summary to them).
KERNEL_SOURCES = {
    "score": ["k_score_tc.cu", "score_tc.cuh", "topk.cuh", "sm100.cuh", "common.cuh"],
    "route": ["k_route.cu", "sm100.cuh", "common.cuh"],
    "inject": ["k_inject.cu", "select.cuh", "common.cuh"],
    "stage": ["k_stage.cu", "common.cuh"],
    "step": ["k_step.cu", "score_tc.cuh", "topk.cuh", "sm100.cuh", "common.cuh"],
}


def kernel_source_sha(kernel="step"):
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[kernel]:
        with open(os.path.join(ROOT, "paper_2607_16305_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def profiled_traffic(kernel, workload):
    """DRAM bytes per launch of `kernel` from its committed ncu summary, if that summary is current."""
    p = os.path.join(ROOT, "profiles", f"ncu_{kernel}_{workload}.md")
    if not os.path.exists(p):
        return None
    txt = open(p).read()
    m = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", txt)
    s = re.search(r"source_sha:\s*([0-9a-f]+)", txt)
    if not m or not s or s.group(1) != kernel_source_sha(kernel):
        return None
    return float(m.group(1))


class ClockSampler:
    """nvidia-smi clock / throttle sampling while the GPU works."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            time.sleep(0.3)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        self.proc.terminate()
        out, _ = self.proc.communicate(timeout=10)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        busy = [s for s in sm if s > 0.5 * max(sm)] if sm else []
        return {"sm_mhz": statistics.median(busy) if busy else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def algorithmic_bytes(w, n_routed, n_sel):
    """Bytes the step must move at least once (the roofline's numerator), by kernel."""
    e = w.elem_bytes
    N, dk, S, P, dv, k, L = w.n_tokens, w.d_key, w.n_scenes, w.n_prims, w.d_value, w.top_k, w.layers_per_table
    score = n_routed * P * dk * e + N * dk * e + N * k * 8 + N * 4
    route = N * dk * e + S * dk * e + S * 4 + N * 8
    inject = n_sel * k * dv * e + 2 * L * n_sel * dv * e + n_sel * k * 8
    return {"score": score, "route": route, "inject": inject,
            "step": score + route + inject + N * 4 * 3 - N * dk * e}  # queries are read once per step


def aggregate_ranks(total_ms, e2e_ms, ws, n_tokens, steps, device):
    """Whole-job numbers over ws replicas (weak scaling): the slowest rank's
    timed totals, and value = tokens all ranks processed / that time.  With
    ws > 1 the process group must be initialised (NCCL on the GPUs; any backend
    whose tensors live on `device`)."""
    if ws > 1:
        import torch
        import torch.distributed as dist

        tt = torch.tensor([total_ms, e2e_ms], dtype=torch.float64, device=device)
        dist.all_reduce(tt, op=dist.ReduceOp.MAX)
        total_ms, e2e_ms = tt.tolist()
    value = ws * n_tokens * steps / (total_ms / 1e3)
    e2e_value = ws * n_tokens * steps / (e2e_ms / 1e3)
    return total_ms, e2e_ms, value, e2e_value


L2_BYTES = 129 << 20
REPLICA_BUDGET = 24 << 30  # device bytes the table replicas may take
MAX_REPLICAS = 16
PIPE_STREAMS = 16          # most batches in flight (streams of the replicated steps)
TABLE_STREAMS = 2          # streams the tables of the multi-table step alternate over
SMALL_GRID_SMS = 16        # routing / bucketing grid with four or more batches in flight
LEVEL2_CTAS = 56           # level-2 CTAs with four or more batches in flight
GRAPH_STEPS = 64           # steps per captured graph in the timed region


def table_bytes(w):
    S, P, e = w.n_scenes, w.n_prims, w.elem_bytes
    return S * P * (w.d_key + w.d_value) * e + S * w.d_key * e


def plan_replicas(w):
    """How many table replicas the timed steps rotate through, and over how many streams.

    Each step reads about step_bytes that the previous steps did not; with R
    replicas used in turn, R - 1 other steps (at least 5x L2 of traffic) pass
    between two uses of one replica, so every step starts with its table data
    out of L2 and no flush is needed.  Within the budget R grows to
    PIPE_STREAMS, one stream (batch in flight) per replica; a table that fits
    fewer copies keeps what the rule asks for, over as many streams.  Returns
    (1, 1) (flush before every step instead) when that many replicas do not fit
    the budget or the table is not HBM-resident."""
    from paper_2607_16305_gb300 import workloads as W

    if w.residency != "device" or w.n_tables != 1:
        return 1, 1
    d = W.expected_distinct(w.n_tokens, w.n_scenes)
    step = algorithmic_bytes(w, d, int(w.n_tokens * w.keep_ratio))["step"]
    need = 1 + math.ceil(5 * L2_BYTES / step)
    fit = min(MAX_REPLICAS, REPLICA_BUDGET // table_bytes(w))
    if need > fit:
        return 1, 1
    r = max(need, min(PIPE_STREAMS, fit))
    return r, min(r, PIPE_STREAMS) if r % min(r, PIPE_STREAMS) == 0 else 1


def run_lookme(args, w, ws, rank, local):
    import torch

    from __graft_entry__ import build
    from paper_2607_16305_gb300 import lookme
    from paper_2607_16305_gb300 import workloads as W

    if rank == 0:
        build()
    if ws > 1:
        import torch.distributed as dist

        dist.barrier()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)

    R, NS = plan_replicas(w)
    if args.replicas > 0:
        R = args.replicas
        NS = max(d for d in range(1, min(PIPE_STREAMS, R) + 1) if R % d == 0)
    if args.streams > 0:
        NS = args.streams
    if R % NS:
        raise SystemExit(f"--streams ({NS}) must divide the replicas ({R})")
    small_grid = args.small_grid if args.small_grid >= 0 else (SMALL_GRID_SMS if NS >= 4 else 0)
    level2_ctas = args.level2_ctas if args.level2_ctas >= 0 else (LEVEL2_CTAS if NS >= 4 else 0)
    tabs = [lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, dtype=w.dtype, device=local,
                         max_tokens=w.n_tokens) for _ in range(R)]
    cent = W.centroids(w, 0, dev)
    for c in range(w.n_chunks):
        k, v = W.table_chunk(w, 0, c, dev, None, cent)
        s0 = c * w.scenes_per_chunk
        for t in tabs:  # every replica holds the same table
            t.load_scenes(s0, k, v, centroids=cent[s0:s0 + k.shape[0]])
        del k, v
    q0 = W.queries(w, dev)
    N, K, L = w.n_tokens, w.top_k, w.layers_per_table
    # Per replica: its own queries, hidden states and outputs.
    qs = [q0 if r == 0 else q0.clone() for r in range(R)]
    hs = [[W.hidden(w, l, dev) for l in range(L)] for _ in range(R)]
    outs = [(torch.empty(N, dtype=torch.int32, device=dev), torch.empty(N, K, dtype=torch.int32, device=dev),
             torch.empty(N, K, dtype=torch.float32, device=dev), torch.empty(N, dtype=torch.uint8, device=dev))
            for _ in range(R)]
    seg = w.segment_offsets if w.n_segments > 1 else None
    flush = torch.empty(FLUSH_BYTES // 4, dtype=torch.int32, device=dev)
    flush_sink = torch.zeros((), dtype=torch.int64, device=dev)
    streams = [torch.cuda.Stream(dev) for _ in range(NS)] if R > 1 else [stream]

    def set_grid(on):
        for t in tabs:
            t.set_grids(small_grid if on else 0, level2_ctas if on else 0)

    def step(r, q=None, hidden=None):
        sc, pr, wt, mk = outs[r]
        tabs[r].lookup_inject(qs[r] if q is None else q, K, hs[r] if hidden is None else hidden, w.keep_ratio,
                              seg_offsets=seg, scene_out=sc, prim_out=pr, weight_out=wt, mask_out=mk)

    def flush_l2(i):
        # Write then read a buffer four times L2's size: the step starts with no
        # table data in L2 and no dirty flush lines left to write back.
        flush.fill_(i & 0xFF)
        flush_sink.copy_(flush.sum(dtype=torch.int64))

    def pipelined(n, body):
        # Step i on replica i % R, issued on stream i % NS: NS batches in
        # flight, each replica always on the same stream.
        cur = torch.cuda.current_stream(dev)
        for s in streams:
            s.wait_stream(cur)
        for i in range(n):
            with torch.cuda.stream(streams[i % len(streams)]):
                body(i % R)
        for s in streams:
            cur.wait_stream(s)

    for i in range(args.warmup):
        if R == 1:
            flush_l2(1)
        step(i % R)
    torch.cuda.synchronize(dev)
    stats = tabs[0].stats()
    n_sel = int(outs[0][3].sum().item())
    c0 = tabs[0].launch_count()
    step(0)
    torch.cuda.synchronize(dev)
    launches_per_step = tabs[0].launch_count() - c0
    ref_out = [o.clone() for o in outs[0]]  # replica 0's results, default grids

    # Graphs of the steps (the library never allocates or syncs inside a call
    # once scratch is reserved).  With replicas: up to GRAPH_STEPS steps per
    # graph, pipelined over the streams; without: one step per graph.
    if R > 1:
        set_grid(True)
    side = torch.cuda.Stream(dev)
    side.wait_stream(stream)
    with torch.cuda.stream(side):
        for r in range(R):
            step(r)
    stream.wait_stream(side)
    torch.cuda.synchronize(dev)

    def capture(n):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            if R > 1:
                pipelined(n, step)
            else:
                step(0)
        return g

    g1 = capture(1) if R == 1 else None
    if R > 1:
        per_graph = min(args.steps, GRAPH_STEPS)
        g_full = capture(per_graph)
        rem = args.steps % per_graph
        g_rem = capture(rem) if rem else None
    torch.cuda.synchronize(dev)

    sampler = ClockSampler(local)
    sampler.start()
    # ---------------------------------------------------------- timed: value
    if ws > 1:
        import torch.distributed as dist

        dist.barrier()
    torch.cuda.synchronize(dev)
    if R > 1:
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ev0.record(stream)
        for _ in range(args.steps // per_graph):
            g_full.replay()
        if g_rem is not None:
            g_rem.replay()
        ev1.record(stream)
        torch.cuda.synchronize(dev)
        total_ms = ev0.elapsed_time(ev1)
    else:
        starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        for i in range(args.steps):
            flush_l2(i)
            starts[i].record(stream)
            g1.replay()
            ends[i].record(stream)
        torch.cuda.synchronize(dev)
        total_ms = sum(s.elapsed_time(e) for s, e in zip(starts, ends))
    if ws > 1:
        dist.barrier()
    launches = launches_per_step * args.steps
    for a, b in zip(ref_out, outs[0]):
        if not torch.equal(a, b):
            raise SystemExit("the timed steps' results differ from the first call's")

    # -------------- one call at a time: L2 flushed, one graph replay per call
    if g1 is None:
        set_grid(False)
        g1 = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g1):
            step(0)
        torch.cuda.synchronize(dev)
    lstarts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    lends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    for i in range(args.steps):
        flush_l2(i)
        lstarts[i].record(stream)
        g1.replay()
        lends[i].record(stream)
    torch.cuda.synchronize(dev)
    latency_ms = sum(s.elapsed_time(e) for s, e in zip(lstarts, lends)) / args.steps

    # ---------------------- the same steps as eager C-ABI calls from Python
    if R > 1:
        set_grid(True)
        ea, eb = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ea.record(stream)
        pipelined(args.steps, step)
        eb.record(stream)
        torch.cuda.synchronize(dev)
        eager_ms = ea.elapsed_time(eb) / args.steps
    else:
        estarts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        eends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        for i in range(args.steps):
            flush_l2(i)
            estarts[i].record(stream)
            step(0)
            eends[i].record(stream)
        torch.cuda.synchronize(dev)
        eager_ms = sum(s.elapsed_time(e) for s, e in zip(estarts, eends)) / args.steps

    # ----------------------------------------- per-kernel durations (traced)
    set_grid(False)
    t0 = tabs[0]
    t0.trace_enable(True)
    t0.trace_read()
    tstarts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    tends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    for i in range(args.steps):
        flush_l2(i)
        tstarts[i].record(stream)
        step(0)
        tends[i].record(stream)
    torch.cuda.synchronize(dev)
    recs = t0.trace_read(max_records=args.steps * 8 + 16)
    t0.trace_enable(False)
    traced_ms = sum(s.elapsed_time(e) for s, e in zip(tstarts, tends))
    per_kernel = {}
    for name, ms in recs:
        per_kernel.setdefault(name, []).append(ms)
    kernels_ms = {k: statistics.mean(v) for k, v in per_kernel.items()}

    # ------------------------------------------------- e2e through host buffers
    # Every step copies its queries and hidden states in from pinned host
    # memory and the updated hidden states back, on the step's stream.
    q_host = [qs[r].cpu().pin_memory() for r in range(R)]
    h_host = [[h.cpu().pin_memory() for h in hs[r]] for r in range(R)]
    h_out = [[torch.empty_like(h).pin_memory() for h in h_host[r]] for r in range(R)]
    q_dev = [torch.empty_like(q0) for _ in range(R)]
    h_dev = [[torch.empty_like(h) for h in hs[r]] for r in range(R)]

    def e2e_step(r):
        q_dev[r].copy_(q_host[r], non_blocking=True)
        for hd, hh in zip(h_dev[r], h_host[r]):
            hd.copy_(hh, non_blocking=True)
        step(r, q=q_dev[r], hidden=h_dev[r])
        for ho, hd in zip(h_out[r], h_dev[r]):
            ho.copy_(hd, non_blocking=True)

    if R > 1:
        # The same graphs of GRAPH_STEPS steps as the timed value, each step with
        # its copies in and out (captured as copy nodes from and to pinned host
        # memory), so the host-side launch cost of one call per step does not
        # stand in for the link.
        set_grid(True)
        for r in range(R):
            e2e_step(r)
        torch.cuda.synchronize(dev)

        def capture_e2e(n):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                pipelined(n, e2e_step)
            return g

        ge_full = capture_e2e(per_graph)
        ge_rem = capture_e2e(args.steps % per_graph) if args.steps % per_graph else None
        ge_full.replay()
        torch.cuda.synchronize(dev)
        xa, xb = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        xa.record(stream)
        for _ in range(args.steps // per_graph):
            ge_full.replay()
        if ge_rem is not None:
            ge_rem.replay()
        xb.record(stream)
        torch.cuda.synchronize(dev)
        e2e_ms = xa.elapsed_time(xb)
    else:
        e_starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        e_ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        for i in range(args.steps):
            flush_l2(i)
            e_starts[i].record(stream)
            e2e_step(0)
            e_ends[i].record(stream)
        torch.cuda.synchronize(dev)
        e2e_ms = sum(s.elapsed_time(e) for s, e in zip(e_starts, e_ends))
    clocks = sampler.stop()
    for t in tabs:
        assert t.device_status() == 0, "a device-side wait timed out"

    total_ms, e2e_ms, value, e2e_value = aggregate_ranks(total_ms, e2e_ms, ws, N, args.steps, dev)

    h2d = q0.numel() * q0.element_size() + sum(h.numel() * h.element_size() for h in hs[0])
    d2h = sum(h.numel() * h.element_size() for h in hs[0])
    ms_per_step = total_ms / args.steps

    peaks, peak_kind = load_peaks()
    hbm = float(peaks["hbm_gbs"])
    ab = algorithmic_bytes(w, stats["n_routed_scenes"], n_sel)
    score_ms = kernels_ms.get("score")
    achieved = ab["score"] / (score_ms * 1e-3) / 1e9 if score_ms else None
    step_gbs = ab["step"] / (ms_per_step * 1e-3) / 1e9
    if R > 1:
        l2 = (f"inputs larger than L2: {R} replicas of the table ({table_bytes(w) * R / 2**30:.1f} GiB) used in turn, "
              f"{R - 1} other steps between two uses of one replica; no flush")
        launch = (f"{NS} batches in flight: step i on replica i % {R} on stream i % {NS}; routing and bucketing "
                  f"grids sized for {small_grid or 'all'} SMs, level 2 on {level2_ctas or 'one CTA per SM'} CTAs; "
                  f"{per_graph} steps per CUDA graph; one event pair around all {args.steps} steps")
    else:
        l2 = f"flushed before every step ({FLUSH_BYTES >> 20} MiB written then read, outside the events)"
        launch = "step replayed as one CUDA graph (kernels chained by programmatic dependent launch)"
    result = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": w.dtype, "data": "synthetic (seeded Gaussian mixture, random tables)",
        "config": {"workload": w.name, "tokens": N, "d_key": w.d_key, "scenes": w.n_scenes, "prims": w.n_prims,
                   "d_value": w.d_value, "top_k": K, "keep_ratio": w.keep_ratio, "layers": L,
                   "replicas": R, "streams": NS, "small_grid_sms": small_grid, "level2_ctas": level2_ctas, "l2": l2,
                   "launch": launch,
                   "parallelism": f"replicas x{ws}" if ws > 1 else "single GPU"},
        "roofline": {"bound": "hbm", "kernel": "score (level-2 key scoring + top-k + softmax)",
                     "achieved": achieved, "peak": hbm, "unit": "GB/s",
                     "frac": achieved / hbm if achieved else None, "peak_source": peak_kind,
                     "algorithmic_bytes": ab["score"], "mean_ms": score_ms,
                     "traffic": profiled_traffic("score", w.name)},
        "step_roofline": {"bound": "hbm", "algorithmic_bytes": ab["step"], "achieved": step_gbs, "peak": hbm,
                          "unit": "GB/s", "frac": step_gbs / hbm, "roofline_us": ab["step"] / hbm / 1e3,
                          "peak_source": peak_kind},
        "latency_ms_per_call": latency_ms,
        "latency_method": "one call at a time: L2 flushed before each, one CUDA-graph replay, events around it",
        "eager_ms_per_step": eager_ms,
        "kernels_ms": kernels_ms, "traced_ms_per_step": traced_ms / args.steps,
        "routed_scenes": stats["n_routed_scenes"], "selected_tokens": n_sel,
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "ms_per_step": e2e_ms / args.steps,
                "launch": "CUDA graphs of the steps with their copies" if R > 1 else "one eager call per step"},
        "gpu_launches": launches,
        "clocks": clocks,
    }
    for t in tabs:
        t.close()
    return result


def run_multitable(args, w, ws, rank, local):
    """Several tables over one query set (each table shared by layers_per_table
    layers), tables in pinned host memory staged to HBM on demand.

    A step = one lookme_lookup_inject per table, tables alternating over two
    streams so that one table's routing, bucketing and key staging overlap the
    previous table's level 2 and injection.  Cold: each table's slot cache is
    emptied and L2 flushed before every step (outside the events), so every
    routed scene's key block crosses the host link; warm: the caches persist
    (the same queries every step, so every routed scene is a hit)."""
    import torch

    from __graft_entry__ import build
    from paper_2607_16305_gb300 import lookme
    from paper_2607_16305_gb300 import workloads as W

    if rank == 0:
        build()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)
    T, L, N, K = w.n_tables, w.layers_per_table, w.n_tokens, w.top_k
    mu = W.means(w, dev)
    tabs = []
    for ti in range(T):
        t = lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, dtype=w.dtype, residency="host",
                         device=local, max_tokens=N)
        cent = W.centroids(w, ti, dev, mu)
        for c in range(w.n_chunks):
            k, v = W.table_chunk(w, ti, c, dev, mu, cent)
            s0 = c * w.scenes_per_chunk
            t.load_scenes(s0, k, v, centroids=cent[s0:s0 + k.shape[0]])
            del k, v
        tabs.append(t)
    q = W.queries(w, dev, mu)
    hidden = [W.hidden(w, l, dev) for l in range(T * L)]
    outs = [(torch.empty(N, dtype=torch.int32, device=dev), torch.empty(N, K, dtype=torch.int32, device=dev),
             torch.empty(N, K, dtype=torch.float32, device=dev), torch.empty(N, dtype=torch.uint8, device=dev))
            for _ in range(T)]
    streams = [torch.cuda.Stream(dev) for _ in range(TABLE_STREAMS)]
    flush = torch.empty(FLUSH_BYTES // 4, dtype=torch.int32, device=dev)
    flush_sink = torch.zeros((), dtype=torch.int64, device=dev)

    def step():
        cur = torch.cuda.current_stream(dev)
        for s in streams:
            s.wait_stream(cur)
        for ti in range(T):
            sc, pr, wt, mk = outs[ti]
            with torch.cuda.stream(streams[ti % len(streams)]):
                tabs[ti].lookup_inject(q, K, hidden[ti * L:(ti + 1) * L], w.keep_ratio, scene_out=sc, prim_out=pr,
                                       weight_out=wt, mask_out=mk)
        for s in streams:
            cur.wait_stream(s)

    def cold_prep(i):
        for t in tabs:
            t.stage_invalidate(stream)
        flush.fill_(i & 0xFF)
        flush_sink.copy_(flush.sum(dtype=torch.int64))

    for i in range(args.warmup):
        cold_prep(i)
        step()
    torch.cuda.synchronize(dev)
    stats = [t.stats() for t in tabs]
    staged = sum(s["staged_bytes"] for s in stats)
    routed = [s["n_routed_scenes"] for s in stats]
    n_sel = int(outs[0][3].sum().item())
    c0 = sum(t.launch_count() for t in tabs)
    step()
    torch.cuda.synchronize(dev)
    launches_per_step = sum(t.launch_count() for t in tabs) - c0

    # Host link reference: one pinned-host -> HBM copy engine transfer.
    hbuf = torch.empty(256 << 20, dtype=torch.uint8).pin_memory()
    dbuf = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    for _ in range(3):
        dbuf.copy_(hbuf, non_blocking=True)
    la, lb = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    la.record(stream)
    for _ in range(10):
        dbuf.copy_(hbuf, non_blocking=True)
    lb.record(stream)
    torch.cuda.synchronize(dev)
    link_gbs = 10 * hbuf.numel() / (la.elapsed_time(lb) * 1e-3) / 1e9
    del dbuf

    sampler = ClockSampler(local)
    sampler.start()
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    torch.cuda.synchronize(dev)
    for i in range(args.steps):
        cold_prep(i)
        starts[i].record(stream)
        step()
        ends[i].record(stream)
    torch.cuda.synchronize(dev)
    total_ms = sum(s.elapsed_time(e) for s, e in zip(starts, ends))
    cold_stats = [t.stats() for t in tabs]
    # Warm: persistent caches, no flush, back to back.
    step()
    wa, wb = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    wa.record(stream)
    for i in range(args.steps):
        step()
    wb.record(stream)
    torch.cuda.synchronize(dev)
    warm_ms = wa.elapsed_time(wb) / args.steps
    warm_stats = [t.stats() for t in tabs]
    # Per-kernel durations of table 0 (cold, one table at a time).
    t0 = tabs[0]
    t0.trace_enable(True)
    t0.trace_read()
    for i in range(min(args.steps, 20)):
        cold_prep(i)
        sc, pr, wt, mk = outs[0]
        t0.lookup_inject(q, K, hidden[:L], w.keep_ratio, scene_out=sc, prim_out=pr, weight_out=wt, mask_out=mk)
    torch.cuda.synchronize(dev)
    recs = t0.trace_read(max_records=400)
    t0.trace_enable(False)
    clocks = sampler.stop()
    for t in tabs:
        assert t.device_status() == 0, "a device-side wait timed out"
    per_kernel = {}
    for name, ms in recs:
        per_kernel.setdefault(name, []).append(ms)
    kernels_ms = {k: statistics.mean(v) for k, v in per_kernel.items()}
    ms_per_step = total_ms / args.steps
    stage_ms = kernels_ms.get("stage")
    stage_gbs = stats[0]["staged_bytes"] / (stage_ms * 1e-3) / 1e9 if stage_ms else None
    peaks, peak_kind = load_peaks()
    result = {
        "metric": METRIC, "value": N / (ms_per_step * 1e-3), "unit": UNIT, "n_gpus": 1, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": w.dtype, "data": "synthetic (seeded Gaussian mixture, random tables)",
        "config": {"workload": w.name, "tokens": N, "tables": T, "layers_per_table": L, "d_key": w.d_key,
                   "scenes": w.n_scenes, "prims": w.n_prims, "d_value": w.d_value, "top_k": K,
                   "keep_ratio": w.keep_ratio, "residency": "pinned host, HBM slot cache per table",
                   "l2": "cold: slot caches emptied and L2 flushed before every step, outside the events",
                   "launch": f"one lookme_lookup_inject per table, tables alternating over {TABLE_STREAMS} streams"},
        "roofline": {"bound": "host link", "staged_key_bytes_per_step": staged,
                     "achieved": staged / (ms_per_step * 1e-3) / 1e9, "peak": link_gbs, "unit": "GB/s",
                     "frac": staged / (ms_per_step * 1e-3) / 1e9 / link_gbs,
                     "peak_source": "pinned host -> HBM copy-engine transfer of 256 MiB, measured in this run",
                     "stage_kernel_gbs": stage_gbs},
        "routed_scenes_per_table": routed, "selected_tokens_per_table": n_sel,
        "cold_staged_bytes": sum(s["staged_bytes"] for s in cold_stats),
        "warm": {"ms_per_step": warm_ms, "value": N / (warm_ms * 1e-3),
                 "staged_bytes": sum(s["staged_bytes"] for s in warm_stats),
                 "hits": sum(s["staged_hits"] for s in warm_stats)},
        "link_gbs": link_gbs, "kernels_ms_table0": kernels_ms, "gpu_launches": launches_per_step * args.steps,
        "clocks": clocks, "hbm_peak": float(peaks["hbm_gbs"]), "peak_kind": peak_kind,
    }
    for t in tabs:
        t.close()
    return result


# ------------------------------------------------------------------------------
# Bench lines of the paper-exact pieces (--path): one call at a time, L2
# flushed before each, events around it, on the single-image sizes (the
# paper's own d_e = 512 for the embedding-space pieces).
PATHS = ("ranked", "fusion", "router", "project", "text")


def _time_calls(fn, steps, warmup, flush, stream, sampler=None, graph=True):
    """Mean device time of one call of fn, L2 flushed before each, events
    around each.  graph: the call is captured once as a CUDA graph and
    replayed, so the host's argument marshalling and launch work of an eager
    call (which the events would otherwise bracket while the GPU waits) is
    left out."""
    import torch

    for i in range(warmup):
        flush(i)
        fn()
    torch.cuda.synchronize()
    run = fn
    if graph:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            fn()
        torch.cuda.synchronize()
        run = g.replay
    st = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    en = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    for i in range(steps):
        flush(i)
        st[i].record(stream)
        run()
        en[i].record(stream)
    torch.cuda.synchronize()
    return statistics.mean(a.elapsed_time(b) for a, b in zip(st, en))


def run_path(args, w):
    """One of PATHS on the single-image sizes; returns the JSON line."""
    import torch

    from __graft_entry__ import build
    from paper_2607_16305_gb300 import lookme
    from paper_2607_16305_gb300 import workloads as W

    build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(0)
    stream = torch.cuda.current_stream(dev)
    flush_buf = torch.empty(FLUSH_BYTES // 4, dtype=torch.int32, device=dev)
    sink = torch.zeros((), dtype=torch.int64, device=dev)

    def flush(i):
        flush_buf.fill_(i & 0xFF)
        sink.copy_(flush_buf.sum(dtype=torch.int64))

    def rnd(shape, seed, scale=1.0, dtype=torch.bfloat16):
        g = torch.Generator(device=dev)
        g.manual_seed(seed)
        return (scale * torch.randn(*shape, generator=g, device=dev)).to(dtype).contiguous()

    peaks, peak_kind = load_peaks()
    hbm, tf = float(peaks["hbm_gbs"]), float(peaks["bf16_tflops"])
    N, K = w.n_tokens, w.top_k
    launches = None
    kernels = {}
    sampler = ClockSampler(0)
    sampler.start()
    if args.path == "ranked":
        dm, R = 256, PIPE_STREAMS  # one table replica per batch in flight, as for the keys path
        W1, b1 = rnd((dm, 2 * w.d_key), 1, 1 / math.sqrt(2 * w.d_key)), rnd((dm,), 2, 0.1, torch.float32)
        W2, b2 = rnd((w.n_prims, dm), 3, 2 / math.sqrt(dm)), rnd((w.n_prims,), 4, 0.1, torch.float32)
        tabs = [lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, dtype=w.dtype, device=0, max_tokens=N)
                for _ in range(R)]
        cent = W.centroids(w, 0, dev)
        for c in range(w.n_chunks):
            k, v = W.table_chunk(w, 0, c, dev, None, cent)
            for t in tabs:
                t.load_scenes(c * w.scenes_per_chunk, k, v, centroids=cent[c * w.scenes_per_chunk:][:k.shape[0]])
            del k, v
        for t in tabs:
            t.set_ranker(W1, b1, W2, b2)
        q0 = W.queries(w, dev)
        delta0 = rnd((N, w.d_value), 5)
        wg = rnd((w.d_value,), 6, 1 / math.sqrt(w.d_value))
        bufs = [dict(q=q0.clone(), delta=delta0.clone(), hidden=[W.hidden(w, 0, dev)],
                     sc=torch.empty(N, dtype=torch.int32, device=dev), pr=torch.empty(N, K, dtype=torch.int32, device=dev),
                     wt=torch.empty(N, K, dtype=torch.float32, device=dev),
                     gate=torch.empty(N, dtype=torch.uint8, device=dev)) for _ in range(R)]

        def fn_r(r):
            b_ = bufs[r]
            lookme.ska_gate(b_["delta"], wg, gate_out=b_["gate"])
            tabs[r].lookup_ranked(b_["q"], K, scene_out=b_["sc"], prim_out=b_["pr"], weight_out=b_["wt"])
            tabs[r].inject_gated(b_["sc"], b_["pr"], b_["wt"], b_["gate"], b_["hidden"])

        def fn():
            fn_r(0)

        for r in range(R):
            fn_r(r)
        torch.cuda.synchronize()
        t = tabs[0]
        n_sel = int(bufs[0]["gate"].sum().item())
        c0 = t.launch_count()
        fn()
        torch.cuda.synchronize()
        launches = t.launch_count() - c0 + 1  # + the gate kernel (table-less)
        latency_ms = _time_calls(fn, args.steps, args.warmup, flush, stream)
        # Batches in flight over the replicas, one stream each (graphs of 64 steps), with the routing
        # grid sized for SMALL_GRID_SMS SMs, as the keys path's value.
        for t_ in tabs:
            t_.set_grids(SMALL_GRID_SMS, 0)
        streams = [torch.cuda.Stream(dev) for _ in range(R)]
        gph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gph):
            cur = torch.cuda.current_stream(dev)
            for s_ in streams:
                s_.wait_stream(cur)
            for i in range(64):
                with torch.cuda.stream(streams[i % R]):
                    fn_r(i % R)
            for s_ in streams:
                cur.wait_stream(s_)
        for _ in range(2):
            gph.replay()
        torch.cuda.synchronize()
        reps = max(1, args.steps // 64)
        ea, eb = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ea.record(stream)
        for _ in range(reps):
            gph.replay()
        eb.record(stream)
        torch.cuda.synchronize()
        ms = ea.elapsed_time(eb) / (reps * 64)
        t.set_grids(0, 0)
        t.trace_enable(True)
        t.trace_read()
        _time_calls(fn, min(args.steps, 50), 1, flush, stream, graph=False)
        for name, v in t.trace_read(max_records=2000):
            kernels.setdefault(name, []).append(v)
        t.trace_enable(False)
        for tt in tabs:
            assert tt.device_status() == 0
        e = w.elem_bytes
        nbytes = (N * w.d_key * e + w.n_scenes * w.d_key * e + N * K * w.d_key * e + N * w.d_value * e
                  + dm * (2 * w.d_key + w.n_prims) * e + n_sel * K * w.d_value * e + 2 * n_sel * w.d_value * e)
        flops = 2 * N * w.n_scenes * w.d_key + 2 * N * (w.d_key * dm + dm * w.n_prims)
        what = (f"SKA gate + level 1 + MLP-ranked level 2 (d_m {dm}, top-{K}) + gated injection; value: two "
                f"batches in flight over {R} table replicas, {reps * 64} steps; latency: one call at a time")
        for tt in tabs:
            tt.close()
    elif args.path == "fusion":
        de, dff, dh, n_st, n = 512, 2048, w.d_value, 4, N // 4
        f = lookme.Fusion(n_st, de, dff, dh, device=0, max_rows=n)
        for k in range(n_st):
            f.load_stage(k, rnd((dff, de), 10 + k, 1 / math.sqrt(de)), rnd((dff, de), 20 + k, 1 / math.sqrt(de)),
                         rnd((dh, dff), 30 + k, 1 / math.sqrt(dff)),
                         rnd((de, de), 40 + k, 0.5 / math.sqrt(de)) if k else None)
        R = rnd((n, de), 50, 0.05)
        rows = torch.arange(0, N, 4, dtype=torch.int32, device=dev)
        hidden = [rnd((N, dh), 60 + k) for k in range(n_st)]

        def fn():
            f.apply(R, rows, hidden)

        ms = _time_calls(fn, args.steps, args.warmup, flush, stream)
        assert f.status() == 0
        launches = 3 * n_st - 1
        flops = n_st * (2 * n * de * 2 * dff + 2 * n * dff * dh) + (n_st - 1) * 2 * n * de * de
        nbytes = 2 * (n_st * (2 * dff * de + dh * dff) + (n_st - 1) * de * de) + n * de * 2 + n_st * 2 * n * dh * 2
        what = f"SwiGLU fusion d_e {de} -> d_ff {dff} -> d_h {dh} on {n} gated tokens, {n_st} layers with R W_p + R"
        f.close()
    elif args.path == "router":
        de, dh, M = 512, w.d_value, 3
        Hs = rnd((N, dh), 70)
        Whe = rnd((de, dh), 71, 1 / math.sqrt(dh))
        Rs = [rnd((N, de), 72 + m, 0.5) for m in range(M)]
        out = torch.empty(N, de, dtype=torch.bfloat16, device=dev)
        ws = torch.empty(N, de, dtype=torch.float32, device=dev)

        def fn():
            lookme.scale_router(Hs, Whe, Rs, out=out, workspace=ws)

        ms = _time_calls(fn, args.steps, args.warmup, flush, stream)
        launches = 2
        flops = 2 * N * dh * de
        nbytes = N * dh * 2 + de * dh * 2 + M * N * de * 2 + N * de * 2 + 2 * N * de * 4
        what = f"multi-scale softmax router over {M} scales (d_h {dh} -> d_e {de})"
    elif args.path == "project":
        dv, de = w.d_value, 512
        x = rnd((N, dv), 80)
        Wv = rnd((de, dv), 81, 1 / math.sqrt(dv))
        out = torch.empty(N, de, dtype=torch.bfloat16, device=dev)

        def fn():
            lookme.project(x, Wv, out=out)

        ms = _time_calls(fn, args.steps, args.warmup, flush, stream)
        launches = 1
        flops = 2 * N * dv * de
        nbytes = N * dv * 2 + de * dv * 2 + N * de * 2
        what = f"projection W_v->e ({dv} -> {de})"
    else:  # text
        V, d = 151936, w.d_value
        E = rnd((V, d), 90, 0.02)
        g = torch.Generator(device=dev)
        g.manual_seed(91)
        ids = torch.randint(0, V, (N,), generator=g, device=dev, dtype=torch.int32)
        ids[::2] = -1  # image positions
        gate = (torch.rand(N, generator=g, device=dev) < 0.5).to(torch.uint8)
        hidden = [rnd((N, d), 92 + l) for l in range(4)]

        def fn():
            lookme.text_inject(E, ids, hidden, gate=gate)

        ms = _time_calls(fn, args.steps, args.warmup, flush, stream)
        n_on = int(((ids >= 0) & (gate > 0)).sum().item())
        launches = 1
        flops = 0
        nbytes = N * 5 + n_on * d * 2 * (1 + 2 * len(hidden))
        what = f"text ID lookup (vocab {V}, d {d}) injected into {len(hidden)} layers"
    clocks = sampler.stop()
    gbs = nbytes / (ms * 1e-3) / 1e9
    tfs = flops / (ms * 1e-3) / 1e12
    t_bytes, t_flops = nbytes / hbm / 1e9, flops / tf / 1e12
    bound = "hbm" if t_bytes >= t_flops else "tensor"
    roof = {"bound": bound, "unit": "GB/s" if bound == "hbm" else "TFLOP/s",
            "achieved": gbs if bound == "hbm" else tfs, "peak": hbm if bound == "hbm" else tf,
            "algorithmic_bytes": nbytes, "algorithmic_flops": flops, "peak_source": peak_kind,
            "roofline_us": max(t_bytes, t_flops) * 1e6}
    roof["frac"] = roof["achieved"] / roof["peak"]
    extra = {"latency_ms_per_call": latency_ms} if args.path == "ranked" else {}
    return {**extra, "metric": METRIC, "value": N / (ms * 1e-3), "unit": UNIT, "n_gpus": 1, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded Gaussian mixture, random weights)",
            "config": {"workload": w.name, "path": args.path, "what": what, "tokens": N,
                       "l2": f"flushed before every call ({FLUSH_BYTES >> 20} MiB written then read, outside the events)",
                       "launch": "one call at a time, events around it"},
            "roofline": roof, "kernels_ms": {k: statistics.mean(v) for k, v in kernels.items()},
            "gpu_launches": launches * args.steps if launches else None, "clocks": clocks, "cpu_baseline": None}


def oracle_step(o, data, idx, w):
    """The oracle's whole path on the tokens idx (route, level 2, selection over all priorities, injection)."""
    import numpy as np

    q = data["q"][idx]
    r = o.route(q, data["cent"])
    p = o.primitives(q, r["scene"], data["keys"], w.top_k)
    s = o.select(data["qnorm_all"], w.keep_ratio, w.segment_offsets)
    m = s["mask"][idx]
    rows = np.nonzero(m)[0]
    vb, bos = data["vblocks"], data["vbos"]
    ok = (bos[r["scene"][rows]] >= 0).all()
    if not ok:
        raise RuntimeError("value block missing for the CPU baseline")
    o.inject(r["scene"][rows], p["prim"][rows], p["weight"][rows], np.ones(rows.size, np.uint8), vb,
             data["h"][idx][rows][None], bos, w.n_scenes)
    return len(idx)


def cpu_data(w, n_sample, seed=0):
    """Host copies of what the oracle needs for a seeded sample of the workload (not timed)."""
    import numpy as np
    import torch

    import oracle as oracle_pkg
    from paper_2607_16305_gb300 import workloads as W

    dev = torch.device("cuda", 0) if torch.cuda.is_available() else torch.device("cpu")
    o = oracle_pkg.Oracle()
    cent = W.centroids(w, 0, dev)
    keys = torch.cat([W.table_chunk(w, 0, c, dev, None, cent)[0] for c in range(w.n_chunks)])
    q = W.queries(w, dev)
    h = W.hidden(w, 0, dev)
    rng = np.random.default_rng(seed)
    idx = np.sort(rng.choice(w.n_tokens, min(n_sample, w.n_tokens), replace=False))
    data = {"q": q.float().cpu().numpy(), "cent": cent.float().cpu().numpy(), "keys": keys.float().cpu().numpy(),
            "h": h.float().cpu().numpy()}
    data["qnorm_all"] = o.query_norms(data["q"])
    r = o.route(data["q"][idx], data["cent"])
    s = o.select(data["qnorm_all"], w.keep_ratio, w.segment_offsets)
    need = np.unique(r["scene"][s["mask"][idx] == 1])
    bos = np.full(w.n_scenes, -1, np.int64)
    blocks = []
    for c in range(w.n_chunks):
        ss = [int(x) for x in need if int(x) // w.scenes_per_chunk == c]
        if not ss:
            continue
        _, v = W.table_chunk(w, 0, c, dev, None, cent)
        for x in ss:
            bos[x] = len(blocks)
            blocks.append(v[x - c * w.scenes_per_chunk].float().cpu().numpy())
    data["vblocks"] = np.stack(blocks) if blocks else np.zeros((1, w.n_prims, w.d_value), np.float32)
    data["vbos"] = bos
    return o, data, idx


def cpu_baseline(w, seconds):
    """The oracle as it stands, timed on this host's cores on a bounded sample of the workload."""
    cores = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    o, data, idx = cpu_data(w, min(w.n_tokens, 256))
    t0 = time.perf_counter()
    n = oracle_step(o, data, idx, w)
    one = time.perf_counter() - t0
    reps = max(1, int(seconds / max(one, 1e-3)))
    t0 = time.perf_counter()
    done = 0
    for _ in range(reps):
        done += oracle_step(o, data, idx, w)
    el = time.perf_counter() - t0
    return {"value": done / el, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{len(idx)} seeded tokens of {w.name} per pass x {reps} passes ({el:.1f} s); "
                      f"routing against all {w.n_scenes} centroids, selection over all {w.n_tokens} priorities"}


def run_reference(args, w):
    """Reference arm: the CPU oracle itself, K timed steps of a bounded token sample each."""
    cores = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    per_step = max(8, min(w.n_tokens, int(120.0 / max(args.steps + args.warmup, 1) / 2e-3)))
    o, data, idx = cpu_data(w, per_step)
    for _ in range(args.warmup):
        oracle_step(o, data, idx, w)
    t0 = time.perf_counter()
    done = 0
    for _ in range(args.steps):
        done += oracle_step(o, data, idx, w)
    el = time.perf_counter() - t0
    value = done / el
    sample = f"{len(idx)} seeded tokens of {w.name} per step"
    return {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": 1, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": el * 1e3 / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded Gaussian mixture)",
            "config": {"workload": w.name, "tokens_per_step": len(idx)},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    args = parse()
    from paper_2607_16305_gb300 import workloads as W

    w = W.WORKLOADS[args.workload]
    if args.value_width > 0:
        w = w.scaled(d_value=args.value_width)
    ws, rank, local = dist_env()
    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args, w)), flush=True)
        return
    if args.path != "keys":
        if rank == 0:
            print(json.dumps(run_path(args, w)), flush=True)
        return
    if ws > 1:
        import torch
        import torch.distributed as dist

        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    res = run_multitable(args, w, ws, rank, local) if w.n_tables > 1 else run_lookme(args, w, ws, rank, local)
    if rank == 0:
        if ws == 1 and not args.no_cpu_baseline:
            res["cpu_baseline"] = cpu_baseline(w, args.cpu_seconds)
        else:
            res["cpu_baseline"] = None
        print(json.dumps(res), flush=True)
    if ws > 1:
        import torch.distributed as dist

        dist.destroy_process_group()


if __name__ == "__main__":
    main()
