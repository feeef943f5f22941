"""Benchmark of the LookME lookup + sparse injection on GB300.

A step is one lookme_lookup_inject call (level-1 routing, bucketing, level-2
scoring with top-k and softmax, token selection, gather and residual add; the
same results as lookme_lookup + lookme_inject) over one batch of seeded
synthetic tokens: the single-image workload
(1,024 tokens, d_k 256, 1,024 scenes x 256 primitives, d_v 2,048, bf16, top-8,
keep 25%) unless --workload says otherwise.

  value      tokens/s over K device-timed steps (CUDA events on the launching
             stream; the step replayed as one CUDA graph of the library's
             kernels; L2 flushed by writing then reading 512 MiB before every
             step, outside the events), inputs resident in HBM.  The eager
             time (the same calls issued one by one from Python) is reported
             beside it.
  e2e        the same through host buffers: pinned-host queries and hidden
             states copied in and the updated hidden states copied out, inside
             the timed region
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
    "score": ["k_score_tc.cu", "score_tc.cuh", "topk.cuh", "sm100.cuh"],
    "step": ["k_step.cu", "score_tc.cuh", "topk.cuh", "sm100.cuh"],
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

    t = lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, dtype=w.dtype, device=local,
                     max_tokens=w.n_tokens)
    cent = W.centroids(w, 0, dev)
    for c in range(w.n_chunks):
        k, v = W.table_chunk(w, 0, c, dev, None, cent)
        s0 = c * w.scenes_per_chunk
        t.load_scenes(s0, k, v, centroids=cent[s0:s0 + k.shape[0]])
        del k, v
    q = W.queries(w, dev)
    hidden = [W.hidden(w, l, dev) for l in range(w.layers_per_table)]
    N, K = w.n_tokens, w.top_k
    scene = torch.empty(N, dtype=torch.int32, device=dev)
    prim = torch.empty(N, K, dtype=torch.int32, device=dev)
    weight = torch.empty(N, K, dtype=torch.float32, device=dev)
    mask = torch.empty(N, dtype=torch.uint8, device=dev)
    seg = w.segment_offsets if w.n_segments > 1 else None
    flush = torch.empty(FLUSH_BYTES // 4, dtype=torch.int32, device=dev)
    flush_sink = torch.zeros((), dtype=torch.int64, device=dev)

    def step():
        t.lookup_inject(q, K, hidden, w.keep_ratio, seg_offsets=seg, scene_out=scene, prim_out=prim,
                        weight_out=weight, mask_out=mask)

    def flush_l2(i):
        # Write then read a buffer four times L2's size: the step starts with no
        # table data in L2 and no dirty flush lines left to write back.
        flush.fill_(i & 0xFF)
        flush_sink.copy_(flush.sum(dtype=torch.int64))

    for _ in range(args.warmup):
        flush_l2(1)
        step()
    torch.cuda.synchronize(dev)
    stats = t.stats()
    n_sel = int(mask.sum().item())

    # The step as one CUDA graph (the library never allocates or syncs inside a
    # call once scratch is reserved), replayed per timed step.
    graph = torch.cuda.CUDAGraph()
    side = torch.cuda.Stream(dev)
    side.wait_stream(stream)
    with torch.cuda.stream(side):
        step()
    stream.wait_stream(side)
    with torch.cuda.graph(graph):
        step()
    torch.cuda.synchronize(dev)

    c0 = t.launch_count()
    step()
    torch.cuda.synchronize(dev)
    launches_per_step = t.launch_count() - c0

    sampler = ClockSampler(local)
    sampler.start()
    # ---------------------------------------------------------- timed: value
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    if ws > 1:
        import torch.distributed as dist

        dist.barrier()
    torch.cuda.synchronize(dev)
    for i in range(args.steps):
        flush_l2(i)
        starts[i].record(stream)
        graph.replay()
        ends[i].record(stream)
    torch.cuda.synchronize(dev)
    if ws > 1:
        dist.barrier()
    step_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    total_ms = sum(step_ms)
    launches = launches_per_step * args.steps

    # ------------------------------------ the same steps as eager C-ABI calls
    estarts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    eends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    for i in range(args.steps):
        flush_l2(i)
        estarts[i].record(stream)
        step()
        eends[i].record(stream)
    torch.cuda.synchronize(dev)
    eager_ms = sum(s.elapsed_time(e) for s, e in zip(estarts, eends)) / args.steps

    # ----------------------------------------- per-kernel durations (traced)
    t.trace_enable(True)
    t.trace_read()
    tstarts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    tends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    for i in range(args.steps):
        flush_l2(i)
        tstarts[i].record(stream)
        step()
        tends[i].record(stream)
    torch.cuda.synchronize(dev)
    recs = t.trace_read(max_records=args.steps * 8 + 16)
    t.trace_enable(False)
    traced_ms = sum(s.elapsed_time(e) for s, e in zip(tstarts, tends))
    per_kernel = {}
    for name, ms in recs:
        per_kernel.setdefault(name, []).append(ms)
    kernels_ms = {k: statistics.mean(v) for k, v in per_kernel.items()}

    # ------------------------------------------------- e2e through host buffers
    q_host = q.cpu().pin_memory()
    h_host = [h.cpu().pin_memory() for h in hidden]
    h_out = [torch.empty_like(h).pin_memory() for h in h_host]
    q_dev = torch.empty_like(q)
    h_dev = [torch.empty_like(h) for h in hidden]
    e_starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    e_ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    for i in range(args.steps):
        flush_l2(i)
        e_starts[i].record(stream)
        q_dev.copy_(q_host, non_blocking=True)
        for hd, hh in zip(h_dev, h_host):
            hd.copy_(hh, non_blocking=True)
        t.lookup_inject(q_dev, K, h_dev, w.keep_ratio, seg_offsets=seg, scene_out=scene, prim_out=prim,
                        weight_out=weight, mask_out=mask)
        for ho, hd in zip(h_out, h_dev):
            ho.copy_(hd, non_blocking=True)
        e_ends[i].record(stream)
    torch.cuda.synchronize(dev)
    e2e_ms = sum(s.elapsed_time(e) for s, e in zip(e_starts, e_ends))
    clocks = sampler.stop()
    assert t.device_status() == 0, "a device-side wait timed out"

    total_ms, e2e_ms, value, e2e_value = aggregate_ranks(total_ms, e2e_ms, ws, N, args.steps, dev)

    h2d = q.numel() * q.element_size() + sum(h.numel() * h.element_size() for h in hidden)
    d2h = sum(h.numel() * h.element_size() for h in hidden)
    ms_per_step = total_ms / args.steps

    peaks, peak_kind = load_peaks()
    hbm = float(peaks["hbm_gbs"])
    ab = algorithmic_bytes(w, stats["n_routed_scenes"], n_sel)
    score_ms = kernels_ms.get("score")
    achieved = ab["score"] / (score_ms * 1e-3) / 1e9 if score_ms else None
    step_gbs = ab["step"] / (ms_per_step * 1e-3) / 1e9
    result = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": w.dtype, "data": "synthetic (seeded Gaussian mixture, random tables)",
        "config": {"workload": w.name, "tokens": N, "d_key": w.d_key, "scenes": w.n_scenes, "prims": w.n_prims,
                   "d_value": w.d_value, "top_k": K, "keep_ratio": w.keep_ratio, "layers": w.layers_per_table,
                   "l2": f"flushed before every step ({FLUSH_BYTES >> 20} MiB written then read, outside the events)",
                   "launch": "step replayed as one CUDA graph (kernels chained by programmatic dependent launch)",
                   "parallelism": f"replicas x{ws}" if ws > 1 else "single GPU"},
        "roofline": {"bound": "hbm", "kernel": "score (level-2 key scoring + top-k + softmax)",
                     "achieved": achieved, "peak": hbm, "unit": "GB/s",
                     "frac": achieved / hbm if achieved else None, "peak_source": peak_kind,
                     "algorithmic_bytes": ab["score"], "mean_ms": score_ms,
                     "traffic": profiled_traffic("score", w.name)},
        "step_roofline": {"bound": "hbm", "algorithmic_bytes": ab["step"], "achieved": step_gbs, "peak": hbm,
                          "unit": "GB/s", "frac": step_gbs / hbm, "roofline_us": ab["step"] / hbm / 1e3},
        "eager_ms_per_step": eager_ms,
        "kernels_ms": kernels_ms, "traced_ms_per_step": traced_ms / args.steps,
        "routed_scenes": stats["n_routed_scenes"], "selected_tokens": n_sel,
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "ms_per_step": e2e_ms / args.steps},
        "gpu_launches": launches,
        "clocks": clocks,
    }
    t.close()
    return result


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
    ws, rank, local = dist_env()
    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args, w)), flush=True)
        return
    if ws > 1:
        import torch
        import torch.distributed as dist

        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    res = run_lookme(args, w, ws, rank, local)
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
