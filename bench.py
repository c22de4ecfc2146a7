"""Benchmark: hyperbatch sampling + gathering on one (or N replica) GB300s.

One step = one hyperbatch through the whole path (bucketing, K hops of
sampling + dedup/relabel, block-wise feature gather) via the C ABI, on the
100M-node RMAT workload (fp16 x128 features, 1 MB blocks, 128 minibatches x
1024 targets from a 1% train split, fanouts [15, 10, 5]).  Inputs are
generated on the device before timing; the graph (~33 GB) is far larger than
L2, so no L2 flush is needed between steps.

Prints one JSON line (rank 0).  --impl reference times the CPU oracle
instead (bounded sample, host cores).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from agnes_inputs import WORKLOADS, build_graph, target_pool, targets_for_step  # noqa: E402

METRIC = "sampled+gathered minibatches/sec per hyperbatch; achieved HBM GB/s vs ~8 TB/s"
UNIT = "minibatches/s"
DEFAULT_WORKLOAD = "rmat100m"
FALLBACK_HBM_GBS = 6800.0


# ----------------------------------------------------------------------------
# helpers
# ----------------------------------------------------------------------------

def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def step_index(rank: int, s: int) -> int:
    """Hyperbatch index of step s on a rank: ranks draw disjoint target sets
    (weak scaling, one independent replica per GPU)."""
    return rank * 1_000_003 + s


def reduce_max(x: float, pg, device) -> float:
    """Max of x over the ranks of the process group (x itself without one)."""
    if pg is None:
        return x
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return float(t.item())


def measured_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


class ClockSampler:
    """Samples nvidia-smi clocks and throttle reasons while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100", "-f", self.path],
                stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.2)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if self.proc is None or not self.path or not os.path.exists(self.path):
            return None
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i] == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(rows)}


def kernel_launches_per_step(K: int) -> int:
    """Kernels libagnes launches per hyperbatch with the graph in HBM (60 at
    K = 3): the sampling-key write and the dst-size fill 2; target bucketing 4
    (count, single-pass scan, scatter, sort); per hop 16 (count, 2-kernel
    segmented scan, fill, single-pass scan, scatter, the cells' lane kernel,
    queue offsets, queue copy, tile kernel, 3-kernel column scan, single-pass
    scan, col fix-up, compaction); after the last hop 3 (feature-block marks,
    their count, gather) and K counts of touched topology blocks."""
    return 2 + 4 + 16 * K + 3 + K


def algorithmic_bytes(c: dict, off_bytes: int) -> dict:
    """Bytes the method must move per hyperbatch (per-unit model):
    per hop h: frontier offsets pair, sampled-id read, col write, indptr,
    node-list write; gather: one read per distinct row, one write per row,
    8 index bytes per row."""
    rb = c["row_bytes"]
    K = len(c["frontier"])
    hop = 0
    for h in range(K):
        f, e = c["frontier"][h], c["edges"][h]
        src = c["frontier"][h + 1] if h + 1 < K else c["rows"]
        hop += f * 2 * off_bytes + e * 4 + e * 4 + f * 8 + (src - f) * 4
    gather = c["rows"] * (rb + 8) + c["distinct_rows"] * rb
    return {"sampling": hop, "gather": gather, "total": hop + gather}


def gather_traffic_from_profile(workload: str):
    """Per-launch DRAM traffic of the gather kernel from the committed ncu
    summary, if it was taken on the current gather source and this workload."""
    if workload != "rmat100m":
        return None
    path = os.path.join(ROOT, "profiles", "gather_rmat100m.md")
    src = os.path.join(ROOT, "paper_2601_01473_gb300", "csrc", "gather_hbm.cu")
    try:
        sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
        vals = {}
        for line in open(path):
            if ":" in line and line.strip().startswith("- "):
                k, v = line.strip()[2:].split(":", 1)
                vals[k.strip()] = v.strip()
        if vals.get("gather_hbm.cu sha256 prefix") != sha:
            return None
        return float(vals["dram bytes per launch (full workload)"])
    except Exception:
        return None


# ----------------------------------------------------------------------------
# oracle (CPU baseline / reference arm)
# ----------------------------------------------------------------------------

def time_oracle(host_graph, w, targets_cpu, seconds_budget: float, max_mbs: int):
    """Runs the oracle (as it stands) on a sample of the workload's
    minibatches on the host cores; returns (minibatches/s, cores, sample)."""
    import concurrent.futures as cf

    import oracle
    og = oracle.Graph(*host_graph)
    cores = max(1, min(os.cpu_count() or 1, max_mbs))
    # calibrate on one minibatch, then size the sample to the budget
    t0 = time.perf_counter()
    oracle.sample_minibatch(og, targets_cpu[0], list(w.fanouts), w.seed, 0)
    one = time.perf_counter() - t0
    n = int(max(cores, min(max_mbs, (seconds_budget / max(one, 1e-3)) * cores)))
    n = max(1, n)
    rows = [targets_cpu[i % targets_cpu.shape[0]] for i in range(n)]

    def run(i):
        oracle.sample_minibatch(og, rows[i], list(w.fanouts), w.seed, i)
        return i

    t0 = time.perf_counter()
    with cf.ThreadPoolExecutor(max_workers=cores) as ex:
        list(ex.map(run, range(n)))
    dt = time.perf_counter() - t0
    return n / dt, cores, f"{n} minibatches of the workload (B={w.B}, fanouts {list(w.fanouts)}) on {cores} threads, {dt:.1f} s"


def time_oracle_single(host_graph, w, targets_cpu):
    """The oracle as written on one core: min(H, 8) minibatches of one
    hyperbatch, one after another, scaled to the hyperbatch (the oracle's
    minibatches are independent, so a hyperbatch of H takes H times one
    minibatch's mean time).  Returns (minibatches/s, sample description)."""
    import oracle
    og = oracle.Graph(*host_graph)
    m = max(1, min(w.H, 8))
    t0 = time.perf_counter()
    for j in range(m):
        oracle.sample_minibatch(og, targets_cpu[j % targets_cpu.shape[0]], list(w.fanouts), w.seed, j)
    dt = time.perf_counter() - t0
    return m / dt, (f"{m} of the hyperbatch's {w.H} minibatches on 1 core in {dt:.2f} s, scaled to "
                    f"the hyperbatch: {w.H * dt / m:.2f} s per hyperbatch (scaled)")


def pinned_h2d_peak(dev, nbytes: int = 1 << 30, reps: int = 5) -> float:
    """Measured pinned host -> device copy bandwidth (GB/s), best of reps."""
    src = torch.empty(nbytes, dtype=torch.uint8).pin_memory()
    dst = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    best = 0.0
    for _ in range(reps + 1):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record()
        dst.copy_(src, non_blocking=True)
        e1.record()
        torch.cuda.synchronize()
        best = max(best, nbytes / (e0.elapsed_time(e1) / 1e3) / 1e9)
    del src, dst
    return best


def host_copy(offsets, indices, features):
    return (offsets.cpu().numpy(), indices.cpu().numpy(), features.cpu().numpy())


# ----------------------------------------------------------------------------
# main
# ----------------------------------------------------------------------------

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="agnes", choices=["agnes", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(WORKLOADS))
    ap.add_argument("--H", type=int, default=None, help="override minibatches per hyperbatch")
    ap.add_argument("--block", type=int, default=None, help="override block bytes")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--sweep", action="store_true",
                    help="hyperbatch size x block size sweep on the workload's graph (one JSON "
                         "line per combination)")
    ap.add_argument("--sweep-H", default="1,2,4,8,16,32,64,128,256")
    ap.add_argument("--sweep-blocks", default="262144,524288,1048576,2097152,4194304")
    ap.add_argument("--stream-topology", action="store_true",
                    help="neighbour lists in pinned host memory, loaded into an HBM graph buffer")
    ap.add_argument("--graph-buffer-gb", type=float, default=4.0)
    ap.add_argument("--topology-io", default="blocks", choices=["blocks", "rows"],
                    help="with --stream-topology: load whole blocks into the graph buffer, or "
                         "read sampled neighbour entries in place")
    ap.add_argument("--stream", action="store_true",
                    help="features in pinned host memory, streamed block-wise per hyperbatch")
    ap.add_argument("--feature-cache-gb", type=float, default=0.0,
                    help="with --stream: HBM feature cache of the most requested blocks")
    ap.add_argument("--feature-cache-threshold", type=int, default=0,
                    help="with --stream: requests a block must exceed to be cached")
    ap.add_argument("--inflight", type=int, default=0,
                    help="time N hyperbatches in flight (N ctxs over one graph, one stream each)")
    ap.add_argument("--ablation", action="store_true",
                    help="AGNES-No (one minibatch per hyperbatch) vs AGNES-HB, three settings")
    ap.add_argument("--ablation-hyperbatches", type=int, default=3)
    ap.add_argument("--sage", action="store_true",
                    help="time the GraphSAGE-mean consumer layer on a prepared hyperbatch")
    ap.add_argument("--sage-d-out", type=int, default=128)
    ap.add_argument("--sage-out", default="f32", choices=["f32", "f16"])
    ap.add_argument("--frontier", default="src", choices=["src", "sampled"],
                    help="next-hop frontier: src_h (default) or Algorithm 1's literal N_out "
                         "(the path byte model then counts dst_{h+1} as src_h)")
    ap.add_argument("--launch-mode", default="graph_pdl", choices=["direct", "graph", "graph_pdl"],
                    help="resident path: direct launches, one CUDA graph per hyperbatch shape, "
                         "or the graph with programmatic kernel edges")
    ap.add_argument("--pipeline-depth", type=int, default=3, choices=[1, 2, 3, 4],
                    help="hyperbatches in flight inside the library (resident graph only)")
    ap.add_argument("--feature-io", default="blocks", choices=["blocks", "rows"],
                    help="with --stream: load whole feature blocks, or read requested rows in place")
    args = ap.parse_args()

    world, rank, local = dist_env()
    if args.warmup < 3:
        args.warmup = 3
    w = WORKLOADS[args.workload]
    if args.H:
        w = w.with_(H=args.H)
    if args.block:
        w = w.with_(adj_block_bytes=args.block, feat_block_bytes=args.block)

    if args.impl == "reference":
        return run_reference(args, w, world, rank)
    if args.sweep:
        return run_sweep(args, w)
    if args.ablation:
        return run_ablation(args, w)
    if args.inflight > 0:
        return run_inflight(args, w)
    if args.sage:
        return run_sage(args, w)

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pg = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
        pg = dist

    from paper_2601_01473_gb300 import Graph

    t_gen = time.perf_counter()
    offsets, indices, features = build_graph(w, dev)
    pool = target_pool(w, dev)
    n_steps = args.warmup + args.steps
    # each rank draws its own hyperbatches (weak scaling: fixed work per GPU)
    step_targets = [targets_for_step(w, pool, step_index(rank, s)) for s in range(n_steps)]
    torch.cuda.synchronize()
    gen_s = time.perf_counter() - t_gen
    torch.cuda.empty_cache()

    stream = torch.cuda.current_stream(dev)
    host_link = None
    if args.stream:
        features = features.cpu().pin_memory()
        torch.cuda.empty_cache()
        host_link = {"h2d_peak_GBps": pinned_h2d_peak(dev)}
    topo = None
    if args.stream_topology:
        indices = indices.cpu().pin_memory()
        torch.cuda.empty_cache()
        topo = {"graph_buffer_bytes": int(args.graph_buffer_gb * 2**30)}
        if host_link is None:
            host_link = {"h2d_peak_GBps": pinned_h2d_peak(dev)}
    g = Graph(offsets, indices, features, w.adj_block_bytes, w.feat_block_bytes, device=local,
              stream=stream, features_on_host=args.stream, topology_on_host=args.stream_topology,
              graph_buffer_bytes=topo["graph_buffer_bytes"] if topo else 0,
              topology_io=args.topology_io if args.stream_topology else "blocks",
              feature_cache_bytes=int(args.feature_cache_gb * 2**30) if args.stream else 0,
              feature_cache_threshold=args.feature_cache_threshold,
              feature_io=args.feature_io if args.stream else "blocks")
    g.set_launch_mode(args.launch_mode)
    g.set_frontier(args.frontier)
    depth = args.pipeline_depth if not (args.stream or args.stream_topology) else 1
    g.set_pipeline_depth(depth)
    info = g.info()
    fan = list(w.fanouts)
    K = len(fan)
    gid = lambda s: step_index(rank, s) * w.H  # noqa: E731

    # warm-up (also allocates the workspace)
    for s in range(args.warmup):
        g.prepare(step_targets[s], fan, w.seed, gid(s), stream)
    torch.cuda.synchronize()

    # timed: device-resident inputs, CUDA events on the launching stream; the
    # library records the gather's start and end events on the same stream
    # (ring of 64) -- two events, since each one splits the launch sequence
    g.set_profiling("gather")
    if pg:
        pg.barrier()
    torch.cuda.synchronize()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    gpu_index = local
    vis = os.environ.get("CUDA_VISIBLE_DEVICES", "").split(",")
    if len(vis) > local and vis[local].strip().isdigit():
        gpu_index = int(vis[local])
    with ClockSampler(gpu_index) as clk:
        ev0.record(stream)
        for s in range(args.warmup, n_steps):
            g.prepare(step_targets[s], fan, w.seed, gid(s), stream)
        g.wait(stream)  # the hyperbatches still in flight on the library's streams
        ev1.record(stream)
        torch.cuda.synchronize()
    if pg:
        pg.barrier()
    elapsed_ms = ev0.elapsed_time(ev1)
    gather_ms = [p[0] for p in (g.phase_times(ago) for ago in range(min(args.steps, 64))) if p]
    elapsed_ms = reduce_max(elapsed_ms, pg, dev)
    clocks = clk.summary()

    # byte accounting and the per-phase breakdown: rerun the timed steps
    # (untimed, every phase profiled) to read their counters and phase times
    g.set_profiling("phases")
    counters = []
    for s in range(args.warmup, n_steps):
        g.prepare(step_targets[s], fan, w.seed, gid(s), stream)
        counters.append(g.counters())
    phases = [g.phase_times(ago) for ago in range(min(args.steps, 64))]
    g.set_profiling(False)
    off_bytes = offsets.element_size()
    algo = [algorithmic_bytes(c, off_bytes) for c in counters]
    gather_bytes = statistics.mean(a["gather"] for a in algo)
    total_bytes = statistics.mean(a["total"] for a in algo)
    iso = [p[-1] for p in phases if p]
    iso_ms = statistics.mean(iso) if iso else None
    stats = g.stats()

    # end to end through the C ABI: host (pinned) targets in, views out
    e2e = None
    if not args.no_e2e:
        host_targets = [t.cpu().pin_memory() for t in step_targets]
        for s in range(2):
            g.prepare(host_targets[s], fan, w.seed, gid(s), stream)
            g.fetch_all()
        if pg:
            pg.barrier()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for s in range(args.warmup, n_steps):
            g.prepare(host_targets[s], fan, w.seed, gid(s), stream)
            if depth == 1:
                g.fetch_all()
            elif s - args.warmup >= depth - 1:  # the oldest one held, while the later ones run
                g.fetch_earlier(depth - 1)
        for ago in range(min(depth, args.steps) - 2, -1, -1):  # the ones still unread
            g.fetch_earlier(ago)
        torch.cuda.synchronize()
        e2e_s = time.perf_counter() - t0
        e2e_s = reduce_max(e2e_s, pg, dev)
        d2h = 4 * (1 + (K + 1) * w.H + K * w.H) + 8 * (K + 1)
        e2e = {"value": world * w.H * args.steps / e2e_s, "unit": UNIT,
               "h2d_bytes_per_step": w.H * w.B * 4, "d2h_bytes_per_step": d2h}

    value = world * w.H * args.steps / (elapsed_ms / 1e3)
    peak, peak_kind = measured_peak()
    g_ms = statistics.mean(gather_ms) if gather_ms else None
    achieved = gather_bytes / (g_ms / 1e3) / 1e9 if g_ms else None
    roofline = {"bound": "hbm", "kernel": "gather_vec_kernel<16,8>",
                "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak if achieved else None,
                "peak_source": f"{peak_kind} (MEASURED_PEAKS.json hbm_gbs)"
                if peak_kind == "measured" else "fallback 6.8 TB/s",
                "traffic": gather_traffic_from_profile(w.name),
                "algorithmic_bytes_per_launch": gather_bytes,
                "avg_launch_ms": g_ms,
                # the gather alone: the untimed re-run fetches each hyperbatch's
                # counters before the next prepare, so nothing overlaps it there
                "isolated_launch_ms": iso_ms,
                "isolated_achieved": gather_bytes / (iso_ms / 1e3) / 1e9 if iso_ms else None,
                "isolated_frac": gather_bytes / (iso_ms / 1e3) / 1e9 / peak if iso_ms else None,
                "path_algorithmic_bytes_per_step": total_bytes,
                "path_GBps": total_bytes / (elapsed_ms / args.steps / 1e3) / 1e9}
    # the whole sample+gather path (every kernel of the step) against the same
    # peak: the fraction the >= 60 %-of-HBM target is stated on
    roofline["path_frac"] = roofline["path_GBps"] / peak

    if topo is not None:
        # counters are cumulative over the ctx: per-step figures from the timed
        # region's re-run (first and last of the re-run steps)
        c0, c1 = counters[0], counters[-1]
        n = max(1, len(counters) - 1)
        topo.update({
            "loaded_bytes_per_step": (c1["topo_loaded_bytes"] - c0["topo_loaded_bytes"]) / n,
            "loaded_blocks_per_step": (c1["topo_loaded_blocks"] - c0["topo_loaded_blocks"]) / n,
            "hit_blocks_per_step": (c1["topo_hit_blocks"] - c0["topo_hit_blocks"]) / n,
            "waves_per_step": (c1["topo_waves"] - c0["topo_waves"]) / n,
            "topology_bytes": indices.numel() * 4})
        hb, lb = topo["hit_blocks_per_step"], topo["loaded_blocks_per_step"]
        topo["hit_rate"] = hb / (hb + lb) if hb + lb else None
        if args.topology_io == "rows":  # graph buffer = topology cache; hits are requests
            req = statistics.mean(sum(c["frontier"]) for c in counters[1:]) if n > 0 else 0
            cr = (c1["topo_cached_requests"] - c0["topo_cached_requests"]) / n
            topo.update({"requests_per_step": req, "cached_requests_per_step": cr,
                         "hit_rate": cr / req if req else None})
        topo["load_GBps_over_step"] = topo["loaded_bytes_per_step"] / (elapsed_ms / args.steps / 1e3) / 1e9
    if host_link is not None and args.stream:
        sb = statistics.mean(c["streamed_bytes"] for c in counters)
        host_link.update({"streamed_bytes_per_step": sb,
                          "streamed_blocks_per_step": statistics.mean(c["streamed_blocks"]
                                                                      for c in counters),
                          "streamed_GBps": sb / (g_ms / 1e3) / 1e9 if g_ms else None})
        host_link["frac"] = (host_link["streamed_GBps"] / host_link["h2d_peak_GBps"]
                             if host_link["streamed_GBps"] else None)
        if args.feature_cache_gb > 0:
            c0, c1 = counters[0], counters[-1]
            n = max(1, len(counters) - 1)
            hits = (c1["fcache_hit_blocks"] - c0["fcache_hit_blocks"]) / n
            loads = (c1["fcache_loaded_blocks"] - c0["fcache_loaded_blocks"]) / n
            host_link["feature_cache"] = {
                "bytes": int(args.feature_cache_gb * 2**30),
                "threshold": args.feature_cache_threshold,
                "hit_blocks_per_step": hits, "loaded_blocks_per_step": loads,
                "hit_rate": hits / (hits + host_link["streamed_blocks_per_step"])
                if hits + host_link["streamed_blocks_per_step"] else None}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        host_graph = host_copy(offsets, indices, features)
        tcpu = step_targets[args.warmup].cpu().numpy()
        v, cores, sample = time_oracle(host_graph, w, tcpu, args.cpu_seconds, 8192)
        v1, sample1 = time_oracle_single(host_graph, w, tcpu)
        cpu = {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample,
               "nproc": os.cpu_count(),
               "single_thread": {"value": v1, "unit": UNIT, "cores": 1, "scaled": True,
                                 "sample": sample1}}

    if rank == 0:
        mean_phases = [statistics.mean(p[i] for p in phases) for i in range(len(phases[0]))] \
            if phases else []
        out = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": elapsed_ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "int32",
            "data": "synthetic",
            "config": {"workload": f"{w.name}: {w.describe()}"
                           + (f" features in pinned host memory ({args.feature_io} I/O)"
                              if args.stream else "")
                           + (f", {args.feature_cache_gb:g} GB feature cache"
                              if args.stream and args.feature_cache_gb > 0 else "")
                           + ((f" topology in pinned host memory, {args.graph_buffer_gb:g} GB graph buffer"
                               if args.topology_io == "blocks" else
                               " topology in pinned host memory (rows I/O)")
                              if args.stream_topology else ""),
                       "graph": {"nodes": info["num_nodes"], "edges": info["num_edges"],
                                 "adj_blocks": info["adj_blocks"], "tiles": info["tiles"],
                                 "feat_blocks": info["feat_blocks"]},
                       "H": w.H, "B": w.B, "fanouts": fan, "parallelism": f"replicas{world}",
                       "launch_mode": args.launch_mode, "frontier": args.frontier,
                       "pipeline_depth": depth,
                       "l2": "inputs larger than L2 (graph ~%.0f GB vs 129 MB L2), no flush"
                             % ((offsets.numel() * offsets.element_size()
                                 + indices.numel() * 4
                                 + features.numel() * features.element_size()) / 1e9),
                       "blocks_touched_last_step": stats,
                       "counters_last_step": counters[-1] if counters else None,
                       "gen_seconds": round(gen_s, 1)},
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "host_link": host_link,
            "topology_streaming": topo,
            # counted for the HBM-resident path (the ncu launch list has 67 per hyperbatch
            # at K = 3); the host-resident modes add per-batch loads and gathers
            "gpu_launches": kernel_launches_per_step(K) * args.steps
            if not (args.stream or args.stream_topology) else None,
            "clocks": clocks,
            "phases_ms": {"names": ["bucket_targets"] + [f"hop{h + 1}_{p}" for h in range(K)
                                                         for p in ("count_scan", "sample", "dedup")]
                          + ["gather"], "mean": mean_phases,
                          "note": "untimed re-run of the timed steps with every phase profiled"},
        }
        print(json.dumps(out), flush=True)
    g.close()
    if pg:
        pg.destroy_process_group()


def run_sweep(args, w):
    """Minibatches/s and blocks touched per hop (the block-wise I/Os of the
    paper's Fig. 7) over hyperbatch sizes and block sizes on one graph."""
    from paper_2601_01473_gb300 import Graph
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    offsets, indices, features = build_graph(w, dev)
    pool = target_pool(w, dev)
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    stream = torch.cuda.current_stream(dev)
    fan = list(w.fanouts)
    for bb in [int(x) for x in args.sweep_blocks.split(",")]:
        g = Graph(offsets, indices, features, bb, bb, device=0, stream=stream)
        # at most two in flight here: H = 256 needs twice config 3's workspace per set
        g.set_pipeline_depth(min(args.pipeline_depth, 2))
        info = g.info()
        for H in [int(x) for x in args.sweep_H.split(",")]:
            wh = w.with_(H=H, adj_block_bytes=bb, feat_block_bytes=bb)
            steps = [targets_for_step(wh, pool, s) for s in range(args.warmup + args.steps)]
            for s in range(args.warmup):
                g.prepare(steps[s], fan, w.seed, s * H, stream)
            torch.cuda.synchronize()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for s in range(args.warmup, args.warmup + args.steps):
                g.prepare(steps[s], fan, w.seed, s * H, stream)
            g.wait(stream)
            e1.record(stream)
            torch.cuda.synchronize()
            ms = e0.elapsed_time(e1) / args.steps
            stats = g.stats()
            print(json.dumps({"sweep": w.name, "block_bytes": bb, "H": H, "B": w.B,
                              "minibatches_per_s": H / (ms / 1e3), "ms_per_step": ms,
                              "adj_blocks_touched_per_hop": stats[:-1],
                              "feat_blocks_touched": stats[-1],
                              "adj_blocks": info["adj_blocks"], "feat_blocks": info["feat_blocks"],
                              "block_io_bytes": (sum(stats[:-1]) + stats[-1]) * bb}), flush=True)
        g.close()


def run_inflight(args, w):
    """Hyperbatches in flight: args.inflight contexts over one borrowed graph,
    one stream each, taking the steps round-robin, so one hyperbatch's gather
    (HBM-bound) overlaps another's sampling and dedup (latency-bound).  One
    JSON line with the pipelined throughput; the default bench line keeps one
    hyperbatch at a time."""
    from paper_2601_01473_gb300 import Graph
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    offsets, indices, features = build_graph(w, dev)
    pool = target_pool(w, dev)
    n = args.inflight
    steps = [targets_for_step(w, pool, s) for s in range(args.warmup + args.steps)]
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    fan = list(w.fanouts)
    gs = [Graph(offsets, indices, features, w.adj_block_bytes, w.feat_block_bytes, device=0)
          for _ in range(n)]
    sts = [torch.cuda.Stream(dev) for _ in range(n)]
    for s in range(args.warmup):
        gs[s % n].prepare(steps[s], fan, w.seed, s * w.H, sts[s % n])
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(sts[0])
    for st in sts[1:]:
        st.wait_event(e0)
    for s in range(args.warmup, args.warmup + args.steps):
        gs[s % n].prepare(steps[s], fan, w.seed, s * w.H, sts[s % n])
    for st in sts[1:]:
        ev = torch.cuda.Event()
        ev.record(st)
        sts[0].wait_event(ev)
    e1.record(sts[0])
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / args.steps
    for g in gs:  # every step's results were produced (sizes read back, status checked)
        g.fetch_all()
        g.close()
    print(json.dumps({"metric": METRIC, "value": w.H / (ms / 1e3), "unit": UNIT, "n_gpus": 1,
                      "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
                      "higher_is_better": True, "inflight": n, "dtype": "int32",
                      "data": "synthetic", "config": {"workload": w.name, "H": w.H, "B": w.B,
                                                      "fanouts": fan}}), flush=True)


def run_ablation(args, w):
    """AGNES-No against AGNES-HB (the paper's EQ2): the same minibatches
    prepared one per hyperbatch (No) and H per hyperbatch (HB), with the graph
    resident in HBM, with features in pinned host memory (block I/O) and with
    topology in pinned host memory (4 GB graph buffer).  Both arms draw
    identical samples (same seed and minibatch ids); one JSON line per setting."""
    from paper_2601_01473_gb300 import Graph
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    offsets, indices, features = build_graph(w, dev)
    pool = target_pool(w, dev)
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream(dev)
    fan = list(w.fanouts)
    H = w.H
    n_hb = max(1, args.ablation_hyperbatches)
    steps = [targets_for_step(w, pool, s) for s in range(1 + n_hb)]
    settings = [("resident", {}, 64), ("features_on_host", {"features_on_host": True}, 4),
                ("topology_on_host", {"topology_on_host": True,
                                      "graph_buffer_bytes": int(args.graph_buffer_gb * 2**30)}, 4)]
    host_feats = host_ind = None
    for name, kw, n_no in settings:
        if kw.get("features_on_host") and host_feats is None:
            host_feats = features.cpu().pin_memory()
        if kw.get("topology_on_host") and host_ind is None:
            host_ind = indices.cpu().pin_memory()
        f = host_feats if kw.get("features_on_host") else features
        ind = host_ind if kw.get("topology_on_host") else indices
        torch.cuda.empty_cache()
        g = Graph(offsets, ind, f, w.adj_block_bytes, w.feat_block_bytes, device=0, stream=stream,
                  **kw)

        def link_bytes():
            c = g.counters()
            return c["streamed_bytes"], c["topo_loaded_bytes"], c

        def timed(calls):
            torch.cuda.synchronize()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            moved = 0
            for t, gid0 in calls:
                g.prepare(t, fan, w.seed, gid0, stream)
                sb, _, _ = link_bytes() if kw.get("features_on_host") else (0, 0, None)
                moved += sb
            e1.record(stream)
            torch.cuda.synchronize()
            return e0.elapsed_time(e1), moved

        # each arm is warmed up right before it is timed (a change of H
        # re-sizes the workspace, which must stay outside the timed region)
        g.prepare(steps[0], fan, w.seed, 0, stream)
        t0 = g.counters()["topo_loaded_bytes"]
        hb_ms, hb_feat = timed([(steps[1 + s], (1 + s) * H) for s in range(n_hb)])
        g.prepare(steps[0][:1], fan, w.seed, 0, stream)
        t1 = g.counters()["topo_loaded_bytes"]
        no_calls = [(steps[1][j:j + 1], H + j) for j in range(min(n_no, H))]
        no_ms, no_feat = timed(no_calls)
        t2 = g.counters()["topo_loaded_bytes"]
        hb_mbs = n_hb * H / (hb_ms / 1e3)
        no_mbs = len(no_calls) / (no_ms / 1e3)
        print(json.dumps({
            "ablation": "AGNES-No vs AGNES-HB", "workload": w.name, "setting": name,
            "H": H, "B": w.B, "fanouts": fan,
            "hb": {"minibatches_per_s": hb_mbs, "minibatches": n_hb * H,
                   "host_link_bytes_per_minibatch": (hb_feat + t1 - t0) / (n_hb * H)},
            "no": {"minibatches_per_s": no_mbs, "minibatches": len(no_calls),
                   "host_link_bytes_per_minibatch": (no_feat + t2 - t1) / len(no_calls)},
            "hb_over_no": hb_mbs / no_mbs}), flush=True)
        g.close()


def run_sage(args, w):
    """The consumer: one GraphSAGE-mean layer (agnes_sage_mean_layer) over the
    outermost hop of a prepared hyperbatch, fed by the gathered features.
    Reports its time per launch against the HBM roofline (each src row read
    once, the output written once) and its tensor-core rate."""
    from paper_2601_01473_gb300 import Graph
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    offsets, indices, features = build_graph(w, dev)
    pool = target_pool(w, dev)
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream(dev)
    fan = list(w.fanouts)
    K = len(fan)
    g = Graph(offsets, indices, features, w.adj_block_bytes, w.feat_block_bytes, device=0,
              stream=stream)
    g.prepare(targets_for_step(w, pool, 0), fan, w.seed, 0, stream)
    allv = g.fetch_all()
    d_in, d_out = w.feat_dim, args.sage_d_out
    out_dtype = torch.float16 if args.sage_out == "f16" else torch.float32
    gen = torch.Generator().manual_seed(7)
    wt = (torch.randn(d_out, 2 * d_in, generator=gen) / (2 * d_in) ** 0.5).to(torch.float16).to(dev)
    bias = (torch.randn(d_out, generator=gen) * 0.1).to(dev)
    x = allv.feats
    for _ in range(args.warmup):
        g.sage_mean_layer(K - 1, x, wt, bias, out_dtype=out_dtype, stream=stream)
    times = []
    with ClockSampler(0) as clk:
        for _ in range(args.steps):
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            g.sage_mean_layer(K - 1, x, wt, bias, out_dtype=out_dtype, stream=stream)
            e1.record(stream)
            torch.cuda.synchronize()
            times.append(e0.elapsed_time(e1))
    ms = statistics.median(times)
    nd = allv.node_size[K - 1].astype(np.int64)
    ns = allv.node_size[K].astype(np.int64)
    ne = allv.edges[K - 1].astype(np.int64)
    rb = d_in * features.element_size()
    ob = 2 if out_dtype == torch.float16 else 4
    algo = int((ns * rb).sum() + (ne * 4).sum() + ((nd + 1) * 8).sum() + (nd * d_out * ob).sum()
               + wt.numel() * 2)
    flops = int((nd * 2 * 2 * d_in * d_out).sum())
    hbm, peak_kind = measured_peak()
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            bf16 = float(json.load(f)["bf16_tflops"])
    except Exception:
        bf16 = None
    gbs = algo / (ms / 1e3) / 1e9
    print(json.dumps({
        "sage": "GraphSAGE-mean layer over the outermost hop (agnes_sage_mean_layer)",
        "workload": f"{w.name}: {w.describe()}", "d_in": d_in, "d_out": d_out,
        "x_dtype": str(features.dtype).replace("torch.", ""), "out_dtype": args.sage_out,
        "dst_rows": int(nd.sum()), "edges": int(ne.sum()), "src_rows": int(ns.sum()),
        "ms_per_launch": ms, "dst_rows_per_s": float(nd.sum()) / (ms / 1e3),
        "roofline": {"bound": "hbm", "achieved": gbs, "peak": hbm, "unit": "GB/s",
                     "frac": gbs / hbm if hbm else None, "algorithmic_bytes_per_launch": algo,
                     "peak_source": f"{peak_kind} (MEASURED_PEAKS.json hbm_gbs)"},
        "tensor": {"tflops": flops / (ms / 1e3) / 1e12, "flops_per_launch": flops,
                   "fp16_dense_peak_tflops": bf16,
                   "peak_source": "measured bf16 burst (MEASURED_PEAKS.json bf16_tflops); "
                                  "fp16 has the same nominal rate"},
        "clocks": clk.summary()}), flush=True)
    g.close()


def run_reference(args, w, world, rank):
    """The oracle as the reference arm: bounded sample on the host cores."""
    if rank != 0:
        return
    t0 = time.perf_counter()
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    offsets, indices, features = build_graph(w, dev)
    pool = target_pool(w, dev)
    targets = targets_for_step(w, pool, 0)
    host_graph = host_copy(offsets, indices, features)
    del offsets, indices, features
    tcpu = targets.cpu().numpy()
    # each step: a bounded sample of the workload's minibatches, ~8 s of host
    # work at most, so --steps K --warmup W ends within a few minutes
    budget = max(2.0, min(8.0, 150.0 / max(1, args.steps)))
    vals, cores, sample = [], 1, ""
    time_oracle(host_graph, w, tcpu, 1.0, 64)
    for _ in range(args.steps):
        v, cores, sample = time_oracle(host_graph, w, tcpu, budget, 8192)
        vals.append(v)
    value = statistics.median(vals)
    out = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": 1e3 * w.H / value,
           "higher_is_better": True, "scaling": "weak",
           "vs_baseline": None, "dtype": "int32", "data": "synthetic", "impl": "reference",
           "config": {"workload": f"{w.name}: {w.describe()}"
                           + (f" features in pinned host memory ({args.feature_io} I/O)"
                              if args.stream else "")
                           + (f" topology in pinned host memory, {args.graph_buffer_gb:g} GB graph buffer"
                              if args.stream_topology else ""), "H": w.H, "B": w.B,
                      "fanouts": list(w.fanouts)},
           "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                            "sample": sample},
           "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0},
           "wall_s": round(time.perf_counter() - t0, 1)}
    print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
