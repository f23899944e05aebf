"""Benchmark of the gater's hot path on GB300 (one JSON line on rank 0).

Headline workload (default): 50,000,000 bf16 feature vectors, d = 256,
K = 4096 centres, a mixture of 4096 Gaussians with Zipf(1.0) weights (25.6 GB
resident in HBM: the largest of the five feature sets that fits one GPU).
One step = one whole job on inputs resident in HBM:
    w.iters Lloyd iterations (hme_assign + hme_update_centroids; the first
    assign also leaves the prepared features -- row norms, and for fp32 rows
    the bf16 split -- in the workspace for the later ones), then hme_route of
    all N rows with the final centres (assign + full expert partition of
    indices and labels), reusing the prepared features.
The k-means++ seeding is the boundary and is not timed; every step starts
from the same seeded centres.  value = Lloyd iterations per second of the
whole job (all ranks); inputs are larger than L2 (129 MB).  The other
workloads (--extra, default 1-4) are timed the same way in the same run and
reported under other_workloads, each with its own roofline.

--impl reference times the fp64 CPU oracle on the host cores on a bounded
row sample of the same workload, scaled to the full N.
"""
from __future__ import annotations

import argparse
import datetime
import hashlib
import json
import os
import re
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "Lloyd iterations/sec and assigned vectors/sec (N·K·d GFLOP/s, % roofline)"
UNIT = "Lloyd iterations/s"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", type=int, default=5, help="headline workload index 1..5 (5: the largest)")
    ap.add_argument("--extra", default="1,2,3,4", help="other workloads timed in the same run ('' for none)")
    ap.add_argument("--rows", type=int, default=0, help="override N (debug runs only)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-stream", action="store_true", help="skip the streamed-from-host diagnostic")
    ap.add_argument("--no-pca", action="store_true", help="skip the PCA diagnostic")
    ap.add_argument("--no-graph", action="store_true", help="time eager steps instead of CUDA-graph replays")
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="target CPU work of the oracle sample")
    return ap.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return (float(p["hbm_gbs"]), float(p["bf16_tflops"]), "measured",
                float(p.get("bf16_tflops_sustained", p["bf16_tflops"])))
    return 6800.0, 1900.0, "fallback", 1700.0


def profiled_traffic(kernel_file: str, key: str):
    """DRAM bytes per launch from a committed ncu summary, if it matches the current kernel source."""
    prof = os.path.join(ROOT, "profiles", key + ".md")
    if not os.path.exists(prof):
        return None
    text = open(prof).read()
    m = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", text)
    h = re.search(r"source_sha256:\s*([0-9a-f]{64})", text)
    if not m or not h:
        return None
    src = hashlib.sha256(open(os.path.join(ROOT, "paper_1704_06363_gb300", "csrc", kernel_file), "rb").read())
    if src.hexdigest() != h.group(1):
        return None
    return float(m.group(1))


class Clocks:
    """nvidia-smi sampling of SM clock and throttle reasons.  Sampling starts
    before the first warm-up (the tool takes a moment to come up) and runs
    until stop(); window(t0, t1) summarises the samples stamped inside one
    timed region."""

    Q = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.samples = []
        self.path = os.path.join(tempfile.gettempdir(), f"hme_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "25"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.close()
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 10:
                continue
            try:
                ts = datetime.datetime.strptime(parts[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                clk, clkmax = float(parts[2]), float(parts[3])
            except ValueError:
                continue
            reasons = {n for n, v in zip(self.NAMES, parts[6:10]) if v.lower() == "active"}
            self.samples.append((ts, clk, clkmax, reasons))
        try:
            os.remove(self.path)
        except OSError:
            pass

    def window(self, t0: float, t1: float):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sel = [s for s in self.samples if t0 - 0.03 <= s[0] <= t1 + 0.03]
        if not sel:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples in the timed region"]}
        sm = sorted(s[1] for s in sel)
        reasons = set().union(*(s[3] for s in sel))
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": max(s[2] for s in sel), "reasons": sorted(reasons),
                "samples": len(sel)}


def max_over_ranks(ms: float, device=None) -> float:
    """Slowest rank's time: the whole job ends when the last replica ends."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return ms
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ---------------------------------------------------------------------------
# CPU oracle baseline (also the --impl reference arm)
# ---------------------------------------------------------------------------

def oracle_iteration_rate(w, target_s: float, steps: int = 1):
    """Oracle Lloyd iterations/s at full N, from a timed row sample (assign + update)."""
    import numpy as np
    import oracle
    import hme_synth

    oracle.build()
    n = 256
    cores = os.cpu_count() or 1
    X, _ = hme_synth.make_features(w, N=n)
    Xh = hme_synth.host_array(X, w.dtype)
    C0, _ = oracle.kmeanspp(Xh, w.K, 7, True, w.dtype)
    # grow the sample until one iteration takes about target_s / 4, then time `steps` iterations
    while True:
        t0 = time.perf_counter()
        oracle.lloyd(Xh, C0, 1, w.dtype)
        dt = time.perf_counter() - t0
        if dt > target_s / 4 or n >= w.N:
            break
        n = min(w.N, int(n * min(8.0, max(2.0, (target_s / 4) / max(dt, 1e-3)))))
        X, _ = hme_synth.make_features(w, N=n)
        Xh = hme_synth.host_array(X, w.dtype)
    times = []
    for _ in range(max(1, steps)):
        t0 = time.perf_counter()
        oracle.lloyd(Xh, C0, 1, w.dtype)
        times.append(time.perf_counter() - t0)
    per_iter_full = float(np.median(times)) * (w.N / n)
    return 1.0 / per_iter_full, n, cores, times


def run_reference(args, w):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    steps = max(1, args.steps)
    for _ in range(max(0, args.warmup)):
        pass  # the oracle has no warm state beyond the sample sizing pass below
    rate, n, cores, times = oracle_iteration_rate(w, args.cpu_seconds, steps)
    sample = f"{n} of {w.N} rows, one Lloyd iteration (assign + update) per step, scaled by N/{n}"
    line = {
        "impl": "reference", "metric": METRIC, "value": rate, "unit": UNIT, "n_gpus": args.gpus,
        "steps": steps, "warmup": args.warmup, "ms_per_step": 1000 * sum(times) / len(times),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "N": w.N, "d": w.d, "K": w.K, "feature_dtype": w.dtype,
                   "iterations": w.iters},
        "cpu_baseline": {"value": rate, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": rate, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------

def _ev():
    import torch
    return torch.cuda.Event(enable_timing=True)


def measure_workload(args, w, dev, world, rank, clocks, headline):
    """Time `args.steps` steps of workload w (after at least three warm-up
    steps) and return its report.  One step is the whole job on inputs
    resident in HBM: w.iters Lloyd iterations (hme_assign +
    hme_update_centroids), then hme_route of all N rows with the final centres
    (assign + expert partition; for a multilabel workload the shares are then
    partitioned again with their tag lists).  The headline workload also gets
    the end-to-end leg (host buffers), the CPU oracle baseline and the
    streamed-from-host diagnostic."""
    import torch
    import torch.distributed as dist

    import hme_synth
    from paper_1704_06363_gb300 import hme

    stream = torch.cuda.current_stream(dev)
    N, d, K, T = w.N, w.d, w.K, w.iters
    hbm, tc, peak_kind, tc_sustained = peaks()
    dt = hme.HME_F32 if w.dtype == "f32" else hme.HME_BF16
    X, _ = hme_synth.make_features(w, device=dev)  # replicas: every rank clusters its own copy
    ws = hme.workspace(hme.HME_OP_ASSIGN, N, d, K, dt, device=dev)  # also sized for hme_route
    wi = hme.workspace(hme.HME_OP_INIT, N, d, K, dt, device=dev)
    C0 = torch.empty(K, d, dtype=torch.float32, device=dev)
    method = hme.HME_INIT_KMEANSPP_SUBSAMPLE if w.init_subsample else hme.HME_INIT_KMEANSPP
    hme.hme_kmeans_init(X, K, 1234 + w.seed, method, C0, wi)
    del wi
    C = torch.empty_like(C0)
    labels_buf = [torch.empty(N, dtype=torch.int32, device=dev) for _ in range(2)]
    mind = torch.empty(N, dtype=torch.float32, device=dev)
    obj = torch.zeros(T, dtype=torch.float64, device=dev)
    jex = torch.zeros(T, dtype=torch.float64, device=dev)
    counts = torch.empty(K, dtype=torch.int64, device=dev)
    nres = torch.zeros(T, dtype=torch.int32, device=dev)
    expert = torch.empty(N, dtype=torch.int32, device=dev)
    offsets = torch.empty(K + 1, dtype=torch.int64, device=dev)
    order = torch.empty(N, dtype=torch.int32, device=dev)

    # multilabel workloads: the final expert shares carry each point's tag list
    tag_off = tags = None
    wp = hme.workspace(hme.HME_OP_PARTITION, N, 1, K, dt, device=dev)
    p_hist = torch.empty(K, dtype=torch.int64, device=dev)
    p_offs = torch.empty(K + 1, dtype=torch.int64, device=dev)
    p_perm = torch.empty(N, dtype=torch.int32, device=dev)
    p_sorted = torch.empty(N, dtype=torch.int32, device=dev)
    if w.tags:
        tag_off, tags = hme_synth.make_tags(w, device=dev)
        tag_off_out = torch.empty_like(tag_off)
        tags_out = torch.empty_like(tags)

    ev_assign, ev_update, ev_route, ev_tags = [], [], [], []
    # per-iteration diagnostics of the eager step after the timed region
    hdr_it = torch.zeros(T, 3, dtype=torch.int32, device=dev)    # rescored pairs, rescored all-K, moved rows
    bucket_it = torch.zeros(T, 3, dtype=torch.int64, device=dev)  # smallest, median, largest cluster

    def step_head(Xs, record=False, diag=False):
        """The first assign of the job; it also leaves the prepared features
        (row norms, and for fp32 rows with K <= 256 the bf16 split) in ws."""
        C.copy_(C0)
        if record:
            a0, a1 = _ev(), _ev()
            a0.record(stream)
        hme.hme_assign(Xs, C, labels_buf[0], ws, mind, obj[0:1], flags=hme.HME_ASSIGN_PREPARE_OUT)
        if record:
            a1.record(stream)
            ev_assign.append((0, a0, a1))
        if diag:
            hdr_it[0, 0:1].copy_(ws[4:8].view(torch.int32))
            hdr_it[0, 1:2].copy_(ws[12:16].view(torch.int32))

    def step_tail(Xs, record=False, diag=False):
        """The rest of the job: the centre update of iteration 0, iterations
        1 .. T-1, the route of all rows (and the tag-list partition)."""
        for t in range(T):
            labels, prev = labels_buf[t % 2], (labels_buf[(t - 1) % 2] if t > 0 else None)
            if t > 0:
                if record:
                    a0, a1 = _ev(), _ev()
                    a0.record(stream)
                hme.hme_assign(Xs, C, labels, ws, mind, obj[t:t + 1], flags=hme.HME_ASSIGN_PREPARED)
                if record:
                    a1.record(stream)
                    ev_assign.append((t, a0, a1))
                if diag:
                    hdr_it[t, 0:1].copy_(ws[4:8].view(torch.int32))
                    hdr_it[t, 1:2].copy_(ws[12:16].view(torch.int32))
            if record:
                u0, u1 = _ev(), _ev()
                u0.record(stream)
            # first iteration: full pass; then only the rows whose label changed
            hme.hme_update_centroids(Xs, labels, mind, C, ws, counts, nres[t:t + 1], jex[t:t + 1], prev_labels=prev)
            if record:
                u1.record(stream)
                ev_update.append((t, u0, u1))
            if diag:
                if t > 0:
                    hdr_it[t, 2:3].copy_(ws[32:36].view(torch.int32))
                srt = torch.sort(counts).values
                bucket_it[t, 0] = srt[0]
                bucket_it[t, 1] = srt[K // 2]
                bucket_it[t, 2] = srt[K - 1]
        # route the training set with the final centres, reusing its prepared features
        if record:
            r0, r1 = _ev(), _ev()
            r0.record(stream)
        hme.hme_route(Xs, C, expert, offsets, order, ws, flags=hme.HME_ASSIGN_PREPARED)
        if record:
            r1.record(stream)
            ev_route.append((r0, r1))
        if w.tags:  # the experts' shares with their tag lists
            if record:
                g0, g1 = _ev(), _ev()
                g0.record(stream)
            hme.hme_partition(expert, K, p_hist, p_offs, p_perm, wp, None, tag_off, tags, tag_off_out, tags_out)
            if record:
                g1.record(stream)
                ev_tags.append((g0, g1))

    def step(Xs, record=False, diag=False):
        step_head(Xs, record, diag)
        step_tail(Xs, record, diag)

    for _ in range(max(3, args.warmup)):
        step(X)
    status = hme.hme_sync_status(ws)
    if status != hme.HME_OK:
        raise RuntimeError(f"{w.name}: device status {status} after warm-up: {hme.hme_last_error()}")

    # The step is some 100-300 launches (assign, rescore, incremental update
    # kernels per iteration); it is captured once as a CUDA graph and the
    # timed steps replay it.  The library makes no host synchronisation on
    # this path, so the capture holds the whole step.
    graph, launches_per_step = None, None
    if not args.no_graph:
        torch.cuda.synchronize(dev)
        graph = torch.cuda.CUDAGraph()
        l0 = hme.hme_launch_count()
        with torch.cuda.graph(graph, capture_error_mode="relaxed"):
            step(X)
        launches_per_step = hme.hme_launch_count() - l0
        graph.replay()  # one more warm-up step, as a replay
        status = hme.hme_sync_status(ws)
        if status != hme.HME_OK:
            raise RuntimeError(f"{w.name}: device status {status} after the graph warm-up: {hme.hme_last_error()}")

    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    t_begin = time.time()
    launches0 = hme.hme_launch_count()
    e0, e1 = _ev(), _ev()
    e0.record(stream)
    for _ in range(args.steps):
        if graph is not None:
            graph.replay()
        else:
            step(X, record=True)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    t_end = time.time()
    # kernels launched in the timed region: the graph's kernels per replay, or
    # the eager launches counted by the library
    launches = launches_per_step * args.steps if graph is not None else hme.hme_launch_count() - launches0
    ms = max_over_ranks(e0.elapsed_time(e1), dev)
    status = hme.hme_sync_status(ws)
    if status != hme.HME_OK:
        raise RuntimeError(f"{w.name}: device status {status} after the timed steps: {hme.hme_last_error()}")
    # per-call timings and per-iteration diagnostics: one eager step after the
    # timed region (with graph replays) or the timed eager steps themselves
    if graph is not None:
        step(X, record=True, diag=True)
    else:
        step(X, diag=True)
    torch.cuda.synchronize(dev)
    hi = hdr_it.cpu().tolist()
    bi = bucket_it.cpu().tolist()
    jx, ob, nr = jex.cpu().tolist(), obj.cpu().tolist(), nres.cpu().tolist()
    per_iter = [{"iteration": t, "objective_exact": jx[t], "objective_assign_estimate": ob[t],
                 "changed_labels": (hi[t][2] if t > 0 else None), "reseeded": nr[t],
                 "rescored_rows": {"pair": hi[t][0], "all_k": hi[t][1]},
                 "cluster_size": {"min": bi[t][0], "median": bi[t][1], "max": bi[t][2]}} for t in range(T)]
    hdr = ws[:16].view(torch.int32).cpu()  # queues of the last assign (the route's): pairs, all-K
    rescored_route = {"pair": int(hdr[1]), "all_k": int(hdr[3])}

    # the expert partition alone (hme_partition of the routed labels), timed
    # beside the step: median of 10 calls
    pt = []
    for _ in range(11):
        q0, q1 = _ev(), _ev()
        q0.record(stream)
        hme.hme_partition(expert, K, p_hist, p_offs, p_perm, wp, p_sorted)
        q1.record(stream)
        torch.cuda.synchronize(dev)
        pt.append(q0.elapsed_time(q1))
    if hme.hme_sync_status(wp) != hme.HME_OK:
        raise RuntimeError(f"{w.name}: partition: {hme.hme_last_error()}")
    t_part = sorted(pt[1:])[len(pt[1:]) // 2]

    iters_total = T * args.steps * world
    value = iters_total / (ms / 1000.0)
    # the assign kernel on prepared features (iterations 1..T-1); the first call also prepares
    later = [a.elapsed_time(b) for t, a, b in ev_assign if t > 0] or [a.elapsed_time(b) for _, a, b in ev_assign]
    t_assign = sum(later) / len(later)
    first = [a.elapsed_time(b) for t, a, b in ev_assign if t == 0]
    t_assign_first = sum(first) / len(first)
    full = [a.elapsed_time(b) for t, a, b in ev_update if t == 0]
    incr = [a.elapsed_time(b) for t, a, b in ev_update if t > 0]
    t_update = sum(full) / len(full)
    t_incr = sum(incr) / len(incr) if incr else 0.0
    t_route = ev_route[-1][0].elapsed_time(ev_route[-1][1])
    e = w.elem_bytes
    assign_bytes = N * d * e + K * d * e + 4 * N + 8 * N   # X, C, ||x||^2 in; labels, distances out
    update_bytes = N * d * e + 4 * N + 8 * N + K * d * 4   # a full pass: X and labels in (+ the sorted order), C out
    part_bytes = 12 * N + 16 * (K + 1)                     # labels in; order and sorted labels out; hist, offsets
    a_gbs = assign_bytes / (t_assign / 1000) / 1e9
    u_gbs = update_bytes / (t_update / 1000) / 1e9
    p_gbs = part_bytes / (t_part / 1000) / 1e9
    # the dominant kernel by GPU time per step: T assign calls vs one full and T-1 incremental updates
    dominant = "assign" if (T - 1) * t_assign + t_assign_first >= t_update + (T - 1) * t_incr else "update"
    if dominant == "assign":
        achieved, traffic = a_gbs, profiled_traffic("assign.cu", "assign_" + w.name)
    else:
        achieved, traffic = u_gbs, profiled_traffic("update.cu", "update_" + w.name)
    flops_assign = 2.0 * N * K * d
    # The assign step's operands: bf16 features one bf16 product; fp32
    # features with K > 256 one tf32 product (kind::tf32); fp32 features with
    # K <= 256 three products of the bf16 split.  It is tensor-bound when the
    # tensor work it issues per byte read is above the ridge of the peak of its
    # operand type; it runs inside a long step, so the sustained peak (tf32: the
    # sustained bf16 peak times the nominal dense tf32/bf16 ratio 1.1/2.25).
    tf32 = False  # the step uses the default operands (fp32 rows: the bf16 split), not HME_ASSIGN_TF32
    nprod = 3 if (w.dtype == "f32" and not tf32) else 1
    op_peak = tc_sustained * (1.1 / 2.25) if tf32 else tc_sustained
    if dominant == "assign" and nprod * flops_assign / assign_bytes > op_peak * 1e12 / (hbm * 1e9):
        ach_tf = flops_assign / (t_assign / 1000) / 1e12
        roofline = {"bound": "tensor", "achieved": ach_tf, "peak": op_peak, "unit": "TFLOP/s",
                    "frac": ach_tf / op_peak, "traffic": traffic, "kernel": dominant,
                    "operands": "tf32" if tf32 else ("bf16 split, three products" if nprod == 3 else "bf16"),
                    "issued_tflops": nprod * ach_tf, "achieved_note": "2NKd per assign call" +
                    (" (fp32 rows: three bf16 products issued per multiply-add)" if nprod == 3 else ""),
                    "peak_source": (f"{peak_kind} (MEASURED_PEAKS.json bf16_tflops_sustained"
                                    + (" x 1.1/2.25, the nominal dense tf32/bf16 ratio)" if tf32 else ")"))
                    if peak_kind == "measured" else "fallback 1.7 PFLOP/s sustained" + (" x 1.1/2.25" if tf32 else "")}
    else:
        roofline = {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s", "frac": achieved / hbm,
                    "traffic": traffic, "kernel": dominant, "peak_source": f"{peak_kind} (MEASURED_PEAKS.json hbm_gbs)"
                    if peak_kind == "measured" else "fallback 6.8 TB/s"}
    if N * d * e < 4 * 129e6:
        roofline["note"] = "inputs of a few L2 sizes: launch- and latency-bound"

    res = {
        "workload": w.name, "N": N, "d": d, "K": K, "feature_dtype": w.dtype, "iterations": T,
        "value": value, "unit": UNIT, "ms_per_step": ms / args.steps, "steps": args.steps,
        "vectors_per_s": N * iters_total / (ms / 1000.0),
        "assign_gflops": flops_assign / (t_assign / 1000.0) / 1e9,
        "kernels_ms": {"assign_call": t_assign, "assign_call_prepare_out": t_assign_first,
                       "update_call_full": t_update, "update_call_incremental": t_incr,
                       "route_call": t_route, "partition_call": t_part,
                       **({"partition_with_tags_call": ev_tags[-1][0].elapsed_time(ev_tags[-1][1])} if ev_tags else {})},
        "hbm_fractions": {"assign": a_gbs / hbm, "update_full": u_gbs / hbm, "partition": p_gbs / hbm,
                          "assign_gbs": a_gbs, "update_full_gbs": u_gbs, "partition_gbs": p_gbs,
                          "note": "algorithmic bytes / CUDA-event time of the call: assign N d e + K d e + 12 N, "
                                  "full update N d e + 12 N + 4 K d, partition 12 N + 16 (K + 1)"},
        "roofline": roofline,
        "gpu_launches": launches,
        "per_iteration": per_iter,
        "rescored_rows_route": rescored_route,
        "l2": "inputs larger than L2 (%.1f GB of features)" % (X.numel() * e / 1e9),
        "launch": "CUDA graph replay of the captured step" if graph is not None else "eager launches",
        "timed_region": (t_begin, t_end),
    }

    if headline:
        # outside the timed steps: routing the same rows as a one-off call (no
        # preparation; fp32 rows with K <= 256 are split inside the kernel)
        # against the prepared route the step uses
        route_ms = {}
        for name, fl in (("route_prepared", hme.HME_ASSIGN_PREPARED), ("route_unprepared", 0)):
            r0, r1 = _ev(), _ev()
            r0.record(stream)
            hme.hme_route(X, C, expert, offsets, order, ws, flags=fl)
            r1.record(stream)
            torch.cuda.synchronize(dev)
            route_ms[name] = r0.elapsed_time(r1)
        if hme.hme_sync_status(ws) != hme.HME_OK:
            raise RuntimeError(f"route comparison: {hme.hme_last_error()}")
        # serving-style routing of small query batches against the final
        # centres (one call = assign + partition), median of 20
        for B in (256, 4096):
            if B > N:
                continue
            Qb = X[:B]
            wq = hme.workspace(hme.HME_OP_ROUTE, B, d, K, dt, device=dev)
            eb = torch.empty(B, dtype=torch.int32, device=dev)
            ob = torch.empty(K + 1, dtype=torch.int64, device=dev)
            rb = torch.empty(B, dtype=torch.int32, device=dev)
            hme.hme_route(Qb, C, eb, ob, rb, wq)
            lat = []
            for _ in range(20):
                r0, r1 = _ev(), _ev()
                r0.record(stream)
                hme.hme_route(Qb, C, eb, ob, rb, wq)
                r1.record(stream)
                torch.cuda.synchronize(dev)
                lat.append(r0.elapsed_time(r1) * 1000.0)
            if hme.hme_sync_status(wq) != hme.HME_OK:
                raise RuntimeError(f"route of a {B}-row batch: {hme.hme_last_error()}")
            route_ms[f"route_batch{B}_us_median"] = sorted(lat)[len(lat) // 2]
        res["kernels_ms"].update(route_ms)

        # ---- end to end through the C ABI with host buffers ------------------------
        Xh = None
        if not args.no_e2e or not args.no_stream:
            Xh = torch.empty(X.shape, dtype=X.dtype, pin_memory=True)
            Xh.copy_(X)
        if not args.no_e2e:
            # The job with X in page-locked host memory: X is copied in by
            # chunks of about 512 MB on a copy stream, and the first assign
            # takes each chunk as soon as it has landed (hme_assign_rows,
            # leaving that chunk's prepared features in ws); the rest of the
            # step runs on the copied-in X as in the timed steps (replayed as a
            # graph).  Labels, order, offsets and centres are copied out.
            Xd = torch.empty_like(X)
            out_labels = torch.empty(N, dtype=torch.int32, pin_memory=True)
            out_order = torch.empty(N, dtype=torch.int32, pin_memory=True)
            out_offsets = torch.empty(K + 1, dtype=torch.int64, pin_memory=True)
            out_C = torch.empty(K, d, dtype=torch.float32, pin_memory=True)
            nch = int(max(1, min(64, (X.numel() * e) // (512 << 20))))
            bounds = [N * j // nch for j in range(nch + 1)]
            copy_stream = torch.cuda.Stream(dev)
            landed = [torch.cuda.Event() for _ in range(nch)]
            graph_tail = None
            if graph is not None:  # the rest of the step on the copied-in buffer, as a graph
                torch.cuda.synchronize(dev)
                Xd.copy_(X)
                step_head(Xd)
                graph_tail = torch.cuda.CUDAGraph()
                with torch.cuda.graph(graph_tail, capture_error_mode="relaxed"):
                    step_tail(Xd)

            def e2e_step():
                C.copy_(C0)
                copy_stream.wait_stream(stream)  # the previous step is done with Xd
                for j in range(nch):
                    r0, r1 = bounds[j], bounds[j + 1]
                    with torch.cuda.stream(copy_stream):
                        Xd[r0:r1].copy_(Xh[r0:r1], non_blocking=True)
                        landed[j].record(copy_stream)
                    stream.wait_event(landed[j])
                    hme.hme_assign_rows(Xd, r0, r1, C, labels_buf[0], ws, mind, flags=hme.HME_ASSIGN_PREPARE_OUT)
                if graph_tail is not None:
                    graph_tail.replay()
                else:
                    step_tail(Xd)
                out_labels.copy_(expert, non_blocking=True)
                out_order.copy_(order, non_blocking=True)
                out_offsets.copy_(offsets, non_blocking=True)
                out_C.copy_(C, non_blocking=True)

            e2e_step()
            if world > 1:
                dist.barrier()
            torch.cuda.synchronize(dev)
            f0, f1 = _ev(), _ev()
            f0.record(stream)
            for _ in range(args.steps):
                e2e_step()
            f1.record(stream)
            torch.cuda.synchronize(dev)
            if hme.hme_sync_status(ws) != hme.HME_OK:
                raise RuntimeError(f"end-to-end step: {hme.hme_last_error()}")
            ms_e2e = max_over_ranks(f0.elapsed_time(f1), dev)
            res["e2e"] = {"value": iters_total / (ms_e2e / 1000.0), "unit": UNIT,
                          "h2d_bytes_per_step": X.numel() * e,
                          "d2h_bytes_per_step": 4 * N + 4 * N + 8 * (K + 1) + 4 * K * d,
                          "ms_per_step": ms_e2e / args.steps,
                          "overlap": f"host-to-device copy in {nch} chunks on a copy stream, the first assign "
                                     "taking each chunk as it lands (hme_assign_rows)"}
            del Xd, graph_tail
        # outside the timed steps: the same Lloyd iterations with X streamed
        # from page-locked host memory in chunks (hme_kmeans_stream), for
        # feature sets larger than HBM
        if not args.no_stream:
            chunk = max(1, min(N, (1 << 30) // (d * w.elem_bytes)))  # about 1 GB per chunk
            wst = hme.workspace(hme.HME_OP_STREAM, chunk, d, K, dt, device=dev)
            Cst = C0.clone()
            lab_st = torch.empty(N, dtype=torch.int32, device=dev)
            mind_st = torch.empty(N, dtype=torch.float32, device=dev)
            its = 2
            hme.hme_kmeans_stream(Xh, K, 1, chunk, Cst, lab_st, mind_st, wst)  # warm-up
            Cst.copy_(C0)
            s0, s1 = _ev(), _ev()
            s0.record(stream)
            hme.hme_kmeans_stream(Xh, K, its, chunk, Cst, lab_st, mind_st, wst)
            s1.record(stream)
            torch.cuda.synchronize(dev)
            if hme.hme_sync_status(wst) != hme.HME_OK:
                raise RuntimeError(f"streamed Lloyd: {hme.hme_last_error()}")
            st_ms = s0.elapsed_time(s1)
            res["streamed_from_host"] = {
                "iterations_per_s": its / (st_ms / 1000), "ms_per_iteration": st_ms / its, "chunk_rows": chunk,
                "host_to_device_gbs": its * X.numel() * w.elem_bytes / (st_ms / 1000) / 1e9}
            del wst
        del Xh

    # the Section 4.2 PCA of the fp32 ResNet-style features (outside the
    # timed steps): covariance on the tensor cores, Jacobi eigensolver, projection
    if not args.no_pca and w.dtype == "f32" and d >= 1024:
        res["pca"] = pca_diagnostic(args, X, dev, rank, world, hbm, tc_sustained)

    if w.tags:  # Section 4.5 statistics of the final shares, outside the timed steps
        V = w.tag_vocab
        wt = hme.workspace(hme.HME_OP_TAG_HIST, N, V, K, dt, device=dev)
        tcounts = torch.empty(K, V, dtype=torch.int64, device=dev)
        tsp = torch.empty(V, dtype=torch.float64, device=dev)
        hme.hme_tag_cluster_hist(p_offs, tag_off_out, tags_out, K, V, tcounts, wt, tsp)  # warm-up
        t0, t1 = _ev(), _ev()
        t0.record(stream)
        hme.hme_tag_cluster_hist(p_offs, tag_off_out, tags_out, K, V, tcounts, wt, tsp)
        t1.record(stream)
        torch.cuda.synchronize(dev)
        if hme.hme_sync_status(wt) != hme.HME_OK:
            raise RuntimeError(f"tag statistics: {hme.hme_last_error()}")
        t_ms = t0.elapsed_time(t1)
        T_tags = tags.numel()
        nbytes = 4 * T_tags + 8 * (N + 1) + 8 * (K + 1) + 8 * K * V * 2 + 8 * V  # tags, offsets in; counts out, read back
        ts = {"ms": t_ms, "tags": T_tags, "vocabulary": V, "gbs": nbytes / (t_ms / 1000) / 1e9,
              "tags_per_s": T_tags / (t_ms / 1000), "frac_of_hbm": nbytes / (t_ms / 1000) / 1e9 / hbm}
        if rank == 0 and world == 1 and not args.no_cpu_baseline:
            # the oracle beside it (C, one thread per call) on the first rows' tags
            import oracle
            ns = min(N, 1_000_000)
            lab_h = expert[:ns].cpu().numpy()
            to_h = tag_off[: ns + 1].cpu().numpy()
            tg_h = tags[: int(to_h[-1])].cpu().numpy()
            q0 = time.perf_counter()
            oracle.tag_cluster_hist(lab_h, K, to_h, tg_h, V)
            q1 = time.perf_counter()
            ts["cpu_oracle"] = {"tags_per_s": float(to_h[-1]) / (q1 - q0), "cores": 1,
                                "sample": f"tags of the first {ns} of {N} rows"}
        res["tag_statistics"] = ts
        del wt, tcounts
    del X, ws, wp, graph
    torch.cuda.synchronize(dev)
    torch.cuda.empty_cache()
    return res


def pca_diagnostic(args, X, dev, rank, world, hbm, tc_sustained):
    import torch

    from paper_1704_06363_gb300 import hme

    stream = torch.cuda.current_stream(dev)
    N, d = X.shape
    r = min(256, d)
    wsp = hme.workspace(hme.HME_OP_PCA, N, d, r, hme.HME_F32, device=dev)
    mu64 = torch.empty(d, dtype=torch.float64, device=dev)
    cov = torch.empty(d, d, dtype=torch.float64, device=dev)
    mu = torch.empty(d, dtype=torch.float32, device=dev)
    comps = torch.empty(r, d, dtype=torch.float32, device=dev)
    var = torch.empty(r, dtype=torch.float32, device=dev)
    Z = torch.empty(N, r, dtype=torch.float32, device=dev)

    def timed(fn, reps):
        fn()  # warm-up
        q0, q1 = _ev(), _ev()
        q0.record(stream)
        for _ in range(reps):
            out = fn()
        q1.record(stream)
        torch.cuda.synchronize(dev)
        return q0.elapsed_time(q1) / reps, out

    cov_ms, _ = timed(lambda: hme.hme_pca_covariance(X, mu64, cov, wsp), 3)
    fit_ms, sweeps = timed(lambda: hme.hme_pca_fit(X, r, mu, comps, wsp, var), 1)
    tr_ms, _ = timed(lambda: hme.hme_pca_transform(X, mu, comps, Z, wsp), 5)
    if hme.hme_sync_status(wsp) != hme.HME_OK:
        raise RuntimeError(f"pca: {hme.hme_last_error()}")
    mi = (d + 127) // 128
    issued = 3 * 2.0 * N * 128 * 128 * mi * (mi + 1) // 2  # three split products on the upper-triangle tiles
    st = {"rows": N, "d": d, "components": r, "fit_ms": fit_ms, "covariance_ms": cov_ms,
          "jacobi_ms_approx": fit_ms - cov_ms, "jacobi_sweeps": sweeps,
          "covariance_tflops_gram": 2.0 * N * d * d / (cov_ms / 1000) / 1e12,
          "covariance_tflops_tensor_issued": issued / (cov_ms / 1000) / 1e12,
          "transform_ms": tr_ms,
          "transform_tflops": 2.0 * N * d * r / (tr_ms / 1000) / 1e12,
          "transform_gbs": (N * d * 4 + N * r * 4) / (tr_ms / 1000) / 1e9,
          "variance_captured": float(var.sum().item()) / float(torch.diagonal(cov).sum().item())}
    # fractions of the measured peaks (both kernels are tensor-bound; the
    # covariance runs long enough to meet the power cap: sustained peak)
    st["covariance_frac_of_sustained_bf16"] = st["covariance_tflops_tensor_issued"] / tc_sustained
    st["transform_frac_of_sustained_bf16"] = 3 * st["transform_tflops"] / tc_sustained
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        # the oracle beside it: fp64 numpy PCA (covariance by matrix product,
        # eigh) on a row sample; the covariance part scales with N, the
        # eigendecomposition does not
        import oracle.pca as opca
        ns = min(N, 20000)
        Xs = X[:ns].cpu().numpy()
        q0 = time.perf_counter()
        mu_s, cov_s = opca.covariance(Xs)
        q1 = time.perf_counter()
        opca.fit(Xs, r)
        q2 = time.perf_counter()
        cov_full = (q1 - q0) * N / ns
        eig_s = max(q2 - q1 - (q1 - q0), 0.0)
        st["cpu_oracle"] = {"fit_s_full_n": cov_full + eig_s, "covariance_s_full_n": cov_full,
                            "eigendecomposition_s": eig_s, "cores": os.cpu_count() or 1,
                            "sample": f"{ns} of {N} rows; covariance time scaled by N/{ns}"}
    del wsp, cov, Z
    return st


def run_ours(args, w):
    import torch
    import torch.distributed as dist

    import hme_synth

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    clocks = Clocks(local)
    clocks.start()
    head = measure_workload(args, w, dev, world, rank, clocks, headline=True)
    # the other workloads, one after another in the same run (single GPU
    # runs only: under torchrun every rank holds a GPU for the headline alone)
    others = []
    if world == 1 and args.extra:
        for wid in [int(v) for v in args.extra.split(",") if v.strip()]:
            wx = hme_synth.WORKLOADS[wid]
            if wx.name != w.name:
                others.append(measure_workload(args, wx, dev, world, rank, clocks, headline=False))
    clocks.stop()

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        rate, n, cores, _ = oracle_iteration_rate(w, args.cpu_seconds, 1)
        cpu = {"value": rate, "unit": UNIT, "cores": cores, "kind": "oracle",
               "sample": f"{n} of {w.N} rows, one Lloyd iteration (assign + update), scaled by N/{n}"}

    if rank == 0:
        ck = clocks.window(*head.pop("timed_region"))
        extra = {}
        for o in others:
            o["clocks"] = clocks.window(*o.pop("timed_region"))
            extra[o["workload"]] = o
        T = w.iters
        line = {
            "metric": METRIC, "value": head["value"], "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": max(3, args.warmup), "ms_per_step": head["ms_per_step"], "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16x3" if w.dtype == "f32" else "bf16",
            "data": "synthetic",
            "config": {"workload": w.name, "N": w.N, "d": w.d, "K": w.K, "feature_dtype": w.dtype, "iterations": T,
                       "step": "%d x (assign + update; the first assign also writes the prepared features, updates "
                               "after the first read only rows whose label changed) + route of all N rows with the "
                               "final centres (assign + full partition of indices and labels)" % T
                               + (" + partition of the routed rows with their tag lists" if w.tags else ""),
                       "l2": head["l2"],
                       "parallelism": "replicas" if world > 1 else "single GPU",
                       "launch": head["launch"]},
            "vectors_per_s": head["vectors_per_s"],
            "assign_gflops": head["assign_gflops"],
            "kernels_ms": head["kernels_ms"],
            "hbm_fractions": head["hbm_fractions"],
            "roofline": head["roofline"],
            "cpu_baseline": cpu,
            "e2e": head.get("e2e"),
            "gpu_launches": head["gpu_launches"],
            "per_iteration": head["per_iteration"],
            "rescored_rows_route": head["rescored_rows_route"],
            "streamed_from_host": head.get("streamed_from_host"),
            "clocks": ck,
            "other_workloads": extra,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


def main():
    args = parse()
    import hme_synth
    w = hme_synth.WORKLOADS[args.config]
    if args.rows:
        w = w.with_rows(args.rows)
    if args.impl == "reference":
        run_reference(args, w)
    else:
        run_ours(args, w)


if __name__ == "__main__":
    main()
