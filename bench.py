"""Benchmark of the gater's hot path on GB300 (one JSON line on rank 0).

Workload (default): 1,000,000 fp32 feature vectors, d = 2048, K = 64 centres,
post-ReLU mixture of 64 Gaussians (about half zeros), the shape of pooled
ResNet-50 features.  One step = one whole job on inputs resident in HBM:
    20 Lloyd iterations (hme_assign + hme_update_centroids; the first assign
    also leaves the prepared features -- row norms, bf16 split -- in the
    workspace for the later ones), then hme_route of all N rows with the final
    centres (assign + expert partition), reusing the prepared features.
The k-means++ seeding is the boundary and is not timed; every step starts
from the same seeded centres.  value = Lloyd iterations per second of the
whole job (all ranks); inputs (8.2 GB) are larger than L2 (129 MB).

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
    ap.add_argument("--config", type=int, default=2, help="workload index 1..5 (2 is the benchmark workload)")
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
    before the warm-up (the tool takes a moment to come up) and only samples
    stamped inside the timed region [begin(), end()] are kept."""

    Q = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.t0 = self.t1 = None
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

    def begin(self):
        self.t0 = time.time()

    def end(self):
        self.t1 = time.time()

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.close()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 10:
                continue
            try:
                ts = datetime.datetime.strptime(parts[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                clk, clkmax = float(parts[2]), float(parts[3])
            except ValueError:
                continue
            if self.t0 is not None and not (self.t0 - 0.03 <= ts <= (self.t1 or ts) + 0.03):
                continue
            sm.append(clk)
            smax.append(clkmax)
            for n, v in zip(names, parts[6:10]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples in the timed region"]}
        sm.sort()
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


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

def run_ours(args, w):
    import torch
    import torch.distributed as dist

    import hme_synth
    from paper_1704_06363_gb300 import hme

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)

    N, d, K, T = w.N, w.d, w.K, w.iters
    hbm, tc, peak_kind, tc_sustained = peaks()
    dt = hme.HME_F32 if w.dtype == "f32" else hme.HME_BF16
    X, _ = hme_synth.make_features(w, device=dev)  # replicas: every rank clusters its own copy
    ws = hme.workspace(hme.HME_OP_ASSIGN, N, d, K, dt, device=dev)  # also sized for hme_route
    wi = hme.workspace(hme.HME_OP_INIT, N, d, K, dt, device=dev)
    C0 = torch.empty(K, d, dtype=torch.float32, device=dev)
    hme.hme_kmeans_init(X, K, 1234 + w.seed, hme.HME_INIT_KMEANSPP_SUBSAMPLE, C0, wi)
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
    if w.tags:
        tag_off, tags = hme_synth.make_tags(w, device=dev)
        wp = hme.workspace(hme.HME_OP_PARTITION, N, 1, K, dt, device=dev)
        p_hist = torch.empty(K, dtype=torch.int64, device=dev)
        p_offs = torch.empty(K + 1, dtype=torch.int64, device=dev)
        p_perm = torch.empty(N, dtype=torch.int32, device=dev)
        tag_off_out = torch.empty_like(tag_off)
        tags_out = torch.empty_like(tags)

    ev_assign, ev_update = [], []
    moved_dev = torch.zeros(1, dtype=torch.int32, device=dev)

    def step(Xs, record=False, diag=False):
        C.copy_(C0)
        for t in range(T):
            labels, prev = labels_buf[t % 2], (labels_buf[(t - 1) % 2] if t > 0 else None)
            if record:
                a0 = torch.cuda.Event(enable_timing=True)
                a1 = torch.cuda.Event(enable_timing=True)
                a0.record(stream)
            # the first assign leaves the prepared features (row norms, bf16 split) in ws
            hme.hme_assign(Xs, C, labels, ws, mind, obj[t:t + 1],
                           flags=hme.HME_ASSIGN_PREPARED if t > 0 else hme.HME_ASSIGN_PREPARE_OUT)
            if record:
                a1.record(stream)
                u1 = torch.cuda.Event(enable_timing=True)
            # first iteration: full pass; then only the rows whose label changed
            hme.hme_update_centroids(Xs, labels, mind, C, ws, counts, nres[t:t + 1], jex[t:t + 1], prev_labels=prev)
            if diag and t == T - 1:  # diagnostic, outside the timed steps
                moved_dev.copy_(ws[32:36].view(torch.int32))
            if record:
                u1.record(stream)
                ev_assign.append((t, a0, a1))
                ev_update.append((t, a1, u1))
        # route the training set with the final centres, reusing its prepared features
        hme.hme_route(Xs, C, expert, offsets, order, ws, flags=hme.HME_ASSIGN_PREPARED)
        if w.tags:  # the experts' shares with their tag lists
            hme.hme_partition(expert, K, p_hist, p_offs, p_perm, wp, None, tag_off, tags, tag_off_out, tags_out)

    clocks = Clocks(local)
    clocks.start()
    for _ in range(max(3, args.warmup)):
        step(X)
    status = hme.hme_sync_status(ws)
    if status != hme.HME_OK:
        raise RuntimeError(f"device status {status} after warm-up: {hme.hme_last_error()}")

    # The step is some 250 small launches (assign, rescore, incremental update
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
            raise RuntimeError(f"device status {status} after the graph warm-up: {hme.hme_last_error()}")

    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    clocks.begin()
    launches0 = hme.hme_launch_count()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        if graph is not None:
            graph.replay()
        else:
            step(X, record=True)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    clocks.end()
    # kernels launched in the timed region: the graph's kernels per replay, or
    # the eager launches counted by the library
    launches = launches_per_step * args.steps if graph is not None else hme.hme_launch_count() - launches0
    ck = clocks.stop()
    ms = max_over_ranks(e0.elapsed_time(e1), dev)
    status = hme.hme_sync_status(ws)
    if status != hme.HME_OK:
        raise RuntimeError(f"device status {status} after the timed steps: {hme.hme_last_error()}")
    # per-call timings and diagnostics: one eager step after the timed region
    # (with graph replays) or the timed eager steps themselves
    if graph is not None:
        step(X, record=True, diag=True)
        torch.cuda.synchronize(dev)
    else:
        step(X, diag=True)
        torch.cuda.synchronize(dev)
    hdr = ws[:16].view(torch.int32).cpu()  # queues of the last assign (the route's): pairs, all-K
    rescored = {"pair": int(hdr[1]), "all_k": int(hdr[3])}
    moved = int(moved_dev.item())  # rows that changed label in the last update of the step

    # outside the timed steps: routing the same rows as a one-off call (no
    # preparation; fp32 rows with K <= 256 are split inside the kernel) against
    # the prepared route the step uses
    route_ms = {}
    for name, fl in (("route_prepared", hme.HME_ASSIGN_PREPARED), ("route_unprepared", 0)):
        r0 = torch.cuda.Event(enable_timing=True)
        r1 = torch.cuda.Event(enable_timing=True)
        r0.record(stream)
        hme.hme_route(X, C, expert, offsets, order, ws, flags=fl)
        r1.record(stream)
        torch.cuda.synchronize(dev)
        route_ms[name] = r0.elapsed_time(r1)
    status = hme.hme_sync_status(ws)
    if status != hme.HME_OK:
        raise RuntimeError(f"device status {status} after the route comparison: {hme.hme_last_error()}")
    # outside the timed steps: serving-style routing of small query batches
    # against the final centres (one call = assign + partition), median of 20
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
            r0 = torch.cuda.Event(enable_timing=True)
            r1 = torch.cuda.Event(enable_timing=True)
            r0.record(stream)
            hme.hme_route(Qb, C, eb, ob, rb, wq)
            r1.record(stream)
            torch.cuda.synchronize(dev)
            lat.append(r0.elapsed_time(r1) * 1000.0)
        if hme.hme_sync_status(wq) != hme.HME_OK:
            raise RuntimeError(f"route of a {B}-row batch: {hme.hme_last_error()}")
        route_ms[f"route_batch{B}_us_median"] = sorted(lat)[len(lat) // 2]
    # outside the timed steps: the same Lloyd iterations with X streamed from
    # page-locked host memory in chunks (hme_kmeans_stream), for feature sets
    # larger than HBM
    stream_stats = None
    if not args.no_stream:
        Xpin = X.to("cpu").pin_memory()
        chunk = max(1, min(N, (1 << 30) // (d * w.elem_bytes)))  # about 1 GB per chunk
        wst = hme.workspace(hme.HME_OP_STREAM, chunk, d, K, dt, device=dev)
        Cst = C0.clone()
        lab_st = torch.empty(N, dtype=torch.int32, device=dev)
        mind_st = torch.empty(N, dtype=torch.float32, device=dev)
        its = 2
        hme.hme_kmeans_stream(Xpin, K, 1, chunk, Cst, lab_st, mind_st, wst)  # warm-up
        Cst.copy_(C0)
        s0 = torch.cuda.Event(enable_timing=True)
        s1 = torch.cuda.Event(enable_timing=True)
        s0.record(stream)
        hme.hme_kmeans_stream(Xpin, K, its, chunk, Cst, lab_st, mind_st, wst)
        s1.record(stream)
        torch.cuda.synchronize(dev)
        if hme.hme_sync_status(wst) != hme.HME_OK:
            raise RuntimeError(f"streamed Lloyd: {hme.hme_last_error()}")
        st_ms = s0.elapsed_time(s1)
        stream_stats = {"iterations_per_s": its / (st_ms / 1000), "ms_per_iteration": st_ms / its,
                        "chunk_rows": chunk, "host_to_device_gbs": its * X.numel() * w.elem_bytes / (st_ms / 1000) / 1e9}
        del Xpin, wst

    # outside the timed steps: the Section 4.2 PCA of the same features (fp32
    # workloads): covariance on the tensor cores, Jacobi eigensolver, projection
    pca_stats = None
    if not args.no_pca and w.dtype == "f32":
        r = min(256, d)
        wsp = hme.workspace(hme.HME_OP_PCA, N, d, r, dt, device=dev)
        mu64 = torch.empty(d, dtype=torch.float64, device=dev)
        cov = torch.empty(d, d, dtype=torch.float64, device=dev)
        mu = torch.empty(d, dtype=torch.float32, device=dev)
        comps = torch.empty(r, d, dtype=torch.float32, device=dev)
        var = torch.empty(r, dtype=torch.float32, device=dev)
        Z = torch.empty(N, r, dtype=torch.float32, device=dev)

        def timed(fn, reps):
            fn()  # warm-up
            q0 = torch.cuda.Event(enable_timing=True)
            q1 = torch.cuda.Event(enable_timing=True)
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
        pca_stats = {"components": r, "fit_ms": fit_ms, "covariance_ms": cov_ms, "jacobi_ms_approx": fit_ms - cov_ms,
                     "jacobi_sweeps": sweeps,
                     "covariance_tflops_gram": 2.0 * N * d * d / (cov_ms / 1000) / 1e12,
                     "covariance_tflops_tensor_issued": issued / (cov_ms / 1000) / 1e12,
                     "transform_ms": tr_ms,
                     "transform_tflops": 2.0 * N * d * r / (tr_ms / 1000) / 1e12,
                     "transform_gbs": (N * d * 4 + N * r * 4) / (tr_ms / 1000) / 1e9,
                     "variance_captured": float(var.sum().item()) / float(torch.diagonal(cov).sum().item())}
        # fractions of the measured peaks (both kernels are tensor-bound; the
        # covariance runs long enough to meet the power cap: sustained peak)
        pca_stats["covariance_frac_of_sustained_bf16"] = pca_stats["covariance_tflops_tensor_issued"] / tc_sustained
        pca_stats["transform_frac_of_sustained_bf16"] = 3 * pca_stats["transform_tflops"] / tc_sustained
        if rank == 0 and not args.no_cpu_baseline:
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
            pca_stats["cpu_oracle"] = {"fit_s_full_n": cov_full + eig_s, "covariance_s_full_n": cov_full,
                                       "eigendecomposition_s": eig_s, "cores": os.cpu_count() or 1,
                                       "sample": f"{ns} of {N} rows; covariance time scaled by N/{ns}"}
        del wsp, cov, Z

    tag_stats = None
    if w.tags:  # Section 4.5 statistics of the final shares, outside the timed steps
        V = w.tag_vocab
        wt = hme.workspace(hme.HME_OP_TAG_HIST, N, V, K, dt, device=dev)
        tcounts = torch.empty(K, V, dtype=torch.int64, device=dev)
        tsp = torch.empty(V, dtype=torch.float64, device=dev)
        hme.hme_tag_cluster_hist(p_offs, tag_off_out, tags_out, K, V, tcounts, wt, tsp)  # warm-up
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        hme.hme_tag_cluster_hist(p_offs, tag_off_out, tags_out, K, V, tcounts, wt, tsp)
        t1.record(stream)
        torch.cuda.synchronize(dev)
        if hme.hme_sync_status(wt) != hme.HME_OK:
            raise RuntimeError(f"tag statistics: {hme.hme_last_error()}")
        t_ms = t0.elapsed_time(t1)
        T_tags = tags.numel()
        nbytes = 4 * T_tags + 8 * (N + 1) + 8 * (K + 1) + 8 * K * V * 2 + 8 * V  # tags, offsets in; counts out, read back
        tag_stats = {"ms": t_ms, "tags": T_tags, "vocabulary": V, "gbs": nbytes / (t_ms / 1000) / 1e9,
                     "tags_per_s": T_tags / (t_ms / 1000), "frac_of_hbm": nbytes / (t_ms / 1000) / 1e9 / hbm}
        if rank == 0 and not args.no_cpu_baseline:
            # the oracle beside it (C, one thread per call) on the first rows' tags
            import oracle
            ns = min(N, 1_000_000)
            lab_h = expert[:ns].cpu().numpy()
            to_h = tag_off[: ns + 1].cpu().numpy()
            tg_h = tags[: int(to_h[-1])].cpu().numpy()
            q0 = time.perf_counter()
            oracle.tag_cluster_hist(lab_h, K, to_h, tg_h, V)
            q1 = time.perf_counter()
            tag_stats["cpu_oracle"] = {"tags_per_s": float(to_h[-1]) / (q1 - q0), "cores": 1,
                                       "sample": f"tags of the first {ns} of {N} rows"}

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
    e = w.elem_bytes
    assign_bytes = N * d * e + K * d * e + 4 * N + 8 * N   # X, C, ||x||^2 in; labels, distances out
    update_bytes = N * d * e + 4 * N + 8 * N + K * d * 4   # a full pass: X and labels in (+ the sorted order), C out
    a_gbs = assign_bytes / (t_assign / 1000) / 1e9
    u_gbs = update_bytes / (t_update / 1000) / 1e9
    # the dominant kernel by GPU time per step: T assign calls vs one full and T-1 incremental updates
    dominant = "assign" if (T - 1) * t_assign + t_assign_first >= t_update + (T - 1) * t_incr else "update"
    if dominant == "assign":
        achieved, traffic = a_gbs, profiled_traffic("assign.cu", "assign_" + w.name)
    else:
        achieved, traffic = u_gbs, profiled_traffic("update.cu", "update_" + w.name)
    flops_assign = 2.0 * N * K * d
    # the assign step is tensor-bound when the tensor work it issues (three
    # split products for fp32 rows) per byte read is above the ridge of the
    # measured peaks; it runs inside a long step, so the sustained bf16 peak
    nprod = 3 if w.dtype == "f32" else 1
    if dominant == "assign" and nprod * flops_assign / assign_bytes > tc_sustained * 1e12 / (hbm * 1e9):
        ach_tf = flops_assign / (t_assign / 1000) / 1e12
        roofline = {"bound": "tensor", "achieved": ach_tf, "peak": tc_sustained, "unit": "TFLOP/s",
                    "frac": ach_tf / tc_sustained, "traffic": traffic, "kernel": dominant,
                    "issued_tflops": nprod * ach_tf, "achieved_note": "2NKd per assign call" +
                    (" (fp32 rows: three bf16 products issued per multiply-add)" if nprod == 3 else ""),
                    "peak_source": f"{peak_kind} (MEASURED_PEAKS.json bf16_tflops_sustained)"
                    if peak_kind == "measured" else "fallback 1.7 PFLOP/s sustained"}
    else:
        roofline = {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s", "frac": achieved / hbm,
                    "traffic": traffic, "kernel": dominant, "peak_source": f"{peak_kind} (MEASURED_PEAKS.json hbm_gbs)"
                    if peak_kind == "measured" else "fallback 6.8 TB/s"}

    # ---- end to end through the C ABI with host buffers ------------------------------
    e2e = None
    if not args.no_e2e:
        Xh = torch.empty(X.shape, dtype=X.dtype, pin_memory=True)
        Xh.copy_(X)
        Xd = torch.empty_like(X)
        out_labels = torch.empty(N, dtype=torch.int32, pin_memory=True)
        out_order = torch.empty(N, dtype=torch.int32, pin_memory=True)
        out_offsets = torch.empty(K + 1, dtype=torch.int64, pin_memory=True)
        out_C = torch.empty(K, d, dtype=torch.float32, pin_memory=True)

        graph_e2e = None
        if graph is not None:  # the same step on the copied-in buffer, as a graph
            torch.cuda.synchronize(dev)
            Xd.copy_(X)
            graph_e2e = torch.cuda.CUDAGraph()
            with torch.cuda.graph(graph_e2e, capture_error_mode="relaxed"):
                step(Xd)

        def e2e_step():
            Xd.copy_(Xh, non_blocking=True)
            if graph_e2e is not None:
                graph_e2e.replay()
            else:
                step(Xd)
            out_labels.copy_(expert, non_blocking=True)
            out_order.copy_(order, non_blocking=True)
            out_offsets.copy_(offsets, non_blocking=True)
            out_C.copy_(C, non_blocking=True)

        e2e_step()
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)
        f0 = torch.cuda.Event(enable_timing=True)
        f1 = torch.cuda.Event(enable_timing=True)
        f0.record(stream)
        for _ in range(args.steps):
            e2e_step()
        f1.record(stream)
        torch.cuda.synchronize(dev)
        ms_e2e = max_over_ranks(f0.elapsed_time(f1), dev)
        e2e = {"value": iters_total / (ms_e2e / 1000.0), "unit": UNIT, "h2d_bytes_per_step": X.numel() * e,
               "d2h_bytes_per_step": 4 * N + 4 * N + 8 * (K + 1) + 4 * K * d, "ms_per_step": ms_e2e / args.steps}
        del Xh, Xd

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        rate, n, cores, _ = oracle_iteration_rate(w, args.cpu_seconds, 1)
        cpu = {"value": rate, "unit": UNIT, "cores": cores, "kind": "oracle",
               "sample": f"{n} of {w.N} rows, one Lloyd iteration (assign + update), scaled by N/{n}"}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": max(3, args.warmup), "ms_per_step": ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16x3" if w.dtype == "f32" else "bf16",
            "data": "synthetic",
            "config": {"workload": w.name, "N": N, "d": d, "K": K, "feature_dtype": w.dtype, "iterations": T,
                       "step": "%d x (assign + update; the first assign also writes the prepared features, updates after the first read only rows whose label changed)"
                    " + route of all N rows" % T + (" + partition of the routed rows with their tag lists"
                                                      if w.tags else ""),
                       "l2": "inputs larger than L2 (%.1f GB of features)" % (X.numel() * e / 1e9),
                       "parallelism": "replicas" if world > 1 else "single GPU",
                       "launch": "CUDA graph replay of the captured step" if graph is not None else "eager launches"},
            "vectors_per_s": N * iters_total / (ms / 1000.0),
            "assign_gflops": flops_assign / (t_assign / 1000.0) / 1e9,
            "kernels_ms": {"assign_call": t_assign, "assign_call_prepare_out": t_assign_first, "update_call_full": t_update, "update_call_incremental": t_incr,
                           **route_ms,
                           "assign_gbs": a_gbs, "update_full_gbs": u_gbs},
            "roofline": roofline,
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": launches,
            "rescored_rows_last_assign": rescored,
            "moved_rows_last_update": moved,
            "tag_statistics": tag_stats,
            "pca": pca_stats,
            "streamed_from_host": stream_stats,
            "clocks": ck,
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
