"""Benchmark of the FASGD parameter-server pass on one or more GB300 GPUs.

Default workload: P = 25,000,000 fp32 parameters with their FASGD statistics
(theta, n, b, v), lambda = 128 clients, K = 8 pending pushes fused into one
pass, Geometric(0.05) staleness capped at 512.  One step = K pushes queued
through the C ABI and one fasgd_apply_pending(K) call: one fused kernel that
reads theta, n, b, v and the K gradient slices once and writes the state once.

Printed (rank 0, one JSON line): parameter-updates/s of the whole job, with
achieved HBM GB/s of the fused kernel against the measured copy bandwidth,
the same metric end to end from pinned host buffers, and the CPU oracle
timed on a bounded sample of the same workload.

Multi-GPU (torchrun): the parameter vector is sharded, each rank owning
P parameters and applying the same pushes to its shard; no collective sits on
the data path (barriers and a max of the timings only).

--impl reference times the CPU oracle instead (rank 0 only).
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_1601_04033_gb300 import streams  # noqa: E402

METRIC = "parameter-updates/sec and achieved HBM GB/s (% of GB300 peak), 1 GPU"
UNIT = "param-updates/s"
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 7900.0    # GB300 HBM3e nominal bandwidth: context only, frac uses the measured peak
FETCH_FRACTION = 0.10   # a 10x cut of fetch traffic (the paper's effective setting, Sec. 4.2)
L2_BYTES = 129 * 1024 * 1024

DENSE_KERNEL_SOURCES = ["paper_1601_04033_gb300/csrc/dense.cu",
                        "paper_1601_04033_gb300/csrc/update.cuh",
                        "paper_1601_04033_gb300/csrc/wait.cuh",
                        "paper_1601_04033_gb300/csrc/kernels.cuh"]
SPARSE_KERNEL_SOURCES = ["paper_1601_04033_gb300/csrc/select.cu",
                         "paper_1601_04033_gb300/csrc/sparse.cu",
                         "paper_1601_04033_gb300/csrc/update.cuh",
                         "paper_1601_04033_gb300/csrc/kernels.cuh"]


# ---------------------------------------------------------------------------
# helpers
# ---------------------------------------------------------------------------
def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def init_dist(world, backend):
    import torch.distributed as dist
    if world > 1 and not dist.is_initialized():
        dist.init_process_group(backend=backend)
    return dist


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int, device=None) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def shard_workload(w: streams.Workload, rank: int) -> streams.Workload:
    """Rank r owns parameters [r*P, (r+1)*P) of an N*P vector: its own slice of
    every gradient and of theta0, the same push sequence on every rank."""
    return w if rank == 0 else w.replace(seed=w.seed + 7919 * rank)


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def physical(roofline: dict) -> dict:
    """Add the DRAM bandwidth the ncu traffic of one launch implies at the
    live launch time, beside the algorithmic figure (when traffic is known)."""
    t, ms = roofline.get("traffic"), roofline.get("launch_ms")
    if t and ms:
        gbs = t / (ms / 1e3) / 1e9
        roofline["traffic_gbs"] = round(gbs, 1)
        roofline["traffic_frac"] = round(gbs / roofline["peak"], 4)
    return roofline


def nominal(achieved: float) -> dict:
    """The same achieved bandwidth against the GB300's nominal HBM3e figure."""
    return {"nominal_peak": NOMINAL_HBM_GBS, "frac_nominal": round(achieved / NOMINAL_HBM_GBS, 4)}


def sources_hash(paths) -> str:
    h = hashlib.sha256()
    for p in paths:
        with open(os.path.join(ROOT, p), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(workload: str, kernel_sources) -> float | None:
    """DRAM bytes per launch from a committed ncu summary, if the kernel
    sources are unchanged since it was taken (else None)."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
        e = d[workload]
        if e["sources_sha256_16"] != sources_hash(kernel_sources):
            return None
        return float(e["dram_bytes_per_launch"])
    except Exception:
        return None


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during a region."""

    FIELDS = ["clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.active",
              "clocks_event_reasons.hw_slowdown", "clocks_event_reasons.hw_thermal_slowdown",
              "clocks_event_reasons.sw_thermal_slowdown", "clocks_event_reasons.sw_power_cap"]

    def __init__(self, gpu_id: str):
        self.gpu_id = gpu_id
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", self.gpu_id, "--query-gpu=" + ",".join(self.FIELDS),
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.thread.join(timeout=2)
        sm, smax, reasons, power = [], [], set(), []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) != len(self.FIELDS):
                continue
            try:
                sm.append(float(parts[0]))
                smax.append(float(parts[1]))
                power.append(float(parts[2]))
            except ValueError:
                continue
            for name, val in zip(names, parts[4:]):
                if val.lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "power_w_max": max(power) if power else None,
                "samples": len(sm), "reasons": sorted(reasons)}


def gpu_identifier(torch) -> str:
    try:
        u = str(torch.cuda.get_device_properties(torch.cuda.current_device()).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        return str(torch.cuda.current_device())


VARIANTS = {"asgd": streams.ASGD, "sasgd": streams.SASGD, "fasgd": streams.FASGD,
            "fasgd-std": streams.FASGD_STD}


def algorithmic_bytes_dense(P: int, K: int, fasgd_rule: bool) -> int:
    """theta (+ n, b, v) read and written once, K gradient slices read once."""
    state = 4 if fasgd_rule else 1
    return P * (8 * state + 4 * K)


# ---------------------------------------------------------------------------
# CPU oracle legs (reference arm and cpu_baseline)
# ---------------------------------------------------------------------------
def oracle_rate(w: streams.Workload, P_sample: int, batches: int | None, seconds: float | None,
                variant: int = streams.FASGD, warmup: int = 0, max_batches: int = 4096):
    """Time the oracle on the first P_sample parameters of the workload, K
    pushes per batch, for a number of batches or of seconds; returns
    (param-updates/s, batches timed, seconds)."""
    import oracle
    K = w.K
    R = max(w.R, 2 * K)
    pool = streams.gradient_pool(w, P_sample, R)
    th0 = streams.theta0(w, P_sample)
    n_batches = warmup + (batches if batches is not None else max_batches)
    ps = streams.push_stream(w.replace(R=R), n_batches * K, K)
    srv = oracle.OracleServer(P_sample, w.lam, w.alpha, variant)
    srv.set_params(th0)

    def run_batch(b):
        for c, j, s in zip(*ps.batch(b)):
            srv.push(int(c), int(j), pool[int(s)])
        srv.apply_pending(K)

    for b in range(warmup):
        run_batch(b)
    t0 = time.perf_counter()
    done = 0
    while warmup + done < n_batches:
        run_batch(warmup + done)
        done += 1
        if batches is None and time.perf_counter() - t0 >= seconds:
            break
    el = time.perf_counter() - t0
    return P_sample * K * done / el, done, el


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------
SMALL_P = 1 << 21   # dense workloads at or below this size also run the C driver


def run_abi_latency(P: int, K: int, variant: int, steps: int) -> dict | None:
    """The C timing driver of the ABI (abi_latency.c) on the same shape."""
    from paper_1601_04033_gb300 import build
    try:
        exe = build.build_latency_driver()
        out = subprocess.run([exe, str(P), str(K), str(steps), str(variant)], capture_output=True,
                             text=True, timeout=300)
    except Exception as e:      # reported, not fatal: the Python numbers stand alone
        return {"error": str(e)[:200]}
    if out.returncode != 0:
        return {"error": out.stderr.strip()[-200:]}
    return json.loads(out.stdout.strip().splitlines()[-1])


def run_dense(args, w, world, rank, local):
    import torch
    from paper_1601_04033_gb300 import fasgd

    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    K, P = w.K, (args.P or w.P)
    variant = VARIANTS[args.variant]
    fasgd_rule = variant in (streams.FASGD, streams.FASGD_STD)
    wr = shard_workload(w, rank)
    pool = streams.gradient_pool(wr, P, w.R)
    th0 = streams.theta0(wr, P)
    n_batches = args.warmup + args.steps
    ps = streams.push_stream(w, n_batches * K, K)
    pool_t, slots = fasgd.aligned_vectors(pool, device)
    stream = torch.cuda.current_stream()
    srv = fasgd.Server(P, w.lam, w.alpha, variant, stream=stream)
    srv.set_exact(args.exact)
    srv.set_params(torch.from_numpy(th0).to(device))
    batches = [ps.batch(b) for b in range(n_batches)]
    batches = [([int(c) for c in cl], [int(j) for j in js], [int(s) for s in sl])
               for cl, js, sl in batches]

    def step(b):
        cl, js, sl = batches[b]
        for c, j, s in zip(cl, js, sl):
            srv.push(c, j, slots[s])
        srv.apply_pending(K)

    for b in range(args.warmup):
        step(b)
    torch.cuda.synchronize()
    clocks = ClockSampler(gpu_identifier(torch))
    ev_a = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ev_b = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    launches0 = srv.launches
    barrier(world)
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)   # let the sampler take its first reading
    start.record(stream)
    h0 = time.perf_counter()
    for i in range(args.steps):
        b = args.warmup + i
        cl, js, sl = batches[b]
        for c, j, s in zip(cl, js, sl):
            srv.push(c, j, slots[s])
        ev_a[i].record(stream)
        srv.apply_pending(K)
        ev_b[i].record(stream)
    host_us = (time.perf_counter() - h0) * 1e6 / args.steps
    end.record(stream)
    torch.cuda.synchronize()
    clock_info = clocks.stop()
    barrier(world)
    launches = srv.launches - launches0
    total_ms = start.elapsed_time(end)
    kern_ms = [a.elapsed_time(b) for a, b in zip(ev_a, ev_b)]
    total_ms = max_over_ranks(total_ms, world, device)
    kern_avg_ms = max_over_ranks(sum(kern_ms) / len(kern_ms), world, device)

    # End to end through the C ABI with host buffers: K gradients copied from
    # pinned host memory into device staging per step, theta pulled back.
    e2e = None
    if args.e2e_steps > 0:
        host_pool = torch.from_numpy(pool).pin_memory()
        host_slots = [host_pool[r] for r in range(host_pool.shape[0])]
        out = torch.empty(P, dtype=torch.float32).pin_memory()
        T0 = srv.T
        e2e_warm = 4    # enough steps for the staging pool to reach its steady size
        e2e_ps = streams.push_stream(w, (args.e2e_steps + e2e_warm) * K, K)

        def e2e_step(b):
            cl, js, sl = e2e_ps.batch(b)
            Tn = srv.T
            for c, j, s in zip(cl, js, sl):
                srv.push_host(int(c), int(min(j + T0, Tn)), host_slots[int(s)])
            srv.apply_pending(K)
            srv.pull(out)

        for b in range(e2e_warm):
            e2e_step(b)
        torch.cuda.synchronize()
        barrier(world)
        t0 = time.perf_counter()
        e_start, e_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e_start.record(stream)
        for b in range(args.e2e_steps):
            e2e_step(e2e_warm + b)
        e_end.record(stream)
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
        e_ms = max_over_ranks(max(e_start.elapsed_time(e_end), wall * 1e3), world, device)
        e2e = {"value": P * world * K * args.e2e_steps / (e_ms / 1e3), "unit": UNIT,
               "h2d_bytes_per_step": K * P * 4, "d2h_bytes_per_step": P * 4,
               "steps": args.e2e_steps, "ms_per_step": e_ms / args.e2e_steps}
    srv.sync()
    srv.close()
    # Small passes are bound by call latency: time the same steps from C
    # through the ABI (host cost of the calls, GPU time of an eager loop and
    # of a graph replay of the same launches) to split it from the binding's.
    abi_latency = None
    if P <= SMALL_P and world == 1 and not args.no_abi_latency:
        abi_latency = run_abi_latency(P, K, variant, max(args.steps, 1000))

    step_s = total_ms / 1e3 / args.steps
    value = P * world * K / step_s
    alg = algorithmic_bytes_dense(P, K, fasgd_rule)
    peak, peak_kind = peaks()
    achieved = alg / (kern_avg_ms / 1e3) / 1e9
    tkey = w.name if not args.P else f"{w.name}-P{P}"
    if args.variant != "fasgd":
        tkey += "-" + ("sgd" if not fasgd_rule else args.variant)
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4), "peak_source": peak_kind, **nominal(achieved),
                "kernel": "fasgd_dense_kernel<%s> (bulk-copy ring)"
                          % ("FASGD" if variant == streams.FASGD else
                             "FASGD_STD" if variant == streams.FASGD_STD else "SGD"),
                "bytes_per_launch": alg, "launch_ms": round(kern_avg_ms, 5),
                "traffic": profiled_traffic(tkey, DENSE_KERNEL_SOURCES)}
    return {
        "value": value, "ms_per_step": total_ms / args.steps, "roofline": roofline,
        "clocks": clock_info, "e2e": e2e, "gpu_launches": launches,
        "pushes_per_s": world * K / step_s,
        "hbm_gbs_step": alg * world / step_s / 1e9,
        "host_us_per_step": round(host_us, 3), "abi_latency": abi_latency,
        "config": {"workload": w.name, "P_per_gpu": P, "P_total": P * world, "lambda": w.lam,
                   "K": K, "variant": args.variant, "alpha": w.alpha, "staleness": w.delay,
                   "gradient_pool_slots": w.R, "pushes_timed": K * args.steps,
                   "parallelism": f"param-shard{world}",
                   "arithmetic": "exact (IEEE sqrt/div, unfused)" if args.exact else
                   "fast (hardware rsqrt/rcp, n and b exact)",
                   "l2": "inputs larger than L2 (%.2f GB per step vs 129 MB L2), no flush"
                   % (alg / 1e9) if alg > 4 * L2_BYTES else "working set may be L2-resident"},
    }


def run_bfasgd(args, w, world, rank, local):
    import torch
    from paper_1601_04033_gb300 import fasgd
    from paper_1601_04033_gb300.calibrate import calibrate_c

    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    P = args.P or w.P
    wr = shard_workload(w, rank)
    R = min(w.R, 8)
    pool = streams.gradient_pool(wr, P, R)
    th0 = streams.theta0(wr, P)
    n_steps = args.warmup + args.steps + w.lam + 100   # + the instrumented stage run
    ps = streams.push_stream(w.replace(R=R), n_steps, 1)
    pool_t, slots = fasgd.aligned_vectors(pool, device)
    stream = torch.cuda.current_stream()
    srv = fasgd.Server(P, w.lam, w.alpha, streams.FASGD, stream=stream, seed=w.seed)
    srv.set_params(torch.from_numpy(th0).to(device))
    # Dense FASGD warm-up of lambda pushes, then c tuned on the live v for the target rate.
    t = 0
    for _ in range(w.lam):
        cl, js, sl = ps.batch(t)
        srv.push(int(cl[0]), int(js[0]), slots[int(sl[0])])
        srv.apply_pending(1)
        t += 1
    v_now = torch.empty(P, device=device)
    srv.get_state(None, None, None, v_now)
    v_host = v_now.cpu().numpy()
    # Large P: calibrate on a strided sample of about 4M parameters (the measured
    # send and fetch fractions are reported either way).
    v_cal = v_host if P <= (1 << 25) else v_host[:: P // (1 << 22)]
    c_push = calibrate_c(v_cal, w.send_frac)
    c_fetch = calibrate_c(v_cal, FETCH_FRACTION)
    srv.set_hparams(0.95, 0.95, 1e-4, c_push, 1e-8, w.seed)
    srv.set_fetch_threshold(c_fetch)
    idx = torch.empty(P, dtype=torch.int32, device=device)
    val = torch.empty(P, dtype=torch.float32, device=device)
    cnt = torch.empty(1, dtype=torch.int64, device=device)
    fidx = torch.empty(P, dtype=torch.int32, device=device)
    fval = torch.empty(P, dtype=torch.float32, device=device)
    fcnt = torch.empty(1, dtype=torch.int64, device=device)
    counts = torch.zeros(args.steps, dtype=torch.int64, device=device)
    fcounts = torch.zeros(args.steps, dtype=torch.int64, device=device)
    # Every client keeps its own (stale) copy of the parameters; at large P the
    # clients share at most 32 GB of copies (client c uses copy c mod n_copies),
    # which changes whose copy a scatter writes, not what it costs.
    n_copies = int(min(w.lam, max(1, (32 << 30) // (4 * P))))
    client_theta = torch.from_numpy(th0).to(device).repeat(n_copies, 1)

    # Per-step host values prepared outside the timed loops (the pushes' ints,
    # the count slots, the clients' copies), so the loops only make the calls.
    pushes = [(int(cl[0]), int(js[0]), int(sl[0])) for cl, js, sl in
              (ps.batch(t) for t in range(n_steps))]
    push_slots = [counts[i:i + 1] for i in range(args.steps)]    # the kernels write the counts
    fetch_slots = [fcounts[i:i + 1] for i in range(args.steps)]
    copies = [client_theta[k] for k in range(n_copies)]

    def step(t, ev=None, i=None):
        """One B-FASGD exchange: client c pushes (decision + compaction, sparse
        server apply) and then refreshes its copy (fetch decision + compaction
        of theta, client scatter)."""
        c, j, s = pushes[t]
        n_push = cnt if i is None else push_slots[i]
        n_fetch = fcnt if i is None else fetch_slots[i]
        if ev is not None:
            ev[0].record(stream)
        srv.select_compact(c, slots[s], idx, val, n_push)      # live server v
        if ev is not None:
            ev[1].record(stream)
        srv.push_sparse(c, j, idx, val, n_dev=n_push, n_max=P)
        srv.apply_pending(1)
        if ev is not None:
            ev[2].record(stream)
        srv.fetch_compact(c, fidx, fval, n_fetch)
        if ev is not None:
            ev[3].record(stream)
        fasgd.fetch_apply(copies[c % n_copies], fidx, fval, n_dev=n_fetch, n_max=P,
                          stream=stream)
        if ev is not None:
            ev[4].record(stream)

    for _ in range(args.warmup):
        step(t)
        t += 1
    torch.cuda.synchronize()
    clocks = ClockSampler(gpu_identifier(torch))
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    launches0 = srv.launches
    barrier(world)
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    start.record(stream)
    h0 = time.perf_counter()
    for i in range(args.steps):     # no events inside: they would split the launch chains
        step(t, None, i)
        t += 1
    host_us = (time.perf_counter() - h0) * 1e6 / args.steps   # above ms_per_step: host-bound
    end.record(stream)
    torch.cuda.synchronize()
    clock_info = clocks.stop()
    barrier(world)
    launches = srv.launches - launches0 + args.steps      # + one fetch scatter per step
    total_ms = max_over_ranks(start.elapsed_time(end), world, device)
    # Stage times from a second, instrumented run of the same exchange.
    n_diag = min(args.steps, 100)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(n_diag)]
    for i in range(n_diag):
        step(t, ev[i])
        t += 1
    torch.cuda.synchronize()
    stage = [sum(e[k].elapsed_time(e[k + 1]) for e in ev) / n_diag for k in range(4)]
    sel_ms, app_ms, fsel_ms, fapp_ms = stage
    sent = counts.cpu().numpy().astype(np.float64)
    fetched = fcounts.cpu().numpy().astype(np.float64)
    frac = float(sent.mean() / P)
    srv.sync()
    srv.close()
    step_s = total_ms / 1e3 / args.steps
    peak, peak_kind = peaks()
    alg_apply = 40.0 * sent.mean()                    # state r/w + idx + val per sent entry
    alg_select = 8.0 * P + 8.0 * sent.mean()          # grad + v read, lists written
    dominant = "sparse_apply" if app_ms >= sel_ms else "select_compact"
    a_ms, a_bytes = (app_ms, alg_apply) if dominant == "sparse_apply" else (sel_ms, alg_select)
    achieved = a_bytes / (a_ms / 1e3) / 1e9
    return {
        "value": P * world / step_s, "ms_per_step": total_ms / args.steps,
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(achieved / peak, 4), "peak_source": peak_kind, **nominal(achieved),
                     "kernel": dominant, "bytes_per_launch": a_bytes, "launch_ms": round(a_ms, 5),
                     "traffic": profiled_traffic(w.name, SPARSE_KERNEL_SOURCES),
                     "select_ms": round(sel_ms, 5), "apply_ms": round(app_ms, 5),
                     "select_gbs": round(alg_select / (sel_ms / 1e3) / 1e9, 1),
                     "apply_gbs": round(alg_apply / (app_ms / 1e3) / 1e9, 1),
                     "fetch_select_ms": round(fsel_ms, 5), "fetch_apply_ms": round(fapp_ms, 5)},
        "clocks": clock_info, "e2e": None, "gpu_launches": launches,
        "host_us_per_step": round(host_us, 3),
        "pushes_per_s": world / step_s, "sent_fraction": round(frac, 4),
        "fetched_fraction": round(float(fetched.mean() / P), 4),
        "sent_updates_per_s": sent.mean() * world / step_s,
        "config": {"workload": w.name, "P_per_gpu": P, "P_total": P * world, "lambda": w.lam,
                   "K": 1, "variant": "b-fasgd", "c_push": c_push, "target_send_fraction": w.send_frac,
                   "c_fetch": c_fetch, "target_fetch_fraction": FETCH_FRACTION,
                   "step": "push select/compact + sparse apply + fetch select/compact + client scatter",
                   "client_copies": n_copies,
                   "staleness": w.delay, "parallelism": f"param-shard{world}",
                   "l2": "inputs larger than L2, no flush"},
    }


def run_message(args, w, world, rank, local):
    """The paper's literal B-FASGD exchange per step: a message push (mean-v
    decision, gradient-cache refresh, dense pass over the cache slot) and a
    message fetch (decision, copy of theta to the client's copy)."""
    import torch
    from paper_1601_04033_gb300 import fasgd

    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    P = args.P or w.P
    wr = shard_workload(w, rank)
    R = min(w.R, 8)
    pool = streams.gradient_pool(wr, P, R)
    th0 = streams.theta0(wr, P)
    n_steps = args.warmup + args.steps + w.lam + 100   # + the instrumented stage run
    ps = streams.push_stream(w.replace(R=R), n_steps, 1)
    pool_t, slots = fasgd.aligned_vectors(pool, device)
    stream = torch.cuda.current_stream()
    srv = fasgd.Server(P, w.lam, w.alpha, streams.FASGD, stream=stream, seed=w.seed)
    srv.set_params(torch.from_numpy(th0).to(device))
    t = 0
    for _ in range(w.lam):          # dense warm-up so that v is settled
        cl, js, sl = ps.batch(t)
        srv.push(int(cl[0]), int(js[0]), slots[int(sl[0])])
        srv.apply_pending(1)
        t += 1
    v_now = torch.empty(P, device=device)
    srv.get_state(None, None, None, v_now)
    vbar = float(v_now.double().mean().item())
    c_push = vbar * (1.0 / w.send_frac - 1.0)        # P(send) = vbar / (vbar + c)
    c_fetch = vbar * (1.0 / FETCH_FRACTION - 1.0)
    srv.set_hparams(0.95, 0.95, 1e-4, c_push, 1e-8, w.seed)
    srv.set_fetch_threshold(c_fetch)
    client_theta = torch.empty((w.lam, (P + 3) // 4 * 4), device=device)
    client_theta[:, :P].copy_(torch.from_numpy(th0).to(device))
    sent = torch.zeros(args.steps, dtype=torch.int32, device=device)
    fetched = torch.zeros(args.steps, dtype=torch.int32, device=device)

    def step(t, ev=None, i=None):
        cl, js, sl = ps.batch(t)
        c = int(cl[0])
        if ev is not None:
            ev[0].record(stream)
        srv.push_message(c, int(js[0]), slots[int(sl[0])],
                         sent_dev=sent[i:i + 1] if i is not None else None)
        srv.apply_pending(1)
        if ev is not None:
            ev[1].record(stream)
        srv.fetch_message(c, client_theta[c, :P], fetched_dev=fetched[i:i + 1] if i is not None else None)
        if ev is not None:
            ev[2].record(stream)

    for _ in range(args.warmup):
        step(t)
        t += 1
    torch.cuda.synchronize()
    clocks = ClockSampler(gpu_identifier(torch))
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    launches0 = srv.launches
    barrier(world)
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    start.record(stream)
    h0 = time.perf_counter()
    for i in range(args.steps):     # no events inside: they would split the launch chains
        step(t, None, i)
        t += 1
    host_us = (time.perf_counter() - h0) * 1e6 / args.steps   # above ms_per_step: host-bound
    end.record(stream)
    torch.cuda.synchronize()
    clock_info = clocks.stop()
    barrier(world)
    launches = srv.launches - launches0
    total_ms = max_over_ranks(start.elapsed_time(end), world, device)
    # Push / fetch times from a second, instrumented run of the same exchange.
    n_diag = min(args.steps, 100)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(n_diag)]
    for i in range(n_diag):
        step(t, ev[i])
        t += 1
    torch.cuda.synchronize()
    push_ms = sum(e[0].elapsed_time(e[1]) for e in ev) / n_diag
    fetch_ms = sum(e[1].elapsed_time(e[2]) for e in ev) / n_diag
    s_frac = float(sent.float().mean().item())
    f_frac = float(fetched.float().mean().item())
    srv.sync()
    srv.close()
    step_s = total_ms / 1e3 / args.steps
    peak, peak_kind = peaks()
    # A push: the cache refresh when sent (8 B per parameter) and the dense
    # K = 1 pass over the cache slot (36 B per parameter); the statistic
    # comes from chunk sums the previous pass left (8 B read + 8 B written
    # per 128 parameters), not from a pass over v.
    push_bytes = P * (8 * s_frac + 36) + 16 * ((P + 127) // 128)
    achieved = push_bytes / (push_ms / 1e3) / 1e9
    return {
        "value": P * world / step_s, "ms_per_step": total_ms / args.steps,
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(achieved / peak, 4), "peak_source": peak_kind, **nominal(achieved),
                     "kernel": "message push (decision + cache refresh + dense pass)",
                     "bytes_per_launch": push_bytes, "launch_ms": round(push_ms, 5),
                     "traffic": None, "fetch_ms": round(fetch_ms, 5)},
        "clocks": clock_info, "e2e": None, "gpu_launches": launches,
        "host_us_per_step": round(host_us, 3),
        "pushes_per_s": world / step_s, "sent_fraction": round(s_frac, 4),
        "fetched_fraction": round(f_frac, 4),
        "config": {"workload": w.name, "P_per_gpu": P, "P_total": P * world, "lambda": w.lam,
                   "K": 1, "variant": "b-fasgd per message", "c_push": c_push, "c_fetch": c_fetch,
                   "vbar_after_warmup": vbar, "target_send_fraction": w.send_frac,
                   "target_fetch_fraction": FETCH_FRACTION,
                   "step": "message push (decision, cache refresh, dense pass) + message fetch",
                   "staleness": w.delay, "parallelism": f"param-shard{world}",
                   "l2": "inputs larger than L2, no flush"},
    }


def run_tensor(args, w, world, rank, local):
    """Per-tensor B-FASGD under a bandwidth budget, one exchange per step: a
    budget push (tensor means of v, budget threshold, per-tensor decisions,
    Eq. 4-8 over the transmitted tensors) and a budget fetch (the same
    decision for the client, copy of the transmitted tensors of theta)."""
    import torch
    from paper_1601_04033_gb300 import fasgd

    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    P = args.P or w.P
    wr = shard_workload(w, rank)
    R = min(w.R, 8)
    pool = streams.gradient_pool(wr, P, R)
    th0 = streams.theta0(wr, P)
    sizes = streams.tensor_sizes(w.seed, P, w.tensors)
    n_steps = args.warmup + args.steps + w.lam + 100   # + the instrumented stage run
    ps = streams.push_stream(w.replace(R=R), n_steps, 1)
    pool_t, slots = fasgd.aligned_vectors(pool, device)
    stream = torch.cuda.current_stream()
    srv = fasgd.Server(P, w.lam, w.alpha, streams.FASGD, stream=stream, seed=w.seed)
    srv.set_params(torch.from_numpy(th0).to(device))
    srv.set_tensors(sizes)
    t = 0
    for _ in range(w.lam):          # dense warm-up so that v is settled
        cl, js, sl = ps.batch(t)
        srv.push(int(cl[0]), int(js[0]), slots[int(sl[0])])
        srv.apply_pending(1)
        t += 1
    push_budget = int(w.send_frac * P)
    fetch_budget = int(FETCH_FRACTION * P)
    client_theta = torch.empty((w.lam, (P + 3) // 4 * 4), device=device)
    client_theta[:, :P].copy_(torch.from_numpy(th0).to(device))
    sent = torch.zeros(args.steps, dtype=torch.int64, device=device)
    fetched = torch.zeros(args.steps, dtype=torch.int64, device=device)
    cvals = torch.zeros(args.steps, dtype=torch.float32, device=device)

    def step(t, ev=None, i=None):
        cl, js, sl = ps.batch(t)
        c = int(cl[0])
        if ev is not None:
            ev[0].record(stream)
        srv.push_budget(c, int(js[0]), slots[int(sl[0])], push_budget,
                        c_dev=cvals[i:i + 1] if i is not None else None,
                        count_dev=sent[i:i + 1] if i is not None else None)
        srv.apply_pending(1)
        if ev is not None:
            ev[1].record(stream)
        srv.fetch_budget(c, client_theta[c, :P], fetch_budget,
                         count_dev=fetched[i:i + 1] if i is not None else None)
        if ev is not None:
            ev[2].record(stream)

    for _ in range(args.warmup):
        step(t)
        t += 1
    torch.cuda.synchronize()
    clocks = ClockSampler(gpu_identifier(torch))
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    launches0 = srv.launches
    barrier(world)
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    start.record(stream)
    h0 = time.perf_counter()
    for i in range(args.steps):     # no events inside: they would split the launch chains
        step(t, None, i)
        t += 1
    host_us = (time.perf_counter() - h0) * 1e6 / args.steps   # above ms_per_step: host-bound
    end.record(stream)
    torch.cuda.synchronize()
    clock_info = clocks.stop()
    barrier(world)
    launches = srv.launches - launches0
    total_ms = max_over_ranks(start.elapsed_time(end), world, device)
    # Push / fetch times from a second, instrumented run of the same exchange.
    n_diag = min(args.steps, 100)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(n_diag)]
    for i in range(n_diag):
        step(t, ev[i])
        t += 1
    torch.cuda.synchronize()
    push_ms = sum(e[0].elapsed_time(e[1]) for e in ev) / n_diag
    fetch_ms = sum(e[1].elapsed_time(e[2]) for e in ev) / n_diag
    s_mean = float(sent.double().mean().item())
    f_mean = float(fetched.double().mean().item())
    c_med = float(cvals.median().item())
    srv.sync()
    srv.close()
    step_s = total_ms / 1e3 / args.steps
    peak, peak_kind = peaks()
    # A push: the K = 1 update of every transmitted parameter (theta, n, b, v
    # read and written, gradient read: 36 B); the tensor means come from item
    # sums the previous apply kept current (8 B per item, no pass over v).
    # A fetch: 8 B per fetched parameter.
    push_bytes = 36.0 * s_mean
    fetch_bytes = 8.0 * f_mean
    achieved = push_bytes / (push_ms / 1e3) / 1e9
    return {
        "value": P * world / step_s, "ms_per_step": total_ms / args.steps,
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(achieved / peak, 4), "peak_source": peak_kind, **nominal(achieved),
                     "kernel": "budget push (decision + ranged apply)",
                     "bytes_per_launch": push_bytes, "launch_ms": round(push_ms, 5),
                     "traffic": None, "fetch_ms": round(fetch_ms, 5),
                     "fetch_gbs": round(fetch_bytes / (fetch_ms / 1e3) / 1e9, 1)},
        "clocks": clock_info, "e2e": None, "gpu_launches": launches,
        "host_us_per_step": round(host_us, 3),
        "pushes_per_s": world / step_s, "sent_fraction": round(s_mean / P, 4),
        "fetched_fraction": round(f_mean / P, 4),
        "sent_updates_per_s": s_mean * world / step_s,
        "config": {"workload": w.name, "P_per_gpu": P, "P_total": P * world, "lambda": w.lam,
                   "K": 1, "variant": "b-fasgd per tensor, bandwidth budget",
                   "tensors": int(sizes.size), "push_budget": push_budget,
                   "fetch_budget": fetch_budget, "c_push_median": c_med,
                   "step": "budget push (decision + ranged apply) + budget fetch (decision + copy)",
                   "staleness": w.delay, "parallelism": f"param-shard{world}",
                   "l2": "inputs larger than L2, no flush"},
    }


# ---------------------------------------------------------------------------
def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2500)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="fasgd-25m-k8", choices=sorted(streams.WORKLOADS))
    ap.add_argument("--P", type=int, default=0, help="override the per-GPU parameter count")
    ap.add_argument("--e2e-steps", type=int, default=40)
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-abi-latency", action="store_true",
                    help="small dense workloads: skip the C driver timing")
    ap.add_argument("--variant", choices=sorted(VARIANTS), default="fasgd",
                    help="dense workloads: update rule (ASGD and SASGD move 8 + 4K bytes per "
                         "parameter, the FASGD rules 32 + 4K)")
    ap.add_argument("--exact", action="store_true",
                    help="dense workloads: time the exact-arithmetic FASGD update")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    world, rank, local = dist_env()
    w = streams.WORKLOADS[args.workload]
    if args.workload == "bfasgd-message-25m":
        mode = "message"
    elif w.tensors:
        mode = "tensor"
    elif w.send_frac is not None and w.K == 1:
        mode = "bfasgd"
    else:
        mode = "dense"

    if args.impl == "reference":
        if rank != 0:
            return
        P_s = min(args.P or w.P, 1 << 20)
        var = VARIANTS[args.variant] if mode == "dense" else streams.FASGD
        rate, done, el = oracle_rate(w, P_s, args.steps, None, variant=var, warmup=args.warmup)
        line = {"impl": "reference", "metric": METRIC, "value": rate, "unit": UNIT,
                "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": el * 1e3 / done, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "f32", "data": "synthetic",
                "config": {"workload": w.name, "P_per_gpu": args.P or w.P,
                           "P_total": (args.P or w.P) * args.gpus, "lambda": w.lam, "K": w.K,
                           "variant": args.variant if mode == "dense" else "fasgd",
                           "alpha": w.alpha, "staleness": w.delay,
                           "parallelism": f"param-shard{args.gpus}",
                           "sample": f"first {P_s} parameters, K={w.K} pushes per step",
                           "oracle": "single-threaded C, fp32"},
                "cpu_baseline": {"value": rate, "unit": UNIT, "cores": 1, "kind": "oracle",
                                 "sample": f"{done} steps x K={w.K} pushes over {P_s} parameters"},
                "e2e": {"value": rate, "unit": UNIT, "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return

    import torch
    backend = "nccl" if torch.cuda.is_available() else "gloo"
    init_dist(world, backend)
    if mode == "dense":
        res = run_dense(args, w, world, rank, local)
    elif mode == "message":
        res = run_message(args, w, world, rank, local)
    elif mode == "tensor":
        res = run_tensor(args, w, world, rank, local)
    else:
        res = run_bfasgd(args, w, world, rank, local)

    if rank == 0:
        cpu = None
        if world == 1 and not args.no_cpu_baseline:
            P_s = min(res["config"]["P_per_gpu"], 1 << 22)
            wc = w if mode == "dense" else w.replace(K=1)
            var = VARIANTS[args.variant] if mode == "dense" else streams.FASGD
            rate, done, el = oracle_rate(wc, P_s, None, args.cpu_seconds, variant=var)
            cpu = {"value": rate, "unit": UNIT, "cores": 1, "kind": "oracle",
                   "sample": f"{done} passes of K={wc.K} dense "
                             f"{streams.VARIANT_NAMES[var].upper()} pushes over the first "
                             f"{P_s} parameters ({el:.1f} s)"}
        line = {"metric": METRIC, "value": res["value"], "unit": UNIT, "n_gpus": world,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": res["ms_per_step"],
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "dtype": "f32", "data": "synthetic", "config": res["config"],
                "roofline": physical(res["roofline"]), "cpu_baseline": cpu, "e2e": res["e2e"],
                "clocks": res["clocks"], "gpu_launches": res["gpu_launches"],
                "pushes_per_s": res["pushes_per_s"]}
        for k in ("hbm_gbs_step", "sent_fraction", "fetched_fraction", "sent_updates_per_s",
                  "host_us_per_step", "abi_latency"):
            if k in res:
                line[k] = res[k]
        print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
