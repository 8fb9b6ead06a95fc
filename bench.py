#!/usr/bin/env python3
"""Benchmark of the ADPSGD hot path on GB300: one JSON line on stdout.

A step is one whole ADPSGD run of the vgg16-n8 workload (n = 8 replicas of a VGG-16-sized fp32
vector, P = 138,357,544; 500 iterations; step size 0.05; momentum 0.9, weight decay 5e-4, noise
sigma 0.5; curvatures LogUniform[1e-3, 1], minimisers N(0, 0.1^2); Algorithm 2 with p_init = 4
and K_s = 125): every iteration one fused local-step launch over all replicas, every sync one
launch that fuses that iteration's step with the average + variance, the period rule on the
host.  Inputs are resident in HBM when the timed region starts (x and v are reset to x0 = 0
inside it); x and v (8.9 GB) are far larger than L2, so no flush is needed between steps.
Other workloads: --workload resnet18-n8, resnet50-n16-bf16noise, quadratic-n4-P1M.

value      replica-params/s of the whole run (n * P * iterations / step time), all ranks
e2e        the same through the C ABI with host buffers: H2D of x0, v0, h, c and D2H of the
           final x inside the timed region
roofline   the local-step kernel (the dominant one): algorithmic bytes per launch
           (16 n P + 8 P) over its mean CUDA-event duration (events around every 4th launch in
           the timed region), against the measured HBM copy bandwidth; avg_variance reports
           the averaging kernel the same way (8 n P + 8 P), sync_step the fused sync step
cpu_baseline  the CPU oracle on a bounded sample of the same workload: on every host core
           (the chunked run) and on one core

--impl reference times the CPU oracle itself (the only reference this build has) on every host
core, on bounded samples of the same workload.  Under torchrun (N ranks, one GPU each) the one
problem is split by columns: each rank holds its column range of x, v, h and c, and the ranks
exchange two fp64 partial sums per sync (strong scaling); rank 0 prints the max-over-ranks time.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "avg+variance GB/s vs HBM peak; fused local-step replica-params/sec"
UNIT = "replica-params/s"
DEFAULT_WORKLOAD = "vgg16-n8"
TIMING_PERIOD = 4  # kernel durations from CUDA events around every 4th launch of each kernel
AVG_SAMPLES = 24  # timed standalone averaging launches
# Bounded oracle samples: the workload's first columns, all replicas, a few iterations with a
# sync every 4 (one core: 2^21 columns; every core: 2^24 columns), a few seconds each.
CPU_SAMPLE_ITERS = 24
CPU_SAMPLE_COLUMNS_ONE_CORE = 1 << 21
CPU_SAMPLE_COLUMNS_ALL_CORES = 1 << 24
# The workload whose ncu capture gives DRAM bytes per replica-param for the others.
TRAFFIC_CAPTURE_WORKLOAD = "resnet18-n8"


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


KERNEL_SOURCES = {
    # kernel -> (file, first line marker, end marker) of the source it is built from
    "local_step_kernel": [("kernels.cu", "struct StepParams", "// Averaging + variance"), ("noise.cuh", "", ""),
                          ("common.cuh", "", "")],
    "average_kernel": [("kernels.cu", "// Averaging + variance", "__global__ void __launch_bounds__(kThreads) philox_fill"),
                       ("average.cuh", "", ""), ("common.cuh", "", "")],
    "sync_step_kernel": [("sync_step.cu", "struct SyncStepParams", "using SyncStepKernel"), ("average.cuh", "", ""),
                         ("noise.cuh", "", ""), ("common.cuh", "", "")],
}


def kernel_source_digest(kernel: str) -> str:
    """sha256 (16 hex) of the code a kernel is compiled from, without comments and whitespace
    (a comment edit does not invalidate a capture)."""
    import hashlib
    import re
    h = hashlib.sha256()
    for fname, begin, end in KERNEL_SOURCES[kernel]:
        text = open(os.path.join(ROOT, "paper_2007_06134_gb300", "csrc", fname)).read()
        a = text.index(begin) if begin else 0
        b = text.index(end, a) if end else len(text)
        code = re.sub(r"/\*.*?\*/", " ", text[a:b], flags=re.S)
        code = re.sub(r"//[^\n]*", " ", code)
        h.update(" ".join(code.split()).encode())
    return h.hexdigest()[:16]


def recorded_traffic(kernel: str, workload: str, algorithmic_bytes: int):
    """DRAM bytes per launch from a committed ncu capture, if the kernel source is unchanged since:
    (bytes, how).  A workload without its own capture takes the capture of
    TRAFFIC_CAPTURE_WORKLOAD scaled by the ratio of algorithmic bytes per launch (the kernels
    stream their arrays once, so traffic grows in proportion to the replica-params processed)."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None, None
    with open(path) as f:
        d = json.load(f)
    rows = d.get(kernel, {})
    e = rows.get(workload)
    how = "ncu capture of this workload"
    scale = 1.0
    if e is None and TRAFFIC_CAPTURE_WORKLOAD in rows:
        e = rows[TRAFFIC_CAPTURE_WORKLOAD]
        scale = algorithmic_bytes / e["algorithmic_bytes_per_launch"]
        how = f"ncu capture of {TRAFFIC_CAPTURE_WORKLOAD} scaled by algorithmic bytes ({scale:.4f})"
    if not e or e.get("source_sha256_16") != kernel_source_digest(kernel):
        return None, None
    return int(round(e["dram_bytes_per_launch"] * scale)), how


# ------------------------------------------------------------------------------------------
# clocks during the timed region
# ------------------------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu_id = gpu_id
        self.proc = None
        self.path = os.path.join("/tmp", f"adpsgd_clocks_{os.getpid()}.csv")

    def __enter__(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu_id}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"], stdout=self.f,
                                         stderr=subprocess.DEVNULL)
        except Exception as e:  # nvidia-smi missing: report no clock data
            log("clock sampling unavailable:", e)
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.f.close()

    def summary(self):
        if self.proc is None or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm, smax, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 8:
                    continue
                try:
                    sm.append(float(parts[0]))
                    smax.append(float(parts[1]))
                except ValueError:
                    continue
                for nm, val in zip(names, parts[4:8]):
                    if val.lower().startswith("active"):
                        reasons.add(nm)
        os.remove(self.path)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------------------------------------
# distributed plumbing (barrier, max over ranks; the per-sync exchange is shard.dist_gather)
# ------------------------------------------------------------------------------------------

def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    pg = None
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if args.impl == "gb300" else "gloo"
        if backend == "nccl":
            import torch
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
        pg = dist
    return world, rank, local, pg


def max_over_ranks(pg, value: float, device=None) -> float:
    if pg is None:
        return value
    import torch
    t = torch.tensor([value], dtype=torch.float64, device=device)
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return float(t.item())


def barrier(pg, device=None):
    if pg is not None:
        if device is not None:
            pg.barrier(device_ids=[device.index])
        else:
            pg.barrier()


# ------------------------------------------------------------------------------------------
# CPU oracle leg
# ------------------------------------------------------------------------------------------

def cpu_model() -> str:
    """The host CPU's model name (x86: /proc/cpuinfo; Arm: lscpu), or the machine type."""
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith("model name"):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    import platform
    return platform.machine()


def oracle_sample(w, seed_offset=0, threads=None):
    """Time the oracle on a bounded sample: CPU_SAMPLE_ITERS iterations of the workload's local step
    and its syncs (constant period 4) on its first columns, all replicas.  threads=None: the
    single-thread run on CPU_SAMPLE_COLUMNS_ONE_CORE columns; threads=t: the chunked run on t host
    threads on CPU_SAMPLE_COLUMNS_ALL_CORES columns.  Returns (replica-params/s, seconds, text)."""
    from oracle import oracle as O
    from paper_2007_06134_gb300 import inputs
    P = min(CPU_SAMPLE_COLUMNS_ONE_CORE if threads is None else CPU_SAMPLE_COLUMNS_ALL_CORES, w.P)
    h, c = inputs.problem(w, P)
    x, v = inputs.zero_state(w.n, P)
    noise = O.noise_bf16(w.seed, w.n, P) if w.noise == "bf16" else None
    spec = O.ScheduleSpec(kind=0, K=CPU_SAMPLE_ITERS, p_init=4, lr0=w.lr0, lr_factor=w.lr_factor,
                          milestones=w.milestones)
    O.build()
    t0 = time.perf_counter()
    O.run(x, v, h, c, spec=spec, seed=w.seed + seed_offset, mu=w.mu, wd=w.wd, sigma=w.sigma, noise=noise,
          threads=threads)
    dt = time.perf_counter() - t0
    rp = w.n * P * CPU_SAMPLE_ITERS
    how = "one core" if threads is None else f"{threads} host threads (chunked run)"
    return rp / dt, dt, (f"{CPU_SAMPLE_ITERS} iterations (syncs every 4) of {w.name} on its first {P} columns, "
                         f"all {w.n} replicas, {how}: {rp} replica-param updates in {dt:.2f} s")


def cpu_baseline(w):
    """The oracle on every host core (the reported figure) and on one core."""
    from oracle import oracle as O
    threads = O.host_threads()
    r_all, _, sample_all = oracle_sample(w, threads=threads)
    r_one, _, sample_one = oracle_sample(w)
    return {"value": r_all, "unit": UNIT, "cores": threads, "kind": "oracle", "sample": sample_all,
            "cpu_model": cpu_model(),
            "single_core": {"value": r_one, "unit": UNIT, "cores": 1, "sample": sample_one}}


def run_reference(args, w):
    world, rank, local, pg = dist_setup(args)
    if rank != 0:
        return 0
    from oracle import oracle as O
    threads = O.host_threads()
    for _ in range(args.warmup):
        oracle_sample(w, threads=threads)
    rates, times, sample = [], [], ""
    for s in range(args.steps):
        r, dt, sample = oracle_sample(w, s + 1, threads=threads)
        rates.append(r)
        times.append(dt)
    value = float(np.mean(rates))
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * float(np.mean(times)),
        "higher_is_better": True, "scaling": "strong", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": w.name, "n": w.n, "P": w.P, "K": w.K,
                   "sample_columns": min(CPU_SAMPLE_COLUMNS_ALL_CORES, w.P), "sample_iterations": CPU_SAMPLE_ITERS},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle", "sample": sample,
                         "cpu_model": cpu_model()},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------------------------------
# GPU leg
# ------------------------------------------------------------------------------------------

def schedule_for(abi, w):
    return abi.make_schedule(abi.ADPSGD, w.K, w.p_init, K_s=w.K_s, lr0=w.lr0, lr_factor=w.lr_factor,
                             milestones=w.milestones)


def run_gpu(args, w):
    import torch

    from paper_2007_06134_gb300 import abi, inputs, shard

    world, rank, local, pg = dist_setup(args)
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    stream = torch.cuda.current_stream(device)
    abi.load()
    seed = w.seed

    # One problem; with N ranks each rank holds a contiguous column range of it (strong scaling).
    n, P_total = w.n, w.P
    col0, P = shard.column_split(P_total, world, rank)
    gather = shard.dist_gather()[0] if world > 1 else None
    h_all, c_all = inputs.problem(w)
    h, c = np.ascontiguousarray(h_all[col0:col0 + P]), np.ascontiguousarray(c_all[col0:col0 + P])
    del h_all, c_all
    hd = torch.from_numpy(h).to(device)
    cd = torch.from_numpy(c).to(device)
    xd = torch.zeros((n, P), dtype=torch.float32, device=device)
    vd = torch.zeros_like(xd)
    noise = None
    if w.noise == "bf16":
        noise = torch.empty((n, P), dtype=torch.int16, device=device)
        abi.adpsgd_noise_fill_bf16_part(w.seed, n, P, 0, col0, noise, stream)
    fuse_sync = not args.no_sync_fusion
    noise_mode = abi.NOISE_BF16 if noise is not None else abi.NOISE_PHILOX

    def context(exchange=True, **kw):
        cfg = abi.make_config(n, P, momentum=w.mu, weight_decay=w.wd, noise_sigma=w.sigma, seed=seed,
                              noise_mode=noise_mode, want_loss=True, **kw)
        ctx = abi.adpsgd_init(cfg, xd, vd, hd, cd, noise, stream)
        if world > 1 and exchange:
            abi.adpsgd_set_shard(ctx, abi.make_shard(world, rank, col0, P_total, gather))
        return ctx

    sched = schedule_for(abi, w)
    ctx = context(time_kernels=TIMING_PERIOD, fuse_sync_step=fuse_sync)
    w0d = torch.zeros(P, dtype=torch.float32, device=device)  # x_0 = 0, the initial model on the device

    def one_run():
        # Algorithm 2 from the start: every replica set to w0 and the momentum zeroed by the
        # library (one broadcast kernel and a memset), then the whole run.
        abi.adpsgd_init_replicas(ctx, w0d)
        st = abi.adpsgd_state_init(sched)
        return abi.adpsgd_run(ctx, sched, st)

    for _ in range(args.warmup):
        stats = one_run()
    abi.adpsgd_reset_kernel_times(ctx)
    torch.cuda.synchronize(device)

    gpu_id = str(local)
    try:
        gpu_id = str(torch.cuda.get_device_properties(device).uuid)
        if not gpu_id.startswith("GPU-"):
            gpu_id = "GPU-" + gpu_id
    except Exception:
        pass
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    rounds, launches = [], 0
    with ClockSampler(gpu_id) as clocks:
        barrier(pg, device)
        torch.cuda.synchronize(device)
        ev0.record(stream)
        for _ in range(args.steps):
            stats = one_run()
            rounds.append(stats.rounds)
            # the broadcast kernel of the initialisation, then the run's kernels
            launches += 1 + stats.local_step_launches + stats.average_launches + stats.sync_step_launches
        ev1.record(stream)
        torch.cuda.synchronize(device)
        barrier(pg, device)
    ms_total = ev0.elapsed_time(ev1)
    ms_total = max_over_ranks(pg, ms_total, device)
    ms_step = ms_total / args.steps
    rp_per_step = n * P_total * w.K  # the whole problem, all ranks together
    value = rp_per_step / (ms_step / 1000.0)
    launches = int(max_over_ranks(pg, float(launches), device)) * world

    kt = abi.adpsgd_kernel_times(ctx)
    kt = dict(kt)
    peak, peak_kind = measured_peaks()
    k1_bytes = 16 * n * P + 8 * P + (2 * n * P if noise is not None else 0)
    k1_ms = kt["local_step_ms"] / max(1, kt["local_step_launches"])
    k1_gbs = k1_bytes / (k1_ms / 1000.0) / 1e9
    # The fused sync step moves the local step's bytes: the averaging adds none.
    ks_ms = kt["sync_step_ms"] / kt["sync_step_launches"] if kt["sync_step_launches"] else None
    ks_gbs = k1_bytes / (ks_ms / 1000.0) / 1e9 if ks_ms else None
    clock_summary = clocks.summary()

    # The averaging kernel on its own, as the unfused path runs it: one launch after each local
    # step, every launch timed (with fused sync steps the run above launches few of them).  Only
    # the kernel is timed here, so this context does not exchange its sums.
    k2_bytes = 8 * n * P + 8 * P
    with context(exchange=False, time_kernels=1) as ctx_k2:
        for r in range(AVG_SAMPLES + 2):
            if r == 2:
                abi.adpsgd_reset_kernel_times(ctx_k2)
            abi.adpsgd_local_steps(ctx_k2, r, [w.lr0])
            abi.adpsgd_average_and_variance(ctx_k2)
        kt2 = dict(abi.adpsgd_kernel_times(ctx_k2))
    k2_ms = kt2["average_ms"] / max(1, kt2["average_launches"])
    k2_gbs = k2_bytes / (k2_ms / 1000.0) / 1e9

    # End to end through the C ABI from pinned host buffers: the run's inputs as Algorithms 1 and
    # 2 define them (one initial model w0 for every replica, momentum zero; h and c) in, the whole
    # run, and its result out: the averaged model (one row) when the run ends with a sync, when
    # every replica holds it, else every replica's row.
    e2e_value, h2d, d2h, e2e_phases = None, 0, 0, None
    if not args.no_e2e:
        w0h = torch.zeros(P, dtype=torch.float32).pin_memory()  # x_0 = 0, this rank's columns
        hh = torch.from_numpy(h).pin_memory()
        ch = torch.from_numpy(c).pin_memory()
        xout = torch.empty((n, P), dtype=torch.float32).pin_memory()
        ctx_e2e = context(fuse_sync_step=fuse_sync)  # set-up, outside the timed region
        trace_e2e = abi.TraceBuffers(w.K + 1)
        out_rows = [n]

        marks = [torch.cuda.Event(enable_timing=True) for _ in range(4)]

        def e2e_step():
            marks[0].record(stream)
            abi.adpsgd_init_replicas(ctx_e2e, w0h)
            abi.adpsgd_copy_h2d(hd, hh, stream=stream)
            abi.adpsgd_copy_h2d(cd, ch, stream=stream)
            marks[1].record(stream)
            abi.adpsgd_run(ctx_e2e, sched, abi.adpsgd_state_init(sched), trace=trace_e2e)
            marks[2].record(stream)
            ended_with_sync = trace_e2e.len > 0 and int(trace_e2e.k[trace_e2e.len - 1]) == w.K - 1
            out_rows[0] = 1 if ended_with_sync else n
            abi.adpsgd_copy_d2h(xout, xd, 4 * out_rows[0] * P, stream=stream)
            marks[3].record(stream)

        e2e_step()
        torch.cuda.synchronize(device)
        barrier(pg, device)
        t0 = time.perf_counter()
        e2e_steps = max(1, min(args.steps, 3))
        for _ in range(e2e_steps):
            e2e_step()
        torch.cuda.synchronize(device)
        log("e2e last step: h2d %.1f ms, run %.1f ms, d2h %.1f ms" % (
            marks[0].elapsed_time(marks[1]), marks[1].elapsed_time(marks[2]), marks[2].elapsed_time(marks[3])))
        dt = max_over_ranks(pg, (time.perf_counter() - t0) / e2e_steps, device)
        e2e_value = rp_per_step / dt
        h2d = 4 * 3 * P_total  # all ranks together: w0, h and c
        d2h = 4 * out_rows[0] * P_total
        e2e_phases = {"h2d_ms": marks[0].elapsed_time(marks[1]), "run_ms": marks[1].elapsed_time(marks[2]),
                      "d2h_ms": marks[2].elapsed_time(marks[3]), "wall_ms": dt * 1000.0}
        ctx_e2e.close()

    # The same run with each sync interval fused into one kernel (separable objective only).
    fused = None
    if not args.no_fused and n <= 32:
        with context(time_kernels=TIMING_PERIOD, fuse_intervals=True) as ctx_f:
            def fused_run():
                abi.adpsgd_init_replicas(ctx_f, w0d)
                return abi.adpsgd_run(ctx_f, sched, abi.adpsgd_state_init(sched))
            fused_run()
            abi.adpsgd_reset_kernel_times(ctx_f)
            torch.cuda.synchronize(device)
            barrier(pg, device)
            ev0.record(stream)
            for _ in range(args.steps):
                fstats = fused_run()
            ev1.record(stream)
            torch.cuda.synchronize(device)
            fms = max_over_ranks(pg, ev0.elapsed_time(ev1), device) / args.steps
            ft = abi.adpsgd_kernel_times(ctx_f)
        fused = {"value": rp_per_step / (fms / 1000.0), "unit": UNIT, "ms_per_step": fms,
                 "interval_launches_per_step": fstats.interval_launches,
                 "interval_ms_per_launch": ft["interval_ms"] / max(1, ft["interval_launches"]),
                 "note": "each sync interval (local steps + averaging) as one kernel; valid for the "
                         "separable surrogate objective only, not for a real model"}

    # The paper's comparison for this workload: ADPSGD against CPSGD at the same number of averaging
    # rounds (p = round(K / R)), and full-communication SGD (one allreduce per iteration), as rounds,
    # equivalent period, final loss and the bytes a ring allreduce would move per node.
    comparison = None
    if not args.no_compare:
        tr_a = abi.TraceBuffers(w.K + 1)
        abi.adpsgd_init_replicas(ctx, w0d)
        sa = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr_a)
        ta = tr_a.arrays()
        p_eq = max(1, round(w.K / max(1, sa.rounds)))
        rows = {"adpsgd": (sched, sa, ta)}
        for label, p_c in (("cpsgd_equal_budget", p_eq), ("cpsgd_p%d" % w.cpsgd_p, w.cpsgd_p)):
            if label in rows or (label != "cpsgd_equal_budget" and p_c == p_eq):
                continue
            sc = abi.make_schedule(abi.CPSGD, w.K, p_c, lr0=w.lr0, lr_factor=w.lr_factor, milestones=w.milestones)
            tr_c = abi.TraceBuffers(w.K + 1)
            abi.adpsgd_init_replicas(ctx, w0d)
            st_c = abi.adpsgd_run(ctx, sc, abi.adpsgd_state_init(sc), trace=tr_c)
            rows[label] = (sc, st_c, tr_c.arrays())
        comparison = {}
        for label, (sc, stt, tt) in rows.items():
            comparison[label] = {"p": int(sc.p_init), "rounds": int(stt.rounds), "equiv_period": stt.equiv_period,
                                 "k_last_sync": int(tt["k"][-1]) if len(tt["k"]) else None,
                                 "loss_at_last_sync": float(tt["loss"][-1]) if len(tt["loss"]) else None,
                                 "S_at_last_sync": float(tt["S"][-1]) if len(tt["S"]) else None,
                                 "wire_bytes_per_node": stt.wire_bytes_per_node,
                                 "wire_bytes_total": stt.wire_bytes_total}
        full_pn, full_tot = abi.adpsgd_wire_bytes(n, P_total, w.K, False)
        comparison["fullsgd"] = {"p": 1, "rounds": w.K, "wire_bytes_per_node": full_pn, "wire_bytes_total": full_tot}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        cpu = cpu_baseline(w)
    ctx.close()
    k1_traffic, k1_traffic_how = recorded_traffic("local_step_kernel", w.name, k1_bytes)
    k2_traffic, k2_traffic_how = recorded_traffic("average_kernel", w.name, k2_bytes)
    ks_traffic, ks_traffic_how = recorded_traffic("sync_step_kernel", w.name, k1_bytes)

    if rank == 0:
        parallelism = "one GPU" if world == 1 else (
            f"columns split over {world} ranks (rank 0 holds {P} of {P_total}); 16 bytes exchanged per sync")
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "strong",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": w.name, "n": n, "P": P_total, "K": w.K,
                       "schedule": f"ADPSGD p_init={w.p_init} K_s={w.K_s}",
                       "rounds_per_step": rounds[-1] if rounds else None,
                       "l2": "inputs larger than L2 (x, v = %.0f MB per rank)" % (8 * n * P / 1e6),
                       "parallelism": parallelism},
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "copies": "in: the initial model w0 [P] (adpsgd_init_replicas: every replica set to it on "
                              "the device, momentum zeroed), h and c; out: the averaged model [P] when the run "
                              "ends with a sync, else every replica's row",
                    "last_step": e2e_phases},
            "gpu_launches": launches,
            "roofline": {"kernel": "local_step_kernel", "bound": "hbm", "achieved": k1_gbs, "peak": peak,
                         "peak_kind": peak_kind, "unit": "GB/s", "frac": k1_gbs / peak,
                         "bytes_per_launch": k1_bytes, "ms_per_launch": k1_ms,
                         "traffic": k1_traffic, "traffic_source": k1_traffic_how},
            "avg_variance": {"kernel": "average_kernel", "bound": "hbm", "achieved": k2_gbs,
                             "peak": peak, "unit": "GB/s", "frac": k2_gbs / peak, "bytes_per_launch": k2_bytes,
                             "ms_per_launch": k2_ms, "launches": kt2["average_launches"],
                             "timed": "alone, each launch right after a local step",
                             "traffic": k2_traffic, "traffic_source": k2_traffic_how},
            "sync_step": None if ks_ms is None else {
                "kernel": "sync_step_kernel", "bound": "hbm", "achieved": ks_gbs, "peak": peak, "unit": "GB/s",
                "frac": ks_gbs / peak, "bytes_per_launch": k1_bytes, "ms_per_launch": ks_ms,
                "launches": kt["sync_step_launches"], "average_launches_in_run": kt["average_launches"],
                "traffic": ks_traffic, "traffic_source": ks_traffic_how,
                "note": "the local step of each sync iteration fused with its averaging (x not written "
                        "and read back in between); 16 n P + 8 P bytes, the local step's"},
            "local_step_rp_per_s": n * P / (k1_ms / 1000.0),
            "fused_intervals": fused,
            "comparison": comparison,
            "clocks": clock_summary,
            "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)
    if pg is not None:
        pg.destroy_process_group()
    return 0


def run_sweep(args):
    """Averaging + variance alone over n x P (the sweep workload): GB/s and fraction of peak per point.
    Every launch starts from distinct replicas (restored from a copy, then the L2 flushed): the
    averaging leaves identical replicas behind, which is not the state a sync finds."""
    import torch

    from paper_2007_06134_gb300 import abi, inputs
    peak, peak_kind = measured_peaks()
    device = torch.device("cuda", 0)
    stream = torch.cuda.current_stream(device)
    l2 = torch.cuda.get_device_properties(device).L2_cache_size
    flush = torch.empty(int(2 * l2) // 4, dtype=torch.float32, device=device)

    def flush_l2():
        # Write a buffer twice the L2, then read it: the timed launch finds neither its own data
        # nor dirty lines in L2 (a write-only flush leaves up to one L2 of dirty lines, whose
        # write-back would then compete with the timed kernel's traffic).
        flush.zero_()
        flush.sum()

    for n in inputs.SWEEP_N:
        for lp in inputs.SWEEP_LOG2P:
            P = 1 << lp
            if 8 * n * P > args.sweep_max_bytes:
                continue
            x0 = torch.randn((n, P), dtype=torch.float32, device=device)
            x0 += torch.arange(n, device=device, dtype=torch.float32)[:, None] * 1e-3
            xd = torch.empty_like(x0)
            z = torch.zeros(P, device=device)
            cfg = abi.make_config(n, P, want_loss=False, time_kernels=True)
            with abi.adpsgd_init(cfg, xd, xd, z, z, None, stream) as ctx:
                reps = max(5, min(50, int(2e10 // (8 * n * P))))
                for _ in range(3):
                    xd.copy_(x0)
                    abi.adpsgd_average_and_variance(ctx, want_loss=False)
                abi.adpsgd_reset_kernel_times(ctx)
                for _ in range(reps):
                    xd.copy_(x0)
                    flush_l2()
                    abi.adpsgd_average_and_variance(ctx, want_loss=False)
                t = abi.adpsgd_kernel_times(ctx)
            ms = t["average_ms"] / t["average_launches"]
            gbs = 8 * n * P / (ms / 1e3) / 1e9
            print(json.dumps({"sweep": "average_and_variance", "n": n, "P": P, "ms": ms, "GB/s": gbs,
                              "frac": gbs / peak, "peak": peak, "peak_kind": peak_kind,
                              "l2_flushed": "write then read a 2 x L2 buffer",
                              "replicas": "distinct at every launch"}), flush=True)
            del xd, x0


def run_local_sweep(args):
    """The local step alone over n x P (Philox noise, weight decay): each point times 20 launches
    with CUDA events, every launch after a write-then-read L2 flush; GB/s on 16 n P + 8 P bytes."""
    import torch

    from paper_2007_06134_gb300 import abi, inputs
    peak, peak_kind = measured_peaks()
    device = torch.device("cuda", 0)
    stream = torch.cuda.current_stream(device)
    l2 = torch.cuda.get_device_properties(device).L2_cache_size
    flush = torch.empty(int(2 * l2) // 4, dtype=torch.float32, device=device)
    w = inputs.WORKLOADS["resnet18-n8"]
    for n in (2, 4, 8, 16, 32):
        for lp in (20, 22, 24, 26, 28):
            P = 1 << lp
            if (16 * n + 8) * P > args.sweep_max_bytes:
                continue
            h, c = inputs.problem(w, P)
            hd, cd = torch.from_numpy(h).to(device), torch.from_numpy(c).to(device)
            xd = torch.zeros((n, P), dtype=torch.float32, device=device)
            vd = torch.zeros_like(xd)
            cfg = abi.make_config(n, P, momentum=w.mu, weight_decay=w.wd, noise_sigma=w.sigma, seed=w.seed,
                                  time_kernels=1)
            with abi.adpsgd_init(cfg, xd, vd, hd, cd, None, stream) as ctx:
                abi.adpsgd_local_steps(ctx, 0, [w.lr0] * 3)
                abi.adpsgd_reset_kernel_times(ctx)
                for k in range(20):
                    flush.zero_()
                    flush.sum()
                    abi.adpsgd_local_steps(ctx, 3 + k, [w.lr0])
                t = abi.adpsgd_kernel_times(ctx)
            ms = t["local_step_ms"] / t["local_step_launches"]
            gbs = (16 * n + 8) * P / (ms / 1e3) / 1e9
            print(json.dumps({"sweep": "local_step", "n": n, "P": P, "ms": ms, "GB/s": gbs, "frac": gbs / peak,
                              "peak": peak, "peak_kind": peak_kind, "l2_flushed": "write then read a 2 x L2 buffer",
                              "replica_params_per_s": n * P / (ms / 1e3)}), flush=True)
            del xd, vd, hd, cd


def run_sync_sweep(args):
    """The fused sync step against the local step and the averaging it replaces, over n x P: a
    CPSGD p = 2 run (every other iteration ends with a sync) with every launch timed, once with
    fused sync steps and once with separate kernels.  Per point: each kernel's time, GB/s on its
    algorithmic bytes, and the time saved per sync."""
    import torch

    from paper_2007_06134_gb300 import abi, inputs
    peak, peak_kind = measured_peaks()
    device = torch.device("cuda", 0)
    stream = torch.cuda.current_stream(device)
    w = inputs.WORKLOADS["resnet18-n8"]
    # the fused step's forms: registers up to 8 replicas, two halves for 9..16 with Philox noise,
    # the 16-replica register form with the bf16 noise tensor
    for n, bf16 in ((2, False), (4, False), (6, False), (8, False), (12, False), (16, False), (8, True), (16, True)):
        for lp in (22, 24, 26):
            P = 1 << lp
            h, c = inputs.problem(w, P)
            hd, cd = torch.from_numpy(h).to(device), torch.from_numpy(c).to(device)
            xd = torch.zeros((n, P), dtype=torch.float32, device=device)
            vd = torch.zeros_like(xd)
            noise = None
            if bf16:
                noise = torch.empty((n, P), dtype=torch.int16, device=device)
                abi.adpsgd_noise_fill_bf16(w.seed, n, P, noise, stream)
            sched = abi.make_schedule(abi.CPSGD, 40, 2, lr0=w.lr0)
            times = {}
            for fused in (True, False):
                cfg = abi.make_config(n, P, momentum=w.mu, weight_decay=w.wd, noise_sigma=w.sigma, seed=w.seed,
                                      noise_mode=abi.NOISE_BF16 if bf16 else abi.NOISE_PHILOX,
                                      time_kernels=1, fuse_sync_step=fused)
                with abi.adpsgd_init(cfg, xd, vd, hd, cd, noise, stream) as ctx:
                    abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched))
                    abi.adpsgd_reset_kernel_times(ctx)
                    abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched))
                    t = abi.adpsgd_kernel_times(ctx)
                if fused:
                    times["sync_step"] = t["sync_step_ms"] / t["sync_step_launches"]
                else:
                    times["local_step"] = t["local_step_ms"] / t["local_step_launches"]
                    times["average"] = t["average_ms"] / t["average_launches"]
            step_bytes = 16 * n * P + 8 * P + (2 * n * P if bf16 else 0)
            avg_bytes = 8 * n * P + 8 * P
            line = {"sweep": "sync_step", "n": n, "P": P, "noise": "bf16" if bf16 else "philox",
                    "peak": peak, "peak_kind": peak_kind,
                    "sync_step_ms": times["sync_step"],
                    "sync_step_frac": step_bytes / (times["sync_step"] / 1e3) / 1e9 / peak,
                    "local_step_ms": times["local_step"],
                    "local_step_frac": step_bytes / (times["local_step"] / 1e3) / 1e9 / peak,
                    "average_ms": times["average"],
                    "average_frac": avg_bytes / (times["average"] / 1e3) / 1e9 / peak,
                    "saved_ms_per_sync": times["local_step"] + times["average"] - times["sync_step"],
                    "l2": "x, v = %.0f MB" % (8 * n * P / 1e6)}
            print(json.dumps(line), flush=True)
            del xd, vd, noise


def run_variance_traces(args):
    """The schedule study of Sec. III on the strategies-n16 surrogate: constant periods, the four
    strategies' piecewise periods, the decreasing period of Sec. V-B and Algorithm 2, each a whole
    run with Var[W_k] recorded every iteration.  One JSON line per schedule: syncs, the weighted
    variance of Eq. metric2, the mean variance per step-size phase, the loss, and the period."""
    import torch

    from paper_2007_06134_gb300 import abi, diagnostics, inputs
    w = inputs.WORKLOADS["strategies-n16"]
    n, P, K = w.n, w.P, w.K
    device = torch.device("cuda", 0)
    stream = torch.cuda.current_stream(device)
    h, c = inputs.problem(w)
    hd, cd = torch.from_numpy(h).to(device), torch.from_numpy(c).to(device)
    xd = torch.zeros((n, P), dtype=torch.float32, device=device)
    vd = torch.zeros_like(xd)
    kw = dict(lr0=w.lr0, lr_factor=w.lr_factor, milestones=w.milestones)
    half = K // 2
    schedules = [
        ("FULLSGD (p=1)", abi.make_schedule(abi.CPSGD, K, 1, **kw)),
        ("CPSGD p=2", abi.make_schedule(abi.CPSGD, K, 2, **kw)),
        ("CPSGD p=4", abi.make_schedule(abi.CPSGD, K, 4, **kw)),
        ("CPSGD p=5 (strategy 4)", abi.make_schedule(abi.CPSGD, K, 5, **kw)),
        ("CPSGD p=8 (strategy 3)", abi.make_schedule(abi.CPSGD, K, 8, **kw)),
        ("strategy 1: p=4 then 8", abi.make_schedule(abi.PIECEWISE, K, 4, period_changes=((half, 8),), **kw)),
        ("strategy 2: p=8 then 4", abi.make_schedule(abi.PIECEWISE, K, 8, period_changes=((half, 4),), **kw)),
        ("decreasing: p=20 then 5", abi.make_schedule(abi.PIECEWISE, K, 20, period_changes=((half, 5),), **kw)),
        ("ADPSGD p_init=4 K_s=1000 K_w=25", abi.make_schedule(abi.ADPSGD, K, 4, K_s=1000, K_w=25, **kw)),
    ]
    gammas = [abi.adpsgd_gamma(schedules[0][1], k) for k in range(K)]
    edges = [0] + list(w.milestones) + [K]
    cfg = abi.make_config(n, P, momentum=w.mu, weight_decay=w.wd, noise_sigma=w.sigma, seed=w.seed, want_loss=True)
    with abi.adpsgd_init(cfg, xd, vd, hd, cd, None, stream) as ctx:
        for name, sched in schedules:
            xd.zero_()
            vd.zero_()
            tr = abi.TraceBuffers(K + 1, var_cap=K)
            t0 = time.perf_counter()
            stats = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=tr)
            dt = time.perf_counter() - t0
            t = tr.arrays()
            line = {"variance_traces": w.name, "schedule": name, "syncs": int(stats.rounds),
                    "equiv_period": K / stats.rounds,
                    "weighted_variance_eq_metric2": diagnostics.weighted_variance(t["var"], gammas),
                    "mean_variance_per_lr_phase": diagnostics.phase_means(t["var"], edges),
                    "mean_V_t": float(np.mean(diagnostics.interval_means(t["var"], t["k"]))),
                    "final_loss": float(t["loss"][-1]), "min_loss": float(np.min(t["loss"])),
                    "wire_bytes_per_node": stats.wire_bytes_per_node, "seconds": dt}
            if sched.kind == abi.ADPSGD:
                pk = {}
                for q in (999, 1999, 2999, K - 1):
                    idx = int(np.searchsorted(t["k"], q, side="right")) - 1
                    pk[str(q + 1)] = int(t["p"][max(idx, 0)])
                line["period_at_iteration"] = pk
                line["C2"] = float(t["C2"][-1])
            print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["gb300", "reference"], default="gb300")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--iters", type=int, default=None,
                    help="override the workload's iteration count (profiling captures only)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--no-fused", action="store_true", help="skip the fused-interval measurement")
    ap.add_argument("--no-sync-fusion", action="store_true",
                    help="run each sync iteration's local step and averaging as two kernels")
    ap.add_argument("--no-compare", action="store_true", help="skip the ADPSGD / CPSGD / FULLSGD comparison runs")
    ap.add_argument("--sweep", action="store_true", help="averaging-kernel sweep over n x P instead")
    ap.add_argument("--sync-sweep", action="store_true",
                    help="fused sync step against the local step + averaging over n x P instead")
    ap.add_argument("--local-sweep", action="store_true", help="the local step alone over n x P instead")
    ap.add_argument("--sweep-max-bytes", type=float, default=70e9)
    ap.add_argument("--variance-traces", action="store_true",
                    help="the schedule study of Sec. III with per-iteration variance instead")
    args = ap.parse_args()
    from paper_2007_06134_gb300 import inputs
    w = inputs.WORKLOADS[args.workload]
    if args.iters is not None:
        import dataclasses
        w = dataclasses.replace(w, K=args.iters, K_s_frac=min(w.K_s_frac, 0.5),
                                milestones=tuple(int(m * args.iters / w.K) for m in w.milestones))
    if args.impl == "reference":
        return run_reference(args, w)
    if args.sweep:
        return run_sweep(args)
    if args.sync_sweep:
        return run_sync_sweep(args)
    if args.local_sweep:
        return run_local_sweep(args)
    if args.variance_traces:
        return run_variance_traces(args)
    return run_gpu(args, w)


if __name__ == "__main__":
    sys.exit(main())
