#!/usr/bin/env python
"""Planner benchmark: PrefixPlace's coordinate-refined plan on one GB300.

One step = one whole plan (pp_plan_run: standalone-score orders, WorkerGreedy
pass, up to R refinement sweeps over S starts, objective + argmax) of the
headline workload, the paper-scale synthetic instance (n = 50,000 chunks,
W = 16 workers, k = 4,096 slots, 16 starts, 6 rounds), inputs resident in HBM.

  value     Eq. 9 cell updates executed (sum over DPs of n * k_h) per second of
            device time, summed over ranks; L2 is flushed between steps, and the
            timed plans carry no per-launch events (the phase breakdown comes
            from the warm-up plans)
  e2e       the same metric through the C ABI from pinned host buffers:
            pp_instance_create (upload + tables) + pp_plan_run (placement
            back to the host) + pp_instance_destroy, every step
  roofline  the tree-DP step (dominant): the algorithmic bytes of the paper's
            table algorithm (decision bits n(k+1)/8, p/w/next 16n, every
            pushed skip row written and read once 16(k+1) per push, the
            traceback's at most n states 8n) per DP, times the DPs of a step,
            over the step's CUDA-event time, against the measured HBM copy
            bandwidth; the dependent row chain that actually limits the kernel
            is reported beside it (t_row_min)
  cpu_baseline  the CPU oracle's whole plan of the same workload on the
            host's cores (one thread per start), outside the timed region
  configs   the same measurements for all five synthetic workloads (tiny,
            RAG, source-dependent, paper-scale, stress), each with its oracle
            baseline (the whole plan, or a bounded sample for the stress one)

--impl reference runs the oracle (the only reference implementation of this
path) on the host cores and prints the same line with "impl": "reference".
Multi-GPU (torchrun): --scaling weak (default) plans 16 starts per GPU out of
16 x N default start orders, --scaling strong splits the 16 starts of one
plan; rank r plans the starts s with s % N == r and the candidates are
compared once after the timed region (no exchange while planning).
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)
# hardware queues for the plan's per-start streams; acts when the CUDA context
# is created, so it is set before torch touches the GPU
os.environ.setdefault("CUDA_DEVICE_MAX_CONNECTIONS", "32")

METRIC = "tree-DP cell-updates/s and end-to-end plan time (n=50k, 16 workers) vs HBM roofline"
UNIT = "cell-updates/s"
HEADLINE_CONFIG = 3         # the n = 50,000 / W = 16 / k = 4,096 workload
SM_COUNT = 152
INT32_LANES_PER_SM = 64     # integer add/compare/select/logic: 16 lanes per scheduler, 4 schedulers
ALU_OPS_PER_CELL = 6        # int64 add, compare, select = 2 + 2 + 2 int32 lane operations
# side configurations: (warm-up plans, timed plans, timed end-to-end plans)
SIDE_STEPS = {0: (3, 5, 3), 1: (3, 5, 3), 2: (3, 5, 3), 4: (3, 1, 1)}


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "sm_max_mhz": 2070.0}, "fallback"


# --------------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(prefix="pp_clocks_", suffix=".csv")
        os.close(fd)
        try:
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.out, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.out.close()

    def summary(self):
        rows = []
        if self.path and os.path.exists(self.path):
            for line in open(self.path):
                p = [x.strip() for x in line.split(",")]
                if len(p) >= 9:
                    try:
                        rows.append((float(p[1]), float(p[2]), p[5:9]))
                    except ValueError:
                        pass
            os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, r in rows for i in range(4) if r[i].lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


# --------------------------------------------------------------------------- byte models
def table_bytes(parent, k: int):
    """Algorithmic bytes of one Eq. 9 DP of budget k over the whole tree, for
    the paper's table algorithm (Theorem 1): B_min = decision bits n(k+1)/8 +
    p, w, next of every row 16n + every skip row that a later row reads,
    written once and read once, 16(k+1) per push of the tree's stack plan +
    the traceback's at most n visited states, 8n; B_stream adds the per-row
    gather of D[next(i)] ((k+1) int64 words) for every internal row
    (next(i) != i + 1), as a table algorithm that streams rows from memory
    reads it."""
    from paper_2608_01655_gb300 import binding as pp
    order, nxt, skipc, pushl, depth = pp.pp_row_plan(parent)
    n = len(parent)
    n_push = int((pushl >= 0).sum())
    n_internal = int((nxt != np.arange(n) + 1).sum())
    bmin = n * (k + 1) / 8 + 16 * n + 16 * (k + 1) * n_push + 8 * n
    bstream = bmin + 8 * (k + 1) * n_internal
    return {"bmin_bytes_per_dp": bmin, "bstream_bytes_per_dp": bstream, "n_push": n_push,
            "n_internal": n_internal}


# --------------------------------------------------------------------------- oracle legs
def _host_cores():
    return len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)


def oracle_plan(inst, threads: int):
    """The oracle's whole plan of the workload (default orders, its own
    standalone-score DPs, safeguards where they apply), one thread per start
    up to `threads`.  Returns (result, seconds)."""
    import oracle
    prob = oracle.Problem.from_instance(inst)
    t0 = time.perf_counter()
    r = oracle.plan(prob, inst.starts, inst.rounds, threads=threads)
    return r, time.perf_counter() - t0


def oracle_updates(inst, count: int, seed: int = 0):
    """A bounded sample: `count` oracle worker updates (Eq. 7 / Eq. 10
    marginals + Eq. 9 DP + backtrack), each against its own random holder
    sets (every worker holds ~5% of the chunks, as in the middle of a plan),
    run concurrently on `count` threads (the oracle releases the interpreter
    while it works).  Returns (cells, seconds)."""
    import oracle
    prob = oracle.Problem.from_instance(inst)
    rng = np.random.default_rng(seed)
    jobs = []
    for x in range(count):
        pl = (rng.random((inst.W, inst.n)) < 0.05).astype(np.uint8)
        jobs.append((int(rng.integers(inst.W)), pl))
    cells = sum(inst.n * int(inst.budget[h]) for h, _ in jobs)
    threads = [threading.Thread(target=oracle.worker_update, args=(prob, h, pl)) for h, pl in jobs]
    t0 = time.perf_counter()
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    return cells, time.perf_counter() - t0


def _config(inst, S, world=1, scaling="weak"):
    """The workload of both arms (the reference arm times the oracle on it)."""
    par = (f"starts ({scaling}: {S} per GPU)" if scaling == "weak" else f"starts ({scaling}: {S} over {world} GPUs)")
    return {"workload": inst.name, "n": inst.n, "W": inst.W, "k": int(inst.budget.max()), "starts": S,
            "rounds": inst.rounds, "mode": "source-dependent" if inst.mode else "requester-side",
            "l2": "flushed between steps (256 MiB write)", "parallelism": par}


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    from paper_2608_01655_gb300 import workloads as wl
    import oracle
    oracle.build()
    inst = wl.make(args.config)
    cores = _host_cores()
    oracle_updates(inst, cores, seed=10_000)           # warm the page cache and the library
    for w in range(args.warmup):
        oracle_updates(inst, cores, seed=w)
    cells = 0
    secs = 0.0
    for s in range(args.steps):
        c, t = oracle_updates(inst, cores, seed=1000 + s)
        cells += c
        secs += t
    value = cells / secs
    sample = (f"{cores} oracle worker updates per step, one per host core, concurrently "
              f"(Eq. 7/10 marginals + Eq. 9 DP + backtrack, {inst.n} x {int(inst.budget[0])} cells each)")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * secs / args.steps,
        "higher_is_better": True, "scaling": args.scaling, "vs_baseline": None, "dtype": "int64",
        "data": "synthetic", "config": _config(inst, inst.starts, args.gpus, args.scaling),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "gpu_launches": 0,
    }
    print(json.dumps(line), flush=True)
    return 0


# --------------------------------------------------------------------------- native arm
def _dist():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


TRAFFIC_SUMMARY = os.path.join(ROOT, "profiles", "k_tree_dp_wave_traffic_paper-n50000-k4096.md")
DP_SOURCES = [os.path.join(ROOT, "paper_2608_01655_gb300", "csrc", f) for f in ("pp_dp.cu", "pp_internal.cuh")]


def dp_source_sha256():
    h = hashlib.sha256()
    for f in DP_SOURCES:
        h.update(open(f, "rb").read())
    return h.hexdigest()


def _traffic_record():
    """DRAM traffic per swept cell of the tree-DP kernel from the committed
    one-kernel ncu capture (its `traffic_record:` line), used only while the DP
    sources are unchanged since the counters were taken."""
    try:
        for line in open(TRAFFIC_SUMMARY):
            if line.startswith("traffic_record:"):
                rec = json.loads(line.split(":", 1)[1])
                return rec if rec.get("kernel_src_sha256") == dp_source_sha256() else None
    except (OSError, ValueError):
        pass
    return None


def _probe_read_gbs(torch, stream, nbytes, iters):
    """Read bandwidth of a device buffer (libpp_probe.so, the benchmark's
    bandwidth probe; not part of the planner)."""
    from paper_2608_01655_gb300 import build
    lib = ctypes.CDLL(build.PROBE_LIB)
    lib.pp_probe_read.argtypes = [ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int32, ctypes.c_void_p,
                                  ctypes.c_void_p]
    lib.pp_probe_read.restype = ctypes.c_int
    sink = torch.zeros(1, dtype=torch.int64, device="cuda")
    buf = torch.ones(nbytes // 8, dtype=torch.int64, device="cuda")
    sp = ctypes.c_void_p(stream.cuda_stream)

    def call(it):
        rc = lib.pp_probe_read(ctypes.c_void_p(buf.data_ptr()), nbytes, it, ctypes.c_void_p(sink.data_ptr()), sp)
        if rc != 0:
            raise RuntimeError(f"pp_probe_read failed ({rc})")

    call(1)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    call(iters)
    e1.record(stream)
    torch.cuda.synchronize()
    del buf
    return nbytes * iters / (e0.elapsed_time(e1) / 1000.0) / 1e9


def _t_row_min(pp, torch, inst, ppi, res, S, stream):
    """Per-row time of the smallest DP launch shape (one warp per DP, 32
    columns, no hand-off between warps) on the plan's last marginals: the
    dependent row chain alone."""
    n = inst.n
    masks = np.zeros((S, n), np.uint32)
    for m in range(inst.W):
        masks |= res.placement[m].astype(np.uint32) << np.uint32(m)
    masks_t = torch.from_numpy(masks.view(np.int32)).cuda()
    workers = torch.arange(S, dtype=torch.int32, device="cuda") % inst.W
    prof = torch.zeros((S, n), dtype=torch.int64, device="cuda")
    pp.pp_marginals(ppi, workers, masks_t, prof)
    kk = 32
    pp.pp_tune_dp(ppi, 1, 1, False, False)
    try:
        bud = torch.full((S,), kk, dtype=torch.int32, device="cuda")
        best = torch.zeros(S, dtype=torch.int64, device="cuda")
        bits = torch.zeros(pp.pp_dp_bits_size(ppi, S, kk) // 4, dtype=torch.int32, device="cuda")
        ts = []
        for it in range(4):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            pp.pp_tree_dp(ppi, prof, bud, kk, best, bits)
            e1.record(stream)
            torch.cuda.synchronize()
            if it:
                ts.append(e0.elapsed_time(e1) / 1000.0)
        ppi.sync()
        rows_max = int(pp.pp_dp_rows_swept(ppi, S, kk, bits).max())
    finally:
        pp.pp_tune_dp(ppi, 0, 0, False, False)
    return min(ts) / rows_max


def measure_plan(pp, torch, ppi, S, R, orders, warmup, steps, flush, stream, sched, sg, barrier=None):
    """`warmup` untimed plans with CUDA events around every launch (the
    phase breakdown: their mean, the first plan left out), then `steps`
    plans timed with CUDA events on the launching stream and no per-launch
    events (they cost ~1% and sit between dependent launches), L2 flushed
    before each.  Returns (last result, per-step seconds, phase ms summed as
    over `steps` plans)."""
    res = None
    acc, nacc = [0.0, 0.0, 0.0], 0
    for w in range(warmup):
        flush.fill_(1)
        torch.cuda.synchronize()
        res = pp.pp_plan_run(ppi, S, orders, R, time_phases=True, safeguards=sg, schedule=sched)
        if w > 0 or warmup == 1:
            for x in range(3):
                acc[x] += res.phase_ms[x]
            nacc += 1
    times = []
    for _ in range(steps):
        flush.fill_(1)
        if barrier:
            barrier()
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        # the NVTX range lets a profiler select the timed plans' launches
        torch.cuda.nvtx.range_push("timed_plan")
        res = pp.pp_plan_run(ppi, S, orders, R, safeguards=sg, schedule=sched)
        torch.cuda.nvtx.range_pop()
        e1.record(stream)
        torch.cuda.synchronize()
        if barrier:
            barrier()
        times.append(e0.elapsed_time(e1) / 1000.0)
    phase = [a / max(nacc, 1) * len(times) for a in acc]
    return res, times, phase


def measure_e2e(pp, torch, inst, S, R, orders, warmup, steps, flush, sched, sg, objective):
    """The plan through the C ABI from pinned host buffers, every step:
    instance creation (upload + tables), pp_plan_run (placement back to the
    host), instance destruction.  Returns (per-step seconds, h2d bytes,
    d2h bytes)."""
    host = {}
    for name in ("parent", "weight", "demand", "recompute", "transfer", "budget"):
        a = np.ascontiguousarray(getattr(inst, name))
        host[name] = torch.from_numpy(a).pin_memory().numpy()
    h2d = sum(v.nbytes for v in host.values())
    d2h = inst.W * inst.n + 8 * (S * 3 + 1)
    times = []
    for it in range(warmup + steps):
        flush.fill_(3)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        with pp.Instance(host["parent"], host["weight"], host["demand"], host["recompute"],
                         host["transfer"], inst.mode, host["budget"]) as ppe:
            r2 = pp.pp_plan_run(ppe, S, orders, R, safeguards=sg, schedule=sched)
        torch.cuda.synchronize()
        if it >= warmup:
            times.append(time.perf_counter() - t0)
        assert r2.objective == objective
    return times, h2d, d2h


def plan_summary(inst, res, times, phase, e2e_times, h2d, d2h, l2_gbs, hbm_gbs):
    """Per-workload figures: plan time with inputs resident and with upload,
    executed and swept cells/s, per-update latency, and the table
    algorithm's B_min / B_stream bytes over the DP step's time as fractions
    of the HBM copy and L2 read bandwidths."""
    k = int(inst.budget.max())
    plan_s = sum(times) / len(times)
    nl = max(res.dp_launches, 1)
    dp_t = phase[1] / 1000.0 / (nl * len(times))
    items = res.dp_count / nl
    tb = table_bytes(inst.parent, k)
    out = {
        "workload": inst.name, "n": inst.n, "W": inst.W, "k": k, "starts": inst.starts, "rounds": inst.rounds,
        "mode": "source-dependent" if inst.mode else "requester-side",
        "steps": len(times), "plan_ms": 1000 * plan_s,
        "plan_ms_with_upload": 1000 * sum(e2e_times) / len(e2e_times) if e2e_times else None,
        "e2e_steps": len(e2e_times), "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
        "cells_per_s_executed": res.dp_cells / plan_s,
        "cells_per_s_swept": res.dp_rows_swept * k / plan_s,
        "update_ms": sum(phase) / (nl * len(times)),
        "dp_step_ms": 1000 * dp_t, "dps_per_step": items,
        "phase_ms": {"marginals": phase[0] / len(times), "tree_dp": phase[1] / len(times),
                     "traceback_accept": phase[2] / len(times)},
        **tb,
        "bmin_gbs": items * tb["bmin_bytes_per_dp"] / dp_t / 1e9,
        "bmin_frac_of_hbm": items * tb["bmin_bytes_per_dp"] / dp_t / 1e9 / hbm_gbs,
        "bstream_frac_of_l2": items * tb["bstream_bytes_per_dp"] / dp_t / 1e9 / l2_gbs,
        "objective": res.objective, "best_start": res.best_start,
        "sweeps": res.per_start_sweeps.tolist(), "dp_count": res.dp_count, "dp_cells": res.dp_cells,
        "dp_rows_swept": res.dp_rows_swept, "schedule": "per-start streams" if res.schedule == 2 else "lock step",
    }
    return out


def _extras(pp, torch, wl, inst, res):
    """Timings of the steps next to the plan (outside the timed region):
    the requester-side safeguard candidates on the RAG workload, one epoch
    update of the paper-scale plan after a popularity shift (log-normal
    sigma = 0.5 on every demand entry, as in RQ5), and the plan at the
    paper's runtime-study budget (k = 128)."""
    out = {}
    rag = wl.make(1)
    with pp.Instance.from_workload(rag) as ppr:
        pp.pp_safeguards(ppr)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        _, sg_obj = pp.pp_safeguards(ppr)
        t_sg = time.perf_counter() - t0
        t0 = time.perf_counter()
        r1 = pp.pp_plan_run(ppr, rag.starts, None, rag.rounds)
        t_plan = time.perf_counter() - t0
    out["safeguards"] = {"workload": rag.name, "ms": 1000 * t_sg, "objectives": [int(x) for x in sg_obj],
                         "plan_ms_with_safeguards": 1000 * t_plan, "plan_objective": r1.objective,
                         "plan_best_candidate": r1.best_start}
    rng = np.random.default_rng(2026)
    dem = np.rint(inst.demand * rng.lognormal(0.0, 0.5, inst.demand.shape)).astype(np.int64)
    shifted = wl.Instance(**{**inst.__dict__, "demand": dem})
    with pp.Instance.from_workload(shifted) as pps:
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        rr = pp.pp_replan(pps, res.placement, inst.starts, inst.rounds, wl.REQUESTS_PER_EPOCH,
                          wl.REQUESTS_PER_EPOCH)
        t_rp = time.perf_counter() - t0
    out["epoch_update"] = {"workload": inst.name, "shift": "popularity, log-normal sigma 0.5", "ms": 1000 * t_rp,
                           "incumbent_objective": rr.incumbent_objective, "new_objective": rr.new_objective,
                           "materialization_cost_us": rr.materialization_cost,
                           "break_even_requests": rr.break_even_requests, "adopted_at_one_epoch": rr.adopted}
    # the paper's runtime study shape (Fig. 7: n = 50,000, M = 16, k = 128 per
    # worker, 12.29 s for its CPU solver) on the same synthetic workload
    small = wl.Instance(**{**inst.__dict__, "budget": np.full(inst.W, 128, np.int32)})
    with pp.Instance.from_workload(small) as ppk:
        pp.pp_plan_run(ppk, small.starts, None, small.rounds)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        rk = pp.pp_plan_run(ppk, small.starts, None, small.rounds)
        t_k = time.perf_counter() - t0
    out["paper_runtime_shape"] = {"workload": "paper-n50000-W16-k128", "starts": small.starts,
                                  "rounds": small.rounds, "ms": 1000 * t_k, "objective": rk.objective,
                                  "context": "the paper's CPU solver: 12.29 s on one EPYC 9V74 (Fig. 7); "
                                             "starts, objective variant and safeguards not stated there"}
    return out


def side_config(pp, torch, wl, cfg, flush, stream, sched, l2_gbs, hbm_gbs, with_oracle):
    """Plan, end-to-end and oracle figures of one more workload (single GPU)."""
    inst = wl.make(cfg)
    warm, steps, e2e_steps = SIDE_STEPS[cfg]
    sg = True
    with pp.Instance.from_workload(inst) as ppi:
        res, times, phase = measure_plan(pp, torch, ppi, inst.starts, inst.rounds, None, warm, steps, flush,
                                         stream, sched, sg)
    e2e_times, h2d, d2h = measure_e2e(pp, torch, inst, inst.starts, inst.rounds, None, 0, e2e_steps, flush,
                                      sched, sg, res.objective)
    out = plan_summary(inst, res, times, phase, e2e_times, h2d, d2h, l2_gbs, hbm_gbs)
    out["warmup"] = warm
    if with_oracle:
        out["oracle"] = oracle_leg(inst, res)
    return out


def oracle_leg(inst, res):
    """The oracle on the host cores: the whole plan where it finishes in
    seconds (cross-checked against the GPU plan's objective and placement), a
    bounded sample of concurrent worker updates for the stress workload."""
    cores = _host_cores()
    if inst.n * int(inst.budget.max()) * inst.W * inst.starts * (1 + inst.rounds) > 2e12:
        count = min(cores, 16)
        cells, secs = oracle_updates(inst, count, seed=7)
        rate = cells / secs
        return {"kind": "oracle sample", "cores": count, "value": rate, "unit": UNIT,
                "sample": f"{count} concurrent worker updates (marginals + Eq. 9 DP + backtrack, "
                          f"{inst.n} x {int(inst.budget.max())} cells each), {secs:.1f} s",
                "plan_s_extrapolated": res.dp_cells / rate,
                "extrapolation": "the GPU plan's executed cells at the sample's rate"}
    threads = min(inst.starts, cores)
    r, secs = oracle_plan(inst, threads)
    return {"kind": "oracle plan", "cores": threads, "value": r.cells / secs, "unit": UNIT, "plan_s": secs,
            "cells": r.cells, "sample": f"the whole plan ({inst.starts} starts, {inst.rounds} rounds), "
                                        f"one thread per start",
            "objective_equal": r.objective == res.objective, "best_start_equal": r.best_start == res.best_start,
            "placement_equal": bool(np.array_equal(r.placement, res.placement))}


def run_native(args):
    import torch
    world, rank, local = _dist()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    else:
        torch.cuda.set_device(0)
    from paper_2608_01655_gb300 import binding as pp
    from paper_2608_01655_gb300 import shard
    from paper_2608_01655_gb300 import workloads as wl

    inst = wl.make(args.config)
    S, R = inst.starts, inst.rounds
    stream = torch.cuda.current_stream()
    ppi = pp.Instance.from_workload(inst)
    orders, my_idx = None, np.arange(S)
    if world > 1:
        # every rank computes the same default orders; rank r plans s % world == r
        orders, my_idx = shard.rank_orders(lambda total: pp.pp_default_orders(ppi, total), S, rank, world,
                                           args.scaling)
    S_mine = len(my_idx) if world > 1 else S
    # the requester-side safeguards are candidates of the whole plan, not of a
    # start: with several ranks only the starts are sharded and compared
    sg = world == 1
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")   # 2x the 129 MB L2

    def barrier():
        if world > 1:
            torch.distributed.barrier()

    sched = {"auto": 0, "lock": 1, "per-start": 2}[args.schedule]
    with ClockSampler(local) as clk:
        res, times, phase = measure_plan(pp, torch, ppi, S_mine, R, orders, args.warmup, args.steps, flush, stream,
                                         sched, sg, barrier=barrier)
    clocks = clk.summary()
    total = sum(times)
    cells_mine = res.dp_cells * args.steps
    if world > 1:
        t = torch.tensor([total, float(cells_mine)], dtype=torch.float64, device="cuda")
        tm = t.clone()
        torch.distributed.all_reduce(tm, op=torch.distributed.ReduceOp.MAX)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.SUM)
        total, cells_all = float(tm[0].item()), float(t[1].item())
    else:
        cells_all = float(cells_mine)
    value = cells_all / total

    # ---- the dominant kernel: the plan's tree-DP steps (row pruning + Eq. 9
    # sweep), CUDA events on the launching streams over the timed region
    peaks, peak_kind = _peaks()
    hbm_peak = float(peaks.get("hbm_gbs", 6800.0))
    k = int(inst.budget.max())
    nl = max(res.dp_launches, 1)
    dp_t = phase[1] / 1000.0 / (nl * args.steps)               # s per DP step
    items = res.dp_count / nl                                   # DPs per step
    rows_swept = res.dp_rows_swept / nl
    cells_swept = rows_swept * k
    tb = table_bytes(inst.parent, k)
    bmin_step = items * tb["bmin_bytes_per_dp"]
    achieved = bmin_step / dp_t / 1e9
    l2_gbs = _probe_read_gbs(torch, stream, 32 << 20, 200)     # 32 MiB: resident in L2
    hbm_read_gbs = _probe_read_gbs(torch, stream, 4 << 30, 3)  # 4 GiB: far larger than L2
    t_row_min = _t_row_min(pp, torch, inst, ppi, res, S_mine, stream)
    sm_mhz = float(peaks.get("sm_max_mhz", 2070.0))
    alu_peak = SM_COUNT * INT32_LANES_PER_SM * sm_mhz * 1e6 / ALU_OPS_PER_CELL   # cells/s
    tr = _traffic_record()
    traffic = None
    if tr and tr.get("bytes_per_swept_cell"):
        traffic = tr["bytes_per_swept_cell"] * cells_swept
    per_start = res.schedule == 2
    roofline = {
        "bound": "hbm", "achieved": achieved, "peak": hbm_peak, "unit": "GB/s", "frac": achieved / hbm_peak,
        "traffic": traffic,
        "peak_source": f"MEASURED_PEAKS.json hbm_gbs ({peak_kind} copy bandwidth)",
        "achieved_source": ("algorithmic bytes of the paper's table algorithm per DP (bmin_bytes_per_dp: "
                            "n(k+1)/8 decision bits + 16n p/w/next + 16(k+1) per skip-row push + 8n "
                            "traceback) x DPs per step / the step's CUDA-event time"),
        "traffic_source": ("DRAM bytes per swept cell of a one-kernel ncu capture of the batched DP on the "
                           "small profile case, times the step's swept cells" if traffic is not None else
                           "no capture of the current DP sources"),
        "limiter": ("latency: the dependent row chain of Eq. 9 (one warp's rows follow one another; "
                    "t_dp_over_rows_x_t_row_min compares the step with that chain alone)"),
        "kernel": ("k_prune + k_tree_dp_wave (one tree-DP step of the plan: every start's DP on its own "
                   "stream, concurrently; duration = mean over starts of the start's DP events)"
                   if per_start else "k_prune + k_tree_dp_wave (one batched tree-DP launch of the plan)"),
        "launches": nl * args.steps, "launch_ms": 1000 * dp_t, "items_per_launch": items,
        **tb,
        "bmin_bytes_per_launch": bmin_step,
        "cells_per_launch": res.dp_cells / nl, "cells_swept_per_launch": cells_swept,
        "rows_swept_per_launch": rows_swept,
        "bstream_gbs": items * tb["bstream_bytes_per_dp"] / dp_t / 1e9,
        "bstream_frac_of_l2": items * tb["bstream_bytes_per_dp"] / dp_t / 1e9 / l2_gbs,
        "l2_read_gbs_probe": l2_gbs, "hbm_read_gbs_probe": hbm_read_gbs,
        "t_row_min_ns": 1e9 * t_row_min,
        "t_row_min_source": "one warp per DP, 32 columns, the same rows (pp_tune_dp(inst, 1, 1))",
        "t_dp_over_rows_x_t_row_min": dp_t / ((rows_swept / items) * t_row_min),
        "alu_model": {"achieved_tcells": cells_swept / dp_t / 1e12, "peak_tcells": alu_peak / 1e12,
                      "frac": cells_swept / dp_t / alu_peak,
                      "source": (f"derived, not measured: {SM_COUNT} SMs x {INT32_LANES_PER_SM} int32 ALU lanes x "
                                 f"{sm_mhz:.0f} MHz / {ALU_OPS_PER_CELL} int32 ops per cell; counts only the "
                                 f"16-lane ALU pipe of each scheduler (adds that issue on the FMA pipe are not "
                                 f"credited), and only the cells the pruned sweep computes")},
    }

    # ---- end to end through the C ABI from pinned host buffers -------------
    e2e_times, h2d, d2h = measure_e2e(pp, torch, inst, S_mine, R, orders, args.warmup, args.steps, flush, sched,
                                      sg, res.objective)
    e2e_total = sum(e2e_times)
    if world > 1:
        t = torch.tensor([e2e_total], dtype=torch.float64, device="cuda")
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        e2e_total = float(t.item())
    e2e_value = cells_all / e2e_total
    headline = plan_summary(inst, res, times, phase, e2e_times, h2d, d2h, l2_gbs, hbm_peak)

    # ---- candidates of all ranks compared once (outside the timed region) ---
    best_obj, best_start = res.objective, res.best_start
    if world > 1:
        won = shard.exchange(res.objective, int(my_idx[res.best_start]), res.placement)
        best_obj, best_start = won.objective, won.best_start

    extras = _extras(pp, torch, wl, inst, res) if rank == 0 and world == 1 and not args.headline_only else None
    geometry = {**pp.pp_dp_geometry(ppi, S_mine, k), "split": pp.pp_dp_split(ppi, S_mine, k)}
    ppi.close()

    # ---- the other four workloads (single GPU) -----------------------------
    configs = {}
    if world == 1 and not args.headline_only:
        for cfg in (0, 1, 2, 4):
            if cfg != args.config:
                configs[wl.make(cfg).name] = side_config(pp, torch, wl, cfg, flush, stream, sched, l2_gbs,
                                                         hbm_peak, not args.no_cpu_baseline)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        leg = oracle_leg(inst, res)
        headline["oracle"] = leg
        cpu = {"value": leg["value"], "unit": UNIT, "cores": leg["cores"], "kind": leg["kind"],
               "sample": leg["sample"], "host_cores": _host_cores()}
        for key in ("plan_s", "objective_equal", "best_start_equal", "placement_equal", "plan_s_extrapolated"):
            if key in leg:
                cpu[key] = leg[key]
        cpu["gpu_plan_s"] = sum(times) / len(times)
    configs = {inst.name: headline, **configs}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1000 * total / args.steps, "higher_is_better": True,
            "scaling": args.scaling, "vs_baseline": None, "dtype": "int64", "data": "synthetic",
            "config": _config(inst, S, world, args.scaling),
            "roofline": roofline,
            "cpu_baseline": cpu,
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "ms_per_step": 1000 * e2e_total / args.steps},
            "gpu_launches": res.kernel_launches * args.steps,
            "clocks": clocks,
            "plan": {"objective": best_obj, "best_start": best_start,
                     "schedule": "per-start streams" if per_start else "lock step",
                     "hw_queues_assumed": res.hw_queues,
                     "dp_count": res.dp_count, "dp_cells": res.dp_cells,
                     "dp_launches": nl, "dp_rows_swept": res.dp_rows_swept,
                     "dp_cells_swept": res.dp_rows_swept * k,
                     "cells_per_s_swept_here": res.dp_rows_swept * k * args.steps / total,
                     "starts_planned_here": int(S_mine),
                     "sweeps": res.per_start_sweeps.tolist(),
                     "step_ms": [round(1000 * t, 3) for t in times]},
            "phase_ms": {"marginals": phase[0] / args.steps, "tree_dp": phase[1] / args.steps,
                         "traceback_accept": phase[2] / args.steps},
            "update_ms": sum(phase) / (nl * args.steps),
            "update_note": ("one worker update (marginals + tree DP + traceback/accept) of every start, "
                            "the starts on their own streams (phase times: mean over starts)" if per_start else
                            "one batched worker update (marginals + tree DP + traceback/accept) of all starts"),
            "configs": configs,
            "next_steps": extras,
            "dp_geometry": geometry,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def run_profile_dp(args):
    """A small case for ncu: marginals, the tree DP and the traceback of
    `--profile-dp B` items of the headline workload, launched twice (ncu
    captures the second)."""
    import torch
    torch.cuda.set_device(0)
    from paper_2608_01655_gb300 import binding as pp
    from paper_2608_01655_gb300 import workloads as wl
    inst = wl.make(args.config)
    ppi = pp.Instance.from_workload(inst)
    B, n, k = args.profile_dp, inst.n, int(inst.budget.max())
    workers = torch.arange(B, dtype=torch.int32, device="cuda") % inst.W
    masks = torch.zeros((B, n), dtype=torch.int32, device="cuda")
    prof = torch.zeros((B, n), dtype=torch.int64, device="cuda")
    bud = torch.full((B,), k, dtype=torch.int32, device="cuda")
    best = torch.zeros(B, dtype=torch.int64, device="cuda")
    bits = torch.zeros(pp.pp_dp_bits_size(ppi, B, k) // 4, dtype=torch.int32, device="cuda")
    chosen = torch.zeros((B, n), dtype=torch.uint8, device="cuda")
    for _ in range(2):
        pp.pp_marginals(ppi, workers, masks, prof)
        pp.pp_tree_dp(ppi, prof, bud, k, best, bits)
        pp.pp_traceback(ppi, bits, bud, k, chosen)
    ppi.sync()
    rows = pp.pp_dp_rows_swept(ppi, B, k, bits)
    print(json.dumps({"profile_dp": B, "geometry": pp.pp_dp_geometry(ppi, B, k), "split": pp.pp_dp_split(ppi, B, k),
                      "rows_swept": rows.tolist(), "cells_swept": int(rows.sum()) * k,
                      "dp_src_sha256": dp_source_sha256(), "best": best.tolist()}))
    ppi.close()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["native", "reference"], default="native")
    ap.add_argument("--config", type=int, default=HEADLINE_CONFIG, choices=range(5),
                    help="headline workload (0 tiny, 1 RAG, 2 source-dependent, 3 paper-scale, 4 stress)")
    ap.add_argument("--scaling", choices=["weak", "strong"], default="weak",
                    help="with several GPUs: weak = 16 starts per GPU, strong = the 16 starts of one plan split")
    ap.add_argument("--headline-only", action="store_true",
                    help="skip the other four workloads and the side timings")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--schedule", choices=["auto", "lock", "per-start"], default="auto",
                    help="plan schedule: automatic (per-start streams when the hardware queues allow), "
                         "lock step, or per-start streams")
    ap.add_argument("--profile-dp", type=int, default=0, metavar="B",
                    help="only launch the tree DP and traceback of B items twice (a small case for ncu) and exit")
    args = ap.parse_args()
    if args.profile_dp:
        return run_profile_dp(args)
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        return run_reference(args)
    return run_native(args)


if __name__ == "__main__":
    sys.exit(main())
