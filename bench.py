"""Benchmark of the batched HexGen-Flow scheduler simulation on GB300.

One step = one pass of the whole path through the C ABI (`hx_sim_run`):
per-call preparation, every (trace x point) simulation, the best-point
reduction, on the ceiling workload (256 traces x 20000 queries, 64
instances of 4 types, 1024 hyper-parameter points = 262144 simulations).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
    python bench.py --recipe faulty --traces 256        # another recipe
    python bench.py --traces 64 --policy rr-fcfs        # a policy variant


Prints one JSON line.  `value` is simulations per second over the timed
steps (inputs resident in HBM; they are larger than L2, so no flush is
needed).  `e2e` is the same metric through the C ABI from pinned host buffers:
upload of the traces, the run, and the read-back of the results per step.
`--impl reference` times the CPU oracle (plain C, one simulation per
process, all host cores) on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2505_05286_gb300 import dist as D  # noqa: E402
from paper_2505_05286_gb300 import workloads as W  # noqa: E402

CFG = 4
METRIC = "scheduler sims/sec (hyperparam×trace) and simulated stage-events/sec on 1 GB300"
UNIT = "sims/s"
L2_BYTES = 129 * 2 ** 20
SM_COUNT_FALLBACK = 152


WARP_INST_PER_EVENT = 300
KERNEL_SRC = os.path.join(ROOT, "paper_2505_05286_gb300", "csrc", "hx_kernels.cu")
# ncu figures of the simulation kernel, each file keyed to the kernel source's
# SHA-256: DRAM traffic of one full ceiling launch (a one-pass capture of the
# DRAM byte counters alone), and issue-slot use and instruction mix per
# simulated call event (a multi-metric capture of a small case that still
# fills the GPU: 64 traces x 2000 queries x 1024 points)
# hx_info.work_order: the order the kernel takes the simulations in
WORK_ORDERS = {0: "trace-major, highest point first", 1: "the subset's",
               2: "every trace's alpha = 1 points first, then trace-major",
               3: "trace-major; the last two waves' traces with their alpha = 1 points first"}
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "hx_sim_kernel_ceiling_dram.txt")
COUNTERS_FILE = os.path.join(ROOT, "profiles", "hx_sim_kernel_small_counters.txt")


# grid-wide policy overrides (Sec. 5.1's ablations and baselines): local queue, dispatch
POLICIES = {"wb-pq": (W.POLICY_PQ, W.DISPATCH_WB), "wb-fcfs": (W.POLICY_FCFS, W.DISPATCH_WB),
            "rr-pq": (W.POLICY_PQ, W.DISPATCH_RR), "rr-fcfs": (W.POLICY_FCFS, W.DISPATCH_RR),
            "wb-llf": (W.POLICY_LLF, W.DISPATCH_WB)}


def _recipe(arg: str):
    return int(arg) if arg.isdigit() else arg


def _workload(args, first_trace: int = 0):
    """The benchmarked workload: a recipe, optionally cut (--traces,
    --queries, --alpha) and with one policy on every grid point (--policy)."""
    wl = W.make_workload(_recipe(args.recipe), n_traces=args.traces, n_queries=args.queries,
                         first_trace=first_trace)
    if args.alpha != "all":
        # profiling: only the alpha = 1 points, or only the others
        keep = (wl.grid.alpha_fp == W.SCALE) if args.alpha == "1" else (wl.grid.alpha_fp != W.SCALE)
        wl = W.Workload(f"{wl.name}[alpha {args.alpha}]", wl.traces, wl.cluster,
                        W.subset_grid(wl.grid, np.nonzero(keep)[0]), wl.objective)
    if args.policy != "grid":
        lp, dp = POLICIES[args.policy]
        g = wl.grid
        g = W.Grid(g.alpha_fp, g.gamma_fp, g.rho, g.beta_us2, np.full(g.n_points, lp, np.uint8),
                   np.full(g.n_points, dp, np.uint8))
        wl = W.Workload(f"{wl.name}[{args.policy}]", wl.traces, wl.cluster, g, wl.objective)
    return wl


def _is_ceiling(args) -> bool:
    return (_recipe(args.recipe) == CFG and args.traces is None and args.queries is None
            and args.alpha == "all" and args.policy == "grid")


def _ncu_figures(path=COUNTERS_FILE):
    """key=value figures of a committed ncu capture of the simulation kernel;
    {} when the kernel source changed since the capture."""
    import hashlib
    try:
        kv = dict(line.strip().split("=", 1) for line in open(path)
                  if "=" in line and not line.startswith("#"))
        with open(KERNEL_SRC, "rb") as f:
            sha = hashlib.sha256(f.read()).hexdigest()
        return kv if kv.get("kernel_sha256") == sha else {}
    except OSError:
        return {}


def _traffic_per_launch(n_sims: int):
    """DRAM bytes (read + write) of one simulation-kernel launch on the
    ceiling workload from the committed full-size capture; None when the
    kernel source changed since the capture."""
    kv = _ncu_figures(TRAFFIC_FILE)
    try:
        return float(kv["dram_bytes_per_launch"]) * n_sims / float(kv["sims_per_launch"])
    except (KeyError, ValueError):
        return None


def summarize_ncu(csv_path: str, bench_json: str, kind: str, command: str) -> str:
    """key=value summary of an ncu CSV (--csv --log-file) of the simulation
    kernel, per launch, with the kernel source's SHA-256; `bench_json` is the
    bench line of the same command run without ncu (events and simulations
    per launch).  kind: "ceiling" (DRAM bytes of a full launch) or "small"
    (issue-slot use and instruction mix per simulated call event)."""
    import csv
    import hashlib
    vals = {}
    launches = set()
    with open(csv_path) as f:
        rows = [r for r in csv.reader(f) if r]
    hdr = next(r for r in rows if r[0] == "ID")
    if kind == "launches":
        # every captured launch: per kernel its launches, total time and share
        per_k = {}
        for r in rows[rows.index(hdr) + 1:]:
            d = dict(zip(hdr, r))
            if d.get("Metric Name") == "gpu__time_duration.sum":
                name = d["Kernel Name"].split("(")[0]
                t = per_k.setdefault(name, [0, 0.0])
                t[0] += 1
                t[1] += float(d["Metric Value"].replace(",", "")) / 1e6
        tot = sum(v[1] for v in per_k.values())
        out = [f"# ncu launch list (gpu__time_duration.sum), command: {command}",
               "| kernel | launches | total ms | share |", "|---|---|---|---|"]
        for name, (n, ms) in sorted(per_k.items(), key=lambda kv: -kv[1][1]):
            out.append(f"| {name} | {n} | {ms:.1f} | {100 * ms / tot:.3f} % |")
        return "\n".join(out) + "\n"
    for r in rows[rows.index(hdr) + 1:]:
        d = dict(zip(hdr, r))
        if "hx_sim_kernel" not in d.get("Kernel Name", ""):
            continue
        launches.add(d["ID"])
        vals.setdefault(d["Metric Name"], []).append(float(d["Metric Value"].replace(",", "")))
    n = len(launches)
    per = {k: sum(v) / n for k, v in vals.items()}
    line = json.loads(open(bench_json).read().strip().splitlines()[-1])
    ev = float(line["roofline"]["events_per_launch"])
    with open(KERNEL_SRC, "rb") as f:
        sha = hashlib.sha256(f.read()).hexdigest()
    out = [f"# ncu capture of hx_sim_kernel ({kind}), mean over {n} captured launch(es)",
           f"# workload: {line['config']['workload']}, {line['config']['sims']} simulations, "
           f"{int(ev)} simulated call events per launch",
           f"# command: {command}", f"kernel_sha256={sha}", f"sims_per_launch={line['config']['sims']}",
           f"events_per_launch={int(ev)}", f"kernel_ns={per.get('gpu__time_duration.sum', 0):.0f}"]
    if "dram__bytes_read.sum" in per:
        rd, wr = per["dram__bytes_read.sum"], per.get("dram__bytes_write.sum", 0.0)
        out += [f"dram_read_bytes_per_launch={rd:.0f}", f"dram_write_bytes_per_launch={wr:.0f}",
                f"dram_bytes_per_launch={rd + wr:.0f}"]
    if kind == "small" and "smsp__inst_executed.sum" in per:
        inst = per["smsp__inst_executed.sum"]
        out += [f"issue_active_frac={per['smsp__issue_active.sum'] / per['smsp__cycles_active.sum']:.4f}",
                f"warp_inst_per_event={inst / ev:.2f}",
                f"threads_per_inst={per['smsp__thread_inst_executed.sum'] / inst:.2f}"]
        for pipe in ("alu", "fma", "lsu", "cbu", "uniform", "adu", "xu"):
            k = f"sm__inst_executed_pipe_{pipe}.sum"
            if k in per:
                out.append(f"{pipe}_inst_per_event={per[k] / ev:.2f}")
        for op, name in (("branch", "branch"), ("shared_ld", "shared_load"), ("shared_st", "shared_store"),
                         ("global_ld", "global_load"), ("global_st", "global_store"), ("local_ld", "local_load")):
            k = f"sm__sass_inst_executed_op_{op}.sum"
            if k in per:
                out.append(f"{name}_inst_per_event={per[k] / ev:.2f}")
        for k, name in (("l1tex__t_sector_hit_rate.pct", "l1_hit_pct"), ("lts__t_sector_hit_rate.pct", "l2_hit_pct"),
                        ("smsp__warps_active.avg.per_cycle_active", "warps_active_per_scheduler")):
            if k in per:
                out.append(f"{name}={per[k]:.2f}")
    return "\n".join(out) + "\n"


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "sm_max_mhz": 2070.0}, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle samples during the timed region."""

    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if self.proc is None or not self.path:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 8:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        sm = [float(r[0]) for r in rows if r[0].replace(".", "").isdigit()]
        mx = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[4 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


def _barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# ------------------------------------------------------------------ oracle
# The CPU oracle as it stands, one simulation per job in a pool of worker
# processes (spawn), each job timing its own simulation on its core.  A
# worker builds only the traces its jobs need (one-trace workloads of the
# same recipe, same cut and same grid).
_ORACLE_ARGS = None
_ORACLE_CACHE = {}


def _oracle_init(args_dict):
    global _ORACLE_ARGS
    import oracle
    oracle.build()
    _ORACLE_ARGS = argparse.Namespace(**args_dict)


def _oracle_one(sim_trace_point):
    import oracle
    sim, t, p = sim_trace_point
    if t not in _ORACLE_CACHE:
        if len(_ORACLE_CACHE) >= 8:
            _ORACLE_CACHE.pop(next(iter(_ORACLE_CACHE)))
        a = argparse.Namespace(**vars(_ORACLE_ARGS))
        a.traces = 1
        _ORACLE_CACHE[t] = _workload(a, first_trace=t)
    wl = _ORACLE_CACHE[t]
    w0 = time.time()
    c0 = time.perf_counter()
    r = oracle.simulate(wl.traces[0], wl.cluster, oracle.point_of(wl.grid, p))
    return sim, time.perf_counter() - c0, w0, time.time(), int(r["events"]), int(r["status"])


def stratified_sims(wl, n: int, seed: int):
    """n simulations drawn evenly over the grid's alpha values (trace and the
    other axes at random, no repeats), or every simulation if n >= n_sims.
    Every recipe's grid gives each alpha value the same number of points, so
    an even draw per alpha value is proportional to the workload."""
    if n >= wl.n_sims:
        return list(range(wl.n_sims))
    g = wl.grid
    P, T = g.n_points, len(wl.traces)
    vals = np.unique(g.alpha_fp)
    rng = np.random.default_rng(seed)
    sims = []
    for i, a in enumerate(vals):
        pts = np.nonzero(g.alpha_fp == a)[0]
        k = n // len(vals) + (1 if i < n % len(vals) else 0)
        pick = rng.choice(T * pts.size, size=min(k, T * pts.size), replace=False)
        sims += (pick // pts.size * P + pts[pick % pts.size]).tolist()
    return sorted(sims)


def oracle_timed(args, wl, sims, procs: int, first_trace: int = 0):
    """Run the listed simulations of `wl` with the oracle; returns the number
    run, their completed calls, the sum of the per-simulation times (one
    core each) and the wall time from the first start to the last end."""
    import multiprocessing as mp
    P = wl.grid.n_points
    jobs = [(s, first_trace + s // P, s % P) for s in sims]
    jobs.sort(key=lambda j: j[1])  # neighbours share a trace in the workers' caches
    spec = {k: v for k, v in vars(args).items()}
    ctx = mp.get_context("spawn")
    with ctx.Pool(procs, initializer=_oracle_init, initargs=(spec,)) as pool:
        out = pool.map(_oracle_one, jobs, chunksize=1)
    if any(o[5] != 0 for o in out):
        raise RuntimeError("the oracle reported a failed simulation")
    core_s = sum(o[1] for o in out)
    wall = max(o[3] for o in out) - min(o[2] for o in out)
    return len(out), sum(o[4] for o in out), core_s, wall


def cpu_baseline(args, wl, n_sample: int):
    """The oracle on the host's cores: every simulation of the workload when
    n_sample >= n_sims, else n_sample drawn evenly over the alpha values.
    The single-core rate is the sample over the sum of its per-simulation
    times (each ran alone on one core); the all-core rate is the sample over
    the wall time of the pool."""
    procs = os.cpu_count() or 1
    sims = stratified_sims(wl, n_sample, 7)
    n, events, core_s, wall = oracle_timed(args, wl, sims, procs)
    whole = n == wl.n_sims
    what = (f"every simulation of {wl.name}" if whole else
            f"{n} of the {wl.n_sims} simulations of {wl.name}, {n // len(np.unique(wl.grid.alpha_fp))} per alpha "
            f"value (proportional to the grid); rates extrapolate to the whole workload as the sample's mean cost")
    return {"value": n / wall, "unit": UNIT, "cores": procs, "kind": "oracle", "events_per_s": events / wall,
            "sample": f"{what}; one simulation per job on {procs} processes, {wall:.1f} s wall",
            "single_core": {"value": n / core_s, "events_per_s": events / core_s,
                            "sample": f"the same {n} simulations, sum of their one-core times {core_s:.1f} s"},
            "sims": n, "whole_workload": whole}


def run_reference(args):
    world, rank, _ = D.env()
    if rank != 0:
        return
    wl = _workload(args)
    procs = os.cpu_count() or 1
    per_step = max(procs, 16)
    for w in range(args.warmup):
        oracle_timed(args, wl, stratified_sims(wl, max(2, procs // 4), 1000 + w), procs)
    t = 0.0
    n_tot = ev_tot = 0
    for k in range(args.steps):
        n, ev, _, dt = oracle_timed(args, wl, stratified_sims(wl, per_step, 2000 + k), procs)
        t += dt
        n_tot += n
        ev_tot += ev
    value = n_tot / t
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * t / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int64",
            "data": "synthetic", "stage_events_per_s": ev_tot / t,
            "config": {"workload": wl.name, "sims": wl.n_sims, "sample_sims_per_step": per_step,
                       "l2": "oracle on host cores"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": procs, "kind": "oracle",
                             "sample": f"{per_step} simulations per step drawn evenly over the alpha values, "
                                       f"one per job on {procs} processes"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_gpu(args):
    import torch
    world, rank, local = D.env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    else:
        torch.cuda.set_device(0)
    from paper_2505_05286_gb300 import build as B
    from paper_2505_05286_gb300 import hxsim as H
    B.build()
    # weak scaling: every rank simulates its own 256 traces (trace seeds offset by rank);
    # --traces / --queries cut the workload down for profiling captures
    r = _recipe(args.recipe)
    nt = args.traces or (W.RECIPES[r] if isinstance(r, int) else W.EXTRA[r]).n_traces
    wl = _workload(args, first_trace=D.first_trace(rank, nt))
    n_calls = wl.n_calls
    P = wl.grid.n_points
    sim = H.Sim(wl.traces, wl.cluster, wl.grid, timing=True)
    info = sim.info()
    stream = torch.cuda.current_stream()
    for _ in range(args.warmup):
        sim.run(stream)
    torch.cuda.synchronize()

    # kernel-only timing: inputs resident, K steps between events on the stream
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    _barrier(world)
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        start.record(stream)
        for _ in range(args.steps):
            sim.run(stream)
        stop.record(stream)
        torch.cuda.synchronize()
    _barrier(world)
    t_ms = start.elapsed_time(stop)
    # per-kernel times of every timed step (events the library records on the same stream)
    sim_ms = [sim.timings(back) for back in range(min(args.steps, 64))]
    t_ms = D.max_over_ranks(t_ms)
    res = sim.results()
    ok = bool((res["status"] == 0).all())
    events_per_step = int(res["events"].sum())
    sims_total = wl.n_sims * world
    value = sims_total * args.steps / (t_ms / 1000.0)
    events_rate = events_per_step * world * args.steps / (t_ms / 1000.0)
    # simulated events with the query arrivals too (a simulation that completes
    # has seen every query arrive, so arrivals = completed queries)
    arrivals_per_step = int(res["n_done"].sum())
    all_events_rate = (events_per_step + arrivals_per_step) * world * args.steps / (t_ms / 1000.0)
    # mean over the timed steps (each step's kernels lie inside that step, so the
    # mean never exceeds ms_per_step); the median beside it
    prep_ms = float(np.mean([x[0] for x in sim_ms]))
    kern_ms = float(np.mean([x[1] for x in sim_ms]))
    best_ms = float(np.mean([x[2] for x in sim_ms]))
    kern_ms_median = float(np.median([x[1] for x in sim_ms]))

    # end to end through the C ABI from pinned host buffers: upload, run, read back
    e2e_steps = 1
    fields = ("arrival_us", "k", "call_base", "prompt", "out", "out_est", "stage", "cand", "retry", "tenant")
    pin = lambda a: None if a is None else torch.from_numpy(np.ascontiguousarray(a)).pin_memory().numpy()
    pinned = [W.Trace(*[pin(getattr(t, f)) for f in fields]) for t in wl.traces]
    res_host = torch.empty(wl.n_sims * H.RESULT_DTYPE.itemsize, dtype=torch.uint8).pin_memory().numpy()
    res_host = res_host.view(H.RESULT_DTYPE)
    h2d = sum(getattr(t, f).nbytes for t in pinned for f in fields if getattr(t, f) is not None)
    d2h = wl.n_sims * H.RESULT_DTYPE.itemsize
    _barrier(world)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        sim.upload(pinned, stream)
        sim.run(stream)
        res2 = sim.results(out=res_host)
    torch.cuda.synchronize()
    e2e_s = D.max_over_ranks(time.perf_counter() - t0)
    e2e_same = bool((res2["digest"] == res["digest"]).all())
    e2e_value = sims_total * e2e_steps / e2e_s
    # best point of the whole job: per-point sums over every rank's traces
    sp, ss, sf = sim.point_sums()
    sp, ss, sf, nq_all = D.global_point_sums(sp, ss, sf, sum(t.n_queries for t in wl.traces))
    best = H.best_of_sums(sp, ss, sf, nq_all, wl.objective)

    peaks, peak_kind = _peaks()
    clocks = clk.summary()
    # Roofline of the dominant kernel (the simulation kernel): the SM issue
    # rate.  Algorithmic work per simulated call event: ~300 warp-instructions
    # (N = 64 instances over 32 lanes, one int64 division, score, argmax,
    # next-event minimum, queue and bookkeeping); peak: every scheduler of
    # every SM issuing one warp-instruction per cycle at the maximum SM clock.
    sm_count = torch.cuda.get_device_properties(0).multi_processor_count
    sm_mhz = float(peaks.get("sm_max_mhz", 2070.0))
    peak = sm_count * 4 * sm_mhz * 1e6
    n_inst = wl.cluster.n_inst
    achieved = WARP_INST_PER_EVENT * events_per_step / (kern_ms / 1000.0)
    roofline = {"bound": "alu", "achieved": achieved / 1e9, "peak": peak / 1e9, "unit": "Gwarp-inst/s",
                "frac": achieved / peak, "traffic": _traffic_per_launch(wl.n_sims) if _is_ceiling(args) else None,
                "work_per_event": WARP_INST_PER_EVENT, "events_per_launch": events_per_step,
                "kernel": "hx_sim_kernel" if info["generic_kernel"] else "hx_sim_kernel_lean", "kernel_ms": kern_ms,
                "peak_source": f"{sm_count} SMs x 4 schedulers x {sm_mhz:.0f} MHz ({peak_kind} sm_max_mhz)"}
    if _is_ceiling(args):
        # issue-slot use and executed instructions per event from the committed ncu capture
        kv = _ncu_figures()
        for key in ("issue_active_frac", "warp_inst_per_event", "threads_per_inst", "alu_inst_per_event",
                    "fma_inst_per_event", "lsu_inst_per_event", "branch_inst_per_event"):
            if key in kv:
                roofline["ncu_small_case_" + key] = float(kv[key])
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": t_ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "int64", "data": "synthetic",
            "stage_events_per_s": events_rate, "events_with_arrivals_per_s": all_events_rate, "all_sims_ok": ok, "e2e_same_results": e2e_same,
            "config": {"workload": wl.name, "traces": len(wl.traces), "queries_per_trace": wl.traces[0].n_queries,
                       "instances": n_inst, "points": P, "sims": wl.n_sims, "calls": n_calls,
                       "l2": (f"inputs larger than L2 ({n_calls * 64 / 2**30:.2f} GiB of call records)"
                              if n_calls * 64 > L2_BYTES else
                              f"inputs fit in L2 ({n_calls * 64 / 2**20:.1f} MiB of call records), not flushed"),
                       "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
                       "resident_warps": info["resident_warps"], "blocks": info["blocks"],
                       "work_order": WORK_ORDERS[info["work_order"]]},
            "kernels_ms": {"prep": prep_ms, "simulate": kern_ms, "best": best_ms, "simulate_median": kern_ms_median,
                           "over_steps": len(sim_ms)},
            "best_point": {"global_point": best[0], "sum_p95_us": best[1], "sum_slo_met": best[2]},
            "roofline": roofline, "clocks": clocks, "gpu_launches": 3 * args.steps,
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
                    "steps": e2e_steps}}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        n_sample = args.cpu_sample if args.cpu_sample else (wl.n_sims if wl.n_sims <= 8192 else 256)
        line["cpu_baseline"] = cpu_baseline(args, wl, n_sample)
    if rank == 0:
        print(json.dumps(line), flush=True)
    sim.close()
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-sample", type=int, default=0,
                    help="simulations the oracle runs for cpu_baseline (default: every one up to 8192, else 256 "
                         "drawn evenly over the alpha values)")
    ap.add_argument("--traces", type=int, default=None, help="cut the workload to this many traces (profiling)")
    ap.add_argument("--queries", type=int, default=None, help="cut each trace to this many queries (profiling)")
    ap.add_argument("--alpha", default="all", choices=["all", "1", "lt1"],
                    help="profiling: keep only the alpha = 1 grid points, or only the others")
    ap.add_argument("--recipe", default=str(CFG),
                    help="index of workloads.RECIPES or a key of workloads.EXTRA (default: the ceiling workload)")
    ap.add_argument("--policy", default="grid", choices=["grid"] + sorted(POLICIES),
                    help="one local-queue / dispatch policy on every grid point (default: the recipe's own)")
    ap.add_argument("--summarize-ncu", nargs=3, metavar=("CSV", "BENCH_JSON", "KIND"), default=None,
                    help="write the summary of an ncu CSV to stdout (KIND: ceiling or small: key=value figures of the "
                         "simulation kernel; launches: the launch list); --ncu-command gives the command")
    ap.add_argument("--ncu-command", default="")
    args = ap.parse_args()
    if args.summarize_ncu:
        csv_path, bench_json, kind = args.summarize_ncu
        sys.stdout.write(summarize_ncu(csv_path, bench_json, kind, args.ncu_command))
        return
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
