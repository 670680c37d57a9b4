"""Row-by-row check of the GPU's complete result tables against the oracle.

The GPU half (`dump`) runs whole recipes through the library, in the
benchmark's launch configuration, and saves every simulation's result with
the SHA-256 of every input trace.  The CPU half (`check`) regenerates the
same traces (refusing any whose hash differs), recomputes the chosen rows
with the oracle in a pool of worker processes, and compares every field that
must be bit-exact.  Splitting the two lets the oracle take hours on a
machine without a GPU; `check` records its progress, so it can be resumed.

    python -m tests.full_tables dump DIR RECIPE [RECIPE ...]    # needs a GPU
    python -m tests.full_tables check DIR RECIPE [--traces A:B] [--procs N]

This is test infrastructure: it imports the oracle, and nothing in the
library imports it.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import multiprocessing as mp
import os
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2505_05286_gb300 import workloads as W  # noqa: E402

FIELDS = ["p95_us", "makespan_us", "events", "digest", "slo_met", "n_done", "status"]
TRACE_FIELDS = ("arrival_us", "k", "call_base", "prompt", "out", "out_est", "stage", "cand", "retry", "tenant")


def _recipe(arg):
    return int(arg) if str(arg).isdigit() else arg


def trace_sha(tr) -> str:
    h = hashlib.sha256()
    for f in TRACE_FIELDS:
        a = getattr(tr, f, None)
        if a is not None:
            h.update(f.encode())
            h.update(np.ascontiguousarray(a).tobytes())
    return h.hexdigest()


def table_sha(res) -> str:
    """SHA-256 of the bit-exact fields of a result table, row-major."""
    h = hashlib.sha256()
    for f in FIELDS:
        h.update(np.ascontiguousarray(res[f]).astype(res[f].dtype.newbyteorder("<")).tobytes())
    return h.hexdigest()


def dump(out_dir: str, recipe) -> dict:
    import torch

    from paper_2505_05286_gb300 import build as B
    from paper_2505_05286_gb300 import hxsim as H
    B.build()
    torch.cuda.set_device(0)
    wl = W.make_workload(_recipe(recipe))
    sim = H.Sim(wl.traces, wl.cluster, wl.grid, timing=True)
    t0 = time.perf_counter()
    sim.run(torch.cuda.current_stream())
    res = sim.results()
    wall = time.perf_counter() - t0
    prep_ms, sim_ms, best_ms = sim.timings()
    best = {str(obj): list(sim.best(obj)[:3]) for obj in (W.OBJ_P95, W.OBJ_P95_SLO95)}
    info = sim.info()
    sim.close()
    os.makedirs(out_dir, exist_ok=True)
    np.save(os.path.join(out_dir, f"table_{recipe}.npy"), res)
    meta = {"recipe": str(recipe), "workload": wl.name, "n_traces": len(wl.traces), "n_points": wl.grid.n_points,
            "n_sims": wl.n_sims, "n_calls": wl.n_calls, "table_sha256": table_sha(res),
            "trace_sha256": [trace_sha(t) for t in wl.traces], "all_ok": bool((res["status"] == 0).all()),
            "gpu": torch.cuda.get_device_name(0), "wall_s": wall, "kernels_ms": [prep_ms, sim_ms, best_ms],
            "resident_warps": info["resident_warps"], "generic_kernel": info["generic_kernel"], "best": best}
    with open(os.path.join(out_dir, f"table_{recipe}.json"), "w") as f:
        json.dump(meta, f, indent=1)
    return meta


# ----------------------------------------------------------------- CPU half
_WL = None


def _init_worker(recipe, traces):
    global _WL
    import oracle
    oracle.build()
    _WL = W.make_workload(_recipe(recipe), n_traces=traces)


def _one(sim: int):
    import oracle
    P = _WL.grid.n_points
    t0 = time.perf_counter()
    r = oracle.simulate(_WL.traces[sim // P], _WL.cluster, oracle.point_of(_WL.grid, sim % P))
    return sim, r, time.perf_counter() - t0


def check(out_dir: str, recipe, traces=None, procs=None, chunk: int = 2048) -> dict:
    import oracle
    oracle.build()
    meta = json.load(open(os.path.join(out_dir, f"table_{recipe}.json")))
    res = np.load(os.path.join(out_dir, f"table_{recipe}.npy"))
    assert table_sha(res) == meta["table_sha256"], "table file does not match its recorded hash"
    T, P = meta["n_traces"], meta["n_points"]
    a, b = (0, T) if traces is None else traces
    wl = W.make_workload(_recipe(recipe), n_traces=b)
    same = [trace_sha(wl.traces[t]) == meta["trace_sha256"][t] for t in range(a, b)]
    sims = [t * P + p for t in range(a, b) if same[t - a] for p in range(P)]
    prog_path = os.path.join(out_dir, f"check_{recipe}_{a}_{b}.progress.npy")
    done = np.load(prog_path) if os.path.exists(prog_path) else np.zeros(0, np.int64)
    done_set = set(done.tolist())
    todo = [s for s in sims if s not in done_set]
    procs = procs or os.cpu_count() or 1
    bad = []
    cpu_s = 0.0
    t_start = time.perf_counter()
    ctx = mp.get_context("spawn")
    with ctx.Pool(procs, initializer=_init_worker, initargs=(str(recipe), b)) as pool:
        for i in range(0, len(todo), chunk):
            part = todo[i:i + chunk]
            for sim, r, dt in pool.imap_unordered(_one, part, chunksize=4):
                cpu_s += dt
                for f in FIELDS:
                    if r[f] != res[f][sim]:
                        bad.append({"sim": int(sim), "field": f, "gpu": int(res[f][sim]), "oracle": int(r[f])})
                        break
            done = np.concatenate([done, np.asarray(part, np.int64)])
            np.save(prog_path, done)
            print(f"  {recipe}: {len(done)}/{len(sims)} rows, {len(bad)} mismatches, "
                  f"{time.perf_counter() - t_start:.0f} s", flush=True)
    summary = {"recipe": str(recipe), "workload": meta["workload"], "traces": [a, b],
               "traces_skipped_hash_differs": [a + i for i, s in enumerate(same) if not s],
               "rows_checked": int(len(done)), "rows_in_table": int(meta["n_sims"]), "mismatches": len(bad),
               "first_mismatches": bad[:16], "table_sha256": meta["table_sha256"],
               "oracle_wall_s_this_pass": time.perf_counter() - t_start, "oracle_cpu_s_this_pass": cpu_s,
               "procs": procs, "gpu_table_from": meta["gpu"]}
    with open(os.path.join(out_dir, f"check_{recipe}_{a}_{b}.json"), "w") as f:
        json.dump(summary, f, indent=1)
    return summary


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("mode", choices=["dump", "check"])
    ap.add_argument("dir")
    ap.add_argument("recipes", nargs="+")
    ap.add_argument("--traces", default=None, help="check only traces A:B")
    ap.add_argument("--procs", type=int, default=None)
    args = ap.parse_args(argv)
    for r in args.recipes:
        if args.mode == "dump":
            m = dump(args.dir, r)
            print(json.dumps({k: m[k] for k in ("recipe", "workload", "n_sims", "table_sha256", "all_ok", "wall_s")}),
                  flush=True)
        else:
            tr = None if args.traces is None else tuple(int(x) for x in args.traces.split(":"))
            s = check(args.dir, r, tr, args.procs)
            print(json.dumps({k: v for k, v in s.items() if k != "first_mismatches"}), flush=True)
            if s["mismatches"]:
                print(json.dumps(s["first_mismatches"]), flush=True)
                return 1
    return 0


if __name__ == "__main__":
    sys.exit(main())
