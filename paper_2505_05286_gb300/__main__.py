"""Command line: simulate one of the seeded recipes on the GPU and print the
best hyper-parameter point (Sec. 4.3's argmin of P95), or run the online
alpha-tuning loop of Sec. 4.3 on a trace whose load shifts and print one line
per window with the wall time of each triggered sweep (Table 3's overhead).

    python -m paper_2505_05286_gb300 --recipe 1
    python -m paper_2505_05286_gb300 --recipe faulty --traces 2 --queries 500 --objective p95_slo95
    python -m paper_2505_05286_gb300 --tune 5,20,5 --seconds 60,40,60 --window-s 20
    python -m paper_2505_05286_gb300 --recipe 4 --tune 20,30,20 --seconds 1500 --window-s 300 --time-sweeps
"""
from __future__ import annotations

import argparse
import json
import time

from . import hxsim as H
from . import workloads as W


def _floats(s: str):
    return [float(x) for x in s.split(",") if x]


def tune(args) -> int:
    """Online tuning on a shifting-load trace of recipe `args.recipe`: one
    JSON line per window, then a summary of the sweeps' wall times."""
    from . import tuner as T
    recipe = int(args.recipe)
    rates, secs = _floats(args.tune), _floats(args.seconds)
    if len(secs) == 1:
        secs = secs * len(rates)
    if len(secs) != len(rates):
        raise SystemExit("--seconds needs one value or one per rate")
    r = W.RECIPES[recipe]
    tr = T.shift_trace(rates, secs, recipe=recipe, seed=args.seed)
    cl = W.make_cluster(r)
    tuner = T.OnlineTuner(cl, backend=T.gpu_backend, window_us=int(args.window_s * 1e6), min_queries=5,
                          beta_us2=r.c_ref_us ** 2)
    T.gpu_backend(T.slice_queries(tr, 0, min(tr.n_queries, 8)), cl, tuner.grid_of([0]))  # load + first-use costs
    reps = tuner.run(tr)
    # --time-sweeps: the wall time of a sweep on every window, triggered or
    # not, over the alpha values and over the recipe's whole grid
    sweep_ms, grid_ms = [], []
    if args.time_sweeps:
        full = W.make_grid(r)
        for i0, i1 in T.windows(tr, tuner.window_us, tuner.min_queries):
            win = T.slice_queries(tr, i0, i1)
            t0 = time.perf_counter()
            T.gpu_backend(win, cl, tuner.grid_of(tuner.alphas))
            sweep_ms.append(1000 * (time.perf_counter() - t0))
            t0 = time.perf_counter()
            sim = H.Sim([win], cl, full)
            sim.run()
            sim.results()
            sim.close()
            grid_ms.append(1000 * (time.perf_counter() - t0))
    for j, rep in enumerate(reps):
        line = {"window": rep.index, "t0_s": rep.t0_us / 1e6, "queries": rep.n_queries,
                "alpha": rep.alpha_fp / W.SCALE, "p95_us": rep.p95_us, "p_value": rep.p_value,
                "triggered": rep.triggered, "new_alpha": rep.new_alpha_fp / W.SCALE,
                "tune_ms": round(rep.tune_ms, 3) if rep.triggered else None}
        if sweep_ms:
            line.update(sweep_ms=round(sweep_ms[j], 3), grid_sweep_ms=round(grid_ms[j], 3))
        print(json.dumps(line))
    ms = [rep.tune_ms for rep in reps if rep.triggered]
    mean = lambda x: round(sum(x) / len(x), 3) if x else None
    top = lambda x: round(max(x), 3) if x else None
    summary = {"recipe": r.name, "rates_qps": rates, "seconds": secs, "queries": tr.n_queries,
               "windows": len(reps), "tunings": len(ms), "alphas_per_sweep": len(tuner.alphas),
               "tune_ms_mean": mean(ms), "tune_ms_max": top(ms)}
    if sweep_ms:
        summary.update(sweep_ms_mean=mean(sweep_ms), sweep_ms_max=top(sweep_ms), grid_points=int(full.n_points),
                       grid_sweep_ms_mean=mean(grid_ms), grid_sweep_ms_max=top(grid_ms))
    print(json.dumps(summary))
    return 0


def main(argv=None) -> int:
    ap = argparse.ArgumentParser(prog="python -m paper_2505_05286_gb300")
    ap.add_argument("--recipe", default="0", help="index of workloads.RECIPES or a key of workloads.EXTRA")
    ap.add_argument("--traces", type=int, default=None, help="use this many traces of the recipe")
    ap.add_argument("--queries", type=int, default=None, help="cut each trace to this many queries")
    ap.add_argument("--objective", choices=["p95", "p95_slo95"], default=None,
                    help="default: the recipe's own objective")
    ap.add_argument("--tune", default=None, metavar="RATES",
                    help="online tuning on a trace whose Poisson rate steps through RATES (q/s, comma-separated)")
    ap.add_argument("--seconds", default="60", help="--tune: seconds per rate (one value or one per rate)")
    ap.add_argument("--window-s", type=float, default=20.0, help="--tune: window length in seconds")
    ap.add_argument("--seed", type=int, default=1, help="--tune: trace seed")
    ap.add_argument("--time-sweeps", action="store_true",
                    help="--tune: also time an alpha sweep and a whole-grid sweep on every window")
    args = ap.parse_args(argv)
    if args.tune is not None:
        return tune(args)
    import torch

    recipe = int(args.recipe) if args.recipe.isdigit() else args.recipe
    wl = W.make_workload(recipe, n_traces=args.traces, n_queries=args.queries)
    obj = wl.objective if args.objective is None else (W.OBJ_P95 if args.objective == "p95" else W.OBJ_P95_SLO95)
    sim = H.Sim(wl.traces, wl.cluster, wl.grid, timing=True)
    t0 = time.perf_counter()
    sim.run(torch.cuda.current_stream())
    res = sim.results()
    wall = time.perf_counter() - t0
    point, sum_p95, slo, per_trace = sim.best(obj)
    g = wl.grid
    out = {
        "workload": wl.name, "simulations": wl.n_sims, "failed": int((res["status"] != 0).sum()),
        "simulate_ms": round(sim.timings()[1], 3), "wall_s": round(wall, 3),
        "best_point": point, "sum_p95_us": sum_p95, "sum_slo_met": slo,
        "alpha": int(g.alpha_fp[point]) / W.SCALE if point >= 0 else None,
        "gamma": int(g.gamma_fp[point]) / W.SCALE if point >= 0 else None,
        "rho": int(g.rho[point]) if point >= 0 else None,
        "beta_us2": int(g.beta_us2[point]) if point >= 0 else None,
        "per_trace_point": per_trace.tolist(),
    }
    print(json.dumps(out))
    sim.close()
    return 0


if __name__ == "__main__":
    raise SystemExit(main())
