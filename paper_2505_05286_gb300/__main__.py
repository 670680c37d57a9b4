"""Command line: simulate one of the seeded recipes on the GPU and print the
best hyper-parameter point (Sec. 4.3's argmin of P95).

    python -m paper_2505_05286_gb300 --recipe 1
    python -m paper_2505_05286_gb300 --recipe faulty --traces 2 --queries 500 --objective p95_slo95
"""
from __future__ import annotations

import argparse
import json
import time

from . import hxsim as H
from . import workloads as W


def main(argv=None) -> int:
    ap = argparse.ArgumentParser(prog="python -m paper_2505_05286_gb300")
    ap.add_argument("--recipe", default="0", help="index of workloads.RECIPES or a key of workloads.EXTRA")
    ap.add_argument("--traces", type=int, default=None, help="use this many traces of the recipe")
    ap.add_argument("--queries", type=int, default=None, help="cut each trace to this many queries")
    ap.add_argument("--objective", choices=["p95", "p95_slo95"], default=None,
                    help="default: the recipe's own objective")
    args = ap.parse_args(argv)
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
