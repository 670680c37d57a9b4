"""Shared pieces of the online-tuning tests."""

import oracle
from paper_2505_05286_gb300 import tuner as T
from paper_2505_05286_gb300 import workloads as W


def oracle_backend(trace, cluster, grid):
    wl = W.Workload("window", [trace], cluster, grid, W.OBJ_P95)
    res = oracle.run(wl)
    _, log = oracle.simulate(trace, cluster, oracle.point_of(grid, 0), log=True)
    lat = log["end"][trace.call_base[1:] - 1] - trace.arrival_us
    return res, lat


def shift_scenario():
    """5 -> 20 -> 5 queries/s on the recipe-0 cluster (about 10 q/s of capacity),
    20-second windows."""
    tr = T.shift_trace([5.0, 20.0, 5.0], [60.0, 40.0, 60.0], recipe=0, seed=1)
    cl = W.make_cluster(W.RECIPES[0])
    return tr, cl, dict(window_us=20_000_000, min_queries=5, beta_us2=400_000 ** 2)
