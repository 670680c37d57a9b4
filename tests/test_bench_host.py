"""Host-side logic of bench.py: the workload options (recipe, cuts, policy
override) and when the committed DRAM-traffic figure applies."""
import argparse

import numpy as np

import bench
from paper_2505_05286_gb300 import workloads as W


def _args(**kw):
    base = dict(recipe=str(bench.CFG), traces=None, queries=None, alpha="all", policy="grid")
    base.update(kw)
    return argparse.Namespace(**base)


def test_policy_override_sets_every_point():
    for name, (lp, dp) in bench.POLICIES.items():
        wl = bench._workload(_args(recipe="0", queries=20, policy=name))
        assert (wl.grid.local_policy == lp).all() and (wl.grid.dispatch_policy == dp).all()
        ref = W.make_workload(0, n_queries=20)
        for f in ("alpha_fp", "gamma_fp", "rho", "beta_us2"):
            assert np.array_equal(getattr(wl.grid, f), getattr(ref.grid, f))
        assert name in wl.name


def test_extra_recipe_and_cuts():
    wl = bench._workload(_args(recipe="faulty", traces=3, queries=50))
    assert len(wl.traces) == 3 and wl.traces[0].n_queries >= 50 and wl.cluster.faults is not None
    a1 = bench._workload(_args(recipe="0", queries=20, alpha="1"))
    assert (a1.grid.alpha_fp == W.SCALE).all() and a1.grid.n_points == 4
    lt = bench._workload(_args(recipe="0", queries=20, alpha="lt1"))
    assert (lt.grid.alpha_fp < W.SCALE).all() and lt.grid.n_points == 12


def test_traffic_only_for_the_ceiling_workload():
    assert bench._is_ceiling(_args())
    for kw in (dict(recipe="3"), dict(traces=8), dict(queries=100), dict(alpha="1"), dict(policy="wb-pq")):
        assert not bench._is_ceiling(_args(**kw)), kw


def test_stratified_sample_is_even_over_alpha():
    wl = W.make_workload(3, n_traces=4, n_queries=10)
    sims = bench.stratified_sims(wl, 256, 7)
    assert len(sims) == len(set(sims)) == 256
    a = wl.grid.alpha_fp[np.asarray(sims) % wl.grid.n_points]
    vals, cnt = np.unique(a, return_counts=True)
    assert vals.size == 8 and (cnt == 32).all()
    assert len(set(np.asarray(sims) // wl.grid.n_points)) == 4
    assert bench.stratified_sims(wl, wl.n_sims, 7) == list(range(wl.n_sims))


def test_cpu_baseline_times_every_simulation_of_a_small_workload():
    args = _args(recipe="0", queries=30)
    wl = bench._workload(args)
    cb = bench.cpu_baseline(args, wl, wl.n_sims)
    assert cb["whole_workload"] and cb["sims"] == wl.n_sims and cb["kind"] == "oracle"
    assert cb["value"] > 0 and cb["single_core"]["value"] > 0
    assert abs(cb["events_per_s"] / cb["value"] - wl.traces[0].n_calls) < 1e-6 * wl.traces[0].n_calls
