"""hx_sim_run_static: the entry point for callers that cannot allocate device
memory (its intermediates live in the library's fixed 64 MiB device array).
It must give exactly what the handle-based path gives, and what the oracle
gives, call after call; leave the handles' launches intact; and refuse a
trace whose intermediates do not fit.  Collected last on purpose."""
import numpy as np
import pytest

import oracle
from paper_2505_05286_gb300 import build as B
from paper_2505_05286_gb300 import hxsim as H
from paper_2505_05286_gb300 import workloads as W

FIELDS = ["p95_us", "makespan_us", "events", "digest", "slo_met", "n_done", "status"]


@pytest.mark.gpu
def test_static_matches_handle_path_twice():
    B.build()
    wl = W.make_workload(1, n_traces=1, n_queries=1000, first_trace=3)
    exact = oracle.run(wl, procs=8)
    for objective in (W.OBJ_P95, W.OBJ_P95_SLO95):
        sim = H.Sim(wl.traces, wl.cluster, wl.grid)
        sim.run()
        want = sim.results()
        wp, ws, wslo, _ = sim.best(objective)
        sim.close()
        op, osum, _ = oracle.best(exact, 1, wl.grid.n_points, [wl.traces[0].n_queries], objective)
        assert (op, osum) == (wp, ws)
        for _ in range(2):  # the second call reuses the array the first one left behind
            got, (gp, gs, gslo) = H.run_static(wl.traces[0], wl.cluster, wl.grid, objective)
            for f in FIELDS:
                assert np.array_equal(got[f], want[f]), f
                assert np.array_equal(got[f], exact[f]), f
            assert (gp, gs, gslo) == (wp, ws, wslo)


@pytest.mark.gpu
def test_static_call_between_runs_of_a_larger_handle():
    """A handle whose cluster needs more shared memory per block (fault
    windows add a flag per slot) still launches after a static call on a
    smaller cluster raised nothing: the kernel's shared-memory limit is only
    ever raised."""
    B.build()
    big = W.make_workload("faulty", n_traces=1, n_queries=600)
    small = W.make_workload(0, n_queries=120)
    g = small.grid  # FCFS on odd points: the static call runs the same (generic) kernel
    small.grid = W.Grid(g.alpha_fp, g.gamma_fp, g.rho, g.beta_us2,
                        (np.arange(g.n_points) % 2).astype(np.uint8) * W.POLICY_FCFS, g.dispatch_policy)
    sim = H.Sim(big.traces, big.cluster, big.grid)
    sim.run()
    first = sim.results()
    got, _ = H.run_static(small.traces[0], small.cluster, small.grid, W.OBJ_P95)
    sim.run()
    again = sim.results()
    sim.close()
    for f in FIELDS:
        assert np.array_equal(again[f], first[f]), f
    assert np.array_equal(got["digest"], oracle.run(small)["digest"])


@pytest.mark.gpu
@pytest.mark.parametrize("name,nq", [("competing-25", 300), ("faulty", 1400)])
def test_static_handles_tenants_single_shots_and_faults(name, nq):
    B.build()
    wl = W.make_workload(name, n_traces=1, n_queries=nq)
    sim = H.Sim(wl.traces, wl.cluster, wl.grid)
    sim.run()
    want = sim.results()
    sim.close()
    got, _ = H.run_static(wl.traces[0], wl.cluster, wl.grid, W.OBJ_P95)
    for f in FIELDS:
        assert np.array_equal(got[f], want[f]), f


def test_static_rejects_a_trace_that_does_not_fit():
    B.build()
    r = W.RECIPES[4]
    tr = W.make_trace(r, 4, 0, n_queries=30000)  # ~227k calls: > 64 MiB of intermediates
    with pytest.raises(H.HxError) as e:
        H.run_static(tr, W.make_cluster(r), W.subset_grid(W.make_grid(r), [0, 1]), stream=0)
    assert e.value.code == H.HX_ERR_INVALID and "too large for the static scratch" in str(e.value)
