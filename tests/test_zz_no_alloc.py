"""hx_sim_run_static: the entry point for callers that cannot allocate device
memory (its intermediates live in the library's fixed 64 MiB device array).
It must give exactly what the handle-based path gives, call after call, and
refuse a trace whose intermediates do not fit.  Collected last on purpose."""
import numpy as np
import pytest

from paper_2505_05286_gb300 import build as B
from paper_2505_05286_gb300 import hxsim as H
from paper_2505_05286_gb300 import workloads as W

FIELDS = ["p95_us", "makespan_us", "events", "digest", "slo_met", "n_done", "status"]


@pytest.mark.gpu
def test_static_matches_handle_path_twice():
    B.build()
    wl = W.make_workload(1, n_traces=1, n_queries=1000, first_trace=3)
    for objective in (W.OBJ_P95, W.OBJ_P95_SLO95):
        sim = H.Sim(wl.traces, wl.cluster, wl.grid)
        sim.run()
        want = sim.results()
        wp, ws, wslo, _ = sim.best(objective)
        sim.close()
        for _ in range(2):  # the second call reuses the array the first one left behind
            got, (gp, gs, gslo) = H.run_static(wl.traces[0], wl.cluster, wl.grid, objective)
            for f in FIELDS:
                assert np.array_equal(got[f], want[f]), f
            assert (gp, gs, gslo) == (wp, ws, wslo)


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
