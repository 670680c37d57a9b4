"""The bounds-checked build (libhxsim_checked.so, compiled with -DHX_CHECKED):
every index the simulation kernel forms is range-checked and a failed check
would stop the simulation with HX_ERR_BOUNDS.  On the hand cases, the random
workloads (both kernels) and the overload case it must raise no status and
give exactly the oracle's results."""
import numpy as np
import pytest

import oracle
from paper_2505_05286_gb300 import build as B
from paper_2505_05286_gb300 import hxsim as H
from paper_2505_05286_gb300 import workloads as W
from tests import cases
from tests.test_gpu_parity import FIELDS, NPROC, assert_extras, assert_logs, assert_same

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()
    H.load_checked()


def checked_sim(wl, **kw):
    sim = H.Sim(wl.traces, wl.cluster, wl.grid, bounds_checked=True, **kw)
    sim.run()
    return sim


@pytest.mark.parametrize("name", sorted(cases.load_golden("hand_cases.json")["cases"].keys()))
def test_hand_cases_checked(name):
    tr, cl, exp = cases.hand_case(name)
    wl = W.Workload(name, [tr], cl, cases.grid_from_points([exp["point"]]), W.OBJ_P95)
    sim = checked_sim(wl, record_sims=[0])
    r = sim.results()[0]
    assert r["status"] == H.HX_OK
    assert sim.records(0)["start"].tolist() == exp["start"]
    assert int(r["p95_us"]) == exp["p95_us"]
    sim.close()


@pytest.mark.parametrize("lean", [False, True])
@pytest.mark.parametrize("seed", range(24))
def test_random_workloads_checked(seed, lean):
    wl = cases.random_workload(seed, lean=lean)
    sim = checked_sim(wl, record_sims=[] if lean else [wl.n_sims - 1])
    assert sim.info()["generic_kernel"] == (0 if lean else 1)
    o, oe = oracle.run(wl, range(wl.n_sims), extra=True)
    g = sim.results()
    assert (g["status"] != H.HX_ERR_BOUNDS).all()
    assert_same(g, o, f"checked {wl.name}")
    if not lean:
        assert_extras(sim.extras(), oe, wl.name)
        assert_logs(sim, wl, 0)
    sim.close()


def test_overload_checked():
    """alpha near 1 on recipe 4: queues of thousands, heaps re-homed many
    times inside the arena."""
    wl = W.make_workload(4, n_traces=1, n_queries=3000)
    pts = list(range(1024 - 16, 1024)) + [0, 5, 300]
    wl.grid = W.subset_grid(wl.grid, pts)
    sim = checked_sim(wl)
    o = oracle.run(wl, range(wl.n_sims), procs=NPROC)
    assert_same(sim.results(), o, "overload checked")
    sim.close()


def test_small_arena_checked_reports_capacity_not_bounds():
    """An arena too small for the alpha = 1 queues still ends in
    HX_ERR_CAPACITY (the capacity check comes first), never HX_ERR_BOUNDS."""
    wl = W.make_workload(4, n_traces=1, n_queries=1500)
    wl.grid = W.subset_grid(wl.grid, list(range(1024 - 128, 1024, 16)) + [0, 64])
    sim = checked_sim(wl, arena_entries=1024)
    r = sim.results()
    assert (r["status"] != H.HX_ERR_BOUNDS).all() and (r["status"] == H.HX_ERR_CAPACITY).any()
    o = oracle.run(wl, range(wl.n_sims), procs=NPROC)
    ok = r["status"] == H.HX_OK
    for f in FIELDS:
        assert np.array_equal(r[f][ok], o[f][ok]), f
    sim.close()
