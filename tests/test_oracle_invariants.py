"""Scheduler invariants of the oracle, re-derived from its per-call logs.

For each call the release time is rebuilt from the workflow of Sec. 2.1
(S at arrival; G_c after S; C_{c,r} after its predecessor in chain c; E after
the last call of every chain) and checked against the log:
  - dispatch happens at release and no call starts before it is released;
  - an instance never runs more calls than it has slots;
  - work conservation: while a call waits, its instance has no free slot;
  - each call runs exactly once for its service time;
  - P95, SLO count, makespan and the digest agree with the logged times.
"""
import numpy as np
import pytest

import oracle
from paper_2505_05286_gb300 import workloads as W


def _release_times(tr, end):
    rel = np.full(tr.n_calls, -1, np.int64)
    for i in range(tr.n_queries):
        b, e = int(tr.call_base[i]), int(tr.call_base[i + 1])
        rel[b] = tr.arrival_us[i]
        if tr.k[i] == 0:
            continue  # a single-shot request: one call, released on arrival
        last_of_chain = {}
        for j in range(b + 1, e - 1):
            c = int(tr.cand[j])
            if tr.stage[j] == W.STAGE_G:
                rel[j] = end[b]
            else:
                rel[j] = end[last_of_chain[c]]
            last_of_chain[c] = j
        rel[e - 1] = max(end[j] for j in last_of_chain.values())
    return rel


def _mix64(z):
    """The splitmix64 output function (Steele, Lea & Flood 2014), in Python
    integers, for the digest recomputed from a log."""
    m = (1 << 64) - 1
    z &= m
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & m
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & m
    return z ^ (z >> 31)


def _p95(lat):
    """Nearest-rank P95 of a latency list sorted here (0 for none)."""
    s = np.sort(np.asarray(lat, np.int64))
    return int(s[-(-95 * s.size // 100) - 1]) if s.size else 0


def _slowdown(cl, inst, start):
    """slow_fp of the first fault window covering each (instance, start), else 0."""
    slow = np.zeros(inst.shape[0], np.int64)
    hit = np.zeros(inst.shape[0], bool)
    if cl.faults is not None:
        for f in cl.faults:
            sel = ~hit & (inst == f["inst"]) & (start >= f["t0_us"]) & (start < f["t1_us"])
            slow[sel] = f["slow_fp"]
            hit |= sel
    return hit, slow


def check_schedule(tr, cl, res, log, reissued=0):
    """With re-issues the log keeps each call's last attempt only: the failed
    attempts' slot time and digest terms are not in it, so work conservation
    and the digest are checked only when nothing was re-issued."""
    p = oracle.prep(tr, cl)
    inst, enq, start, end = log["inst"], log["enq"], log["start"], log["end"]
    assert (inst >= 0).all() and (start >= 0).all()
    rel = _release_times(tr, end)
    if reissued:
        assert (enq >= rel).all()
    else:
        assert (enq == rel).all(), "dispatch must happen when the predecessors finish"
    assert (start >= enq).all()
    types = cl.inst_type[inst]
    svc = p["svc"][np.arange(tr.n_calls), types]
    hit, slow = _slowdown(cl, inst, start)
    assert (slow[hit] > 0).all(), "no attempt that finished started on a stopped instance"
    want = np.where(hit, -(-svc * slow // W.SCALE), svc)
    assert (end - start == want).all()
    for m in range(cl.n_inst):
        slots = int(cl.slots[cl.inst_type[m]])
        on = np.nonzero(inst == m)[0]
        if on.size == 0:
            continue
        times = np.unique(np.concatenate([start[on], end[on], enq[on]]))
        # running count after all events at time t
        running = np.array([np.sum((start[on] <= t) & (end[on] > t)) for t in times])
        assert running.max() <= slots
        if reissued:
            continue
        for c in on[start[on] > enq[on]]:
            sel = (times >= enq[c]) & (times < start[c])
            assert (running[sel] == slots).all(), "a call waited while a slot was free"
    lat = end[tr.call_base[1:] - 1] - tr.arrival_us
    n = tr.n_queries
    assert int(res["n_done"]) == n and int(res["events"]) == tr.n_calls
    if n:
        rank = -(-95 * n // 100)
        assert int(res["p95_us"]) == int(np.sort(lat)[rank - 1])
        assert int(res["slo_met"]) == int(np.sum(lat <= p["t_slo"]))
        assert int(res["makespan_us"]) == int(end.max())
    if reissued:
        return
    gold, m64 = 0x9E3779B97F4A7C15, (1 << 64) - 1

    def term(t, idtag):
        return _mix64(((t * gold) & m64) ^ idtag)

    dig = 0
    for c in range(tr.n_calls):
        dig += term(int(start[c]), (c << 8) | int(inst[c]))
    for i in range(n):
        dig += term(int(end[tr.call_base[i + 1] - 1]), (i << 8) | 0xFF)
    assert dig % (1 << 64) == int(res["digest"])


CASES = [
    (0, None, None, list(range(16))),
    (1, 1, 250, [0, 7, 9, 36, 63]),
    (2, 1, 200, [0, 5, 77, 130, 255]),
    (3, 1, 200, [0, 100, 300, 511]),
    (4, 1, 150, [0, 517, 1023]),
]


@pytest.mark.parametrize("cfg,nt,nq,points", CASES)
def test_invariants_pq_wb(cfg, nt, nq, points):
    wl = W.make_workload(cfg, n_traces=nt, n_queries=nq)
    tr = wl.traces[0]
    for p in points:
        res, log = oracle.simulate(tr, wl.cluster, oracle.point_of(wl.grid, p), check=True, log=True)
        assert res["status"] == 0
        check_schedule(tr, wl.cluster, res, log)


@pytest.mark.parametrize("local,dispatch", [(W.POLICY_FCFS, W.DISPATCH_WB), (W.POLICY_PQ, W.DISPATCH_RR),
                                            (W.POLICY_FCFS, W.DISPATCH_RR), (W.POLICY_LLF, W.DISPATCH_WB),
                                            (W.POLICY_LLF, W.DISPATCH_RR)])
def test_invariants_policies(local, dispatch):
    wl = W.make_workload(1, n_traces=1, n_queries=200)
    tr = wl.traces[0]
    for p in [0, 18, 63]:
        pt = oracle.point_of(wl.grid, p)
        pt["local_policy"], pt["dispatch_policy"] = local, dispatch
        res, log = oracle.simulate(tr, wl.cluster, pt, check=True, log=True)
        assert res["status"] == 0
        check_schedule(tr, wl.cluster, res, log)


def test_overloaded_queue():
    """alpha = 1 sends everything to the fastest instance: a long queue forms
    and the invariants still hold."""
    wl = W.make_workload(4, n_traces=1, n_queries=400)
    tr = wl.traces[0]
    pt = oracle.point_of(wl.grid, wl.grid.n_points - 1)
    res, log = oracle.simulate(tr, wl.cluster, pt, check=True, log=True)
    assert res["status"] == 0
    check_schedule(tr, wl.cluster, res, log)
    assert len(set(log["inst"].tolist())) == 1
    waits = log["start"] - log["enq"]
    assert waits.max() > 2 * 10 ** 6  # queued for more than 2 s


def test_empty_trace():
    wl = W.make_workload(0, n_queries=0)
    res = oracle.simulate(wl.traces[0], wl.cluster, oracle.point_of(wl.grid, 0), check=True)
    assert res["status"] == 0 and res["n_done"] == 0 and res["p95_us"] == 0 and res["digest"] == 0


def test_rejects_malformed():
    wl = W.make_workload(0, n_queries=5)
    tr = wl.traces[0]
    bad = W.Trace(*[getattr(tr, f).copy() for f in ("arrival_us", "k", "call_base", "prompt", "out",
                                                       "out_est", "stage", "cand", "retry")])
    bad.arrival_us[2] = bad.arrival_us[1] - 1  # unsorted
    assert oracle.simulate(bad, wl.cluster, oracle.point_of(wl.grid, 0))["status"] == 1
    bad2 = W.Trace(*[getattr(tr, f).copy() for f in ("arrival_us", "k", "call_base", "prompt", "out",
                                                        "out_est", "stage", "cand", "retry")])
    bad2.stage[1] = W.STAGE_E  # broken workflow structure
    assert oracle.simulate(bad2, wl.cluster, oracle.point_of(wl.grid, 0))["status"] == 1
    pt = oracle.point_of(wl.grid, 0)
    pt["alpha_fp"] = W.SCALE + 1
    assert oracle.simulate(tr, wl.cluster, pt)["status"] == 1


@pytest.mark.parametrize("name", ["paper-shaped", "noisy-estimate"])
def test_invariants_extra_recipes(name):
    wl = W.make_workload(name, n_traces=1, n_queries=120)
    tr = wl.traces[0]
    for p in [0, wl.grid.n_points // 2, wl.grid.n_points - 1]:
        res, log = oracle.simulate(tr, wl.cluster, oracle.point_of(wl.grid, p), check=True, log=True)
        assert res["status"] == 0
        check_schedule(tr, wl.cluster, res, log)


@pytest.mark.parametrize("name", ["two-tenant", "competing-25", "competing-50"])
def test_tenants_and_single_shots(name):
    """Per-tenant SLO counts add up and match each tenant's own T_slo; the
    single-shot requests (k = 0) run as one call released on arrival."""
    wl = W.make_workload(name, n_traces=1, n_queries=150)
    tr = wl.traces[0]
    p = oracle.prep(tr, wl.cluster)
    lat_ok = None
    for pt_i in [0, wl.grid.n_points // 2, wl.grid.n_points - 1]:
        res, log, ext = oracle.simulate(tr, wl.cluster, oracle.point_of(wl.grid, pt_i), check=True, log=True,
                                        extra=True)
        assert res["status"] == 0 and int(ext["reissued"]) == 0
        check_schedule(tr, wl.cluster, res, log)
        lat = log["end"][tr.call_base[1:] - 1] - tr.arrival_us
        for t in range(4):
            sel = tr.tenant == t
            assert int(ext["n_done"][t]) == int(sel.sum())
            assert int(ext["slo_met"][t]) == int(np.sum(lat[sel] <= p["t_slo"][sel]))
            assert int(ext["p95_us"][t]) == _p95(lat[sel])
        assert int(ext["slo_met"].sum()) == int(res["slo_met"])
    if name.startswith("competing"):
        single = tr.k == 0
        frac = float(name.split("-")[1]) / 100
        assert int(single.sum()) == int(np.floor(frac * (tr.n_calls - single.sum()) + 0.5))
        assert (tr.stage[tr.call_base[:-1][single]] == W.STAGE_E).all()
        assert (np.diff(tr.call_base)[single] == 1).all()
        assert (tr.tenant[single] == 1).all() and (tr.tenant[~single] == 0).all()


def test_equal_tenant_slos_change_nothing():
    """Tenants whose SLO multipliers all equal the cluster's give the one-tenant result."""
    wl = W.make_workload(1, n_traces=1, n_queries=200)
    tr = wl.traces[0]
    tr2 = W.Trace(*[getattr(tr, f) for f in ("arrival_us", "k", "call_base", "prompt", "out", "out_est",
                                             "stage", "cand", "retry")],
                  (np.arange(tr.n_queries) % 3).astype(np.uint8))
    cl = wl.cluster
    cl2 = W.Cluster(cl.prefill_tok_s, cl.decode_us_tok, cl.slots, cl.inst_type, cl.ref_type, cl.slo_mult_fp,
                    cl.rmax, cl.stage_ref_prompt, cl.stage_ref_out, np.full(3, cl.slo_mult_fp, np.int64))
    for p in [0, 30, 63]:
        a = oracle.simulate(tr, cl, oracle.point_of(wl.grid, p))
        b, ext = oracle.simulate(tr2, cl2, oracle.point_of(wl.grid, p), extra=True)
        assert a.tolist() == b.tolist()
        assert ext["n_done"].tolist()[:3] == [int(np.sum(tr2.tenant == t)) for t in range(3)]


def _with_faults(cl, faults, timeout_fp):
    f = np.zeros(len(faults), W.FAULT_DTYPE)
    for j, x in enumerate(faults):
        f[j] = (x[0], 0, x[1], x[2], x[3])
    return W.Cluster(cl.prefill_tok_s, cl.decode_us_tok, cl.slots, cl.inst_type, cl.ref_type, cl.slo_mult_fp,
                     cl.rmax, cl.stage_ref_prompt, cl.stage_ref_out, None, timeout_fp, f)


def test_neutral_faults_change_nothing():
    """An empty window, or a 1x slow-down without a timeout, is no fault."""
    wl = W.make_workload(1, n_traces=1, n_queries=200)
    tr, cl = wl.traces[0], wl.cluster
    for faults, to in (([(0, 5_000_000, 5_000_000, 0)], 3 * W.SCALE), ([(1, 0, 10 ** 9, W.SCALE)], 0)):
        cl2 = _with_faults(cl, faults, to)
        for p in [0, 40, 63]:
            a = oracle.simulate(tr, cl, oracle.point_of(wl.grid, p))
            b, ext = oracle.simulate(tr, cl2, oracle.point_of(wl.grid, p), extra=True)
            assert a.tolist() == b.tolist() and int(ext["reissued"]) == 0


@pytest.mark.parametrize("dispatch", [W.DISPATCH_WB, W.DISPATCH_RR])
def test_faulty_recipe_reissues(dispatch):
    """Timeouts on slow or stopped instances re-issue requests elsewhere; every
    call still completes once, and no finished attempt started on a stopped
    instance inside its window."""
    wl = W.make_workload("faulty", n_traces=1, n_queries=1400)
    tr = wl.traces[0]
    total = 0
    for p in [0, 33, 63]:
        pt = oracle.point_of(wl.grid, p)
        pt["dispatch_policy"] = dispatch
        res, log, ext = oracle.simulate(tr, wl.cluster, pt, check=True, log=True, extra=True)
        assert res["status"] == 0
        check_schedule(tr, wl.cluster, res, log, reissued=int(ext["reissued"]))
        total += int(ext["reissued"])
    assert total > 0


@pytest.mark.parametrize("lean", [False, True])
@pytest.mark.parametrize("seed", range(24))
def test_invariants_random_workloads(seed, lean):
    """Random clusters, traces (k from 0 to 8), tenants, fault windows and
    mixed policies (or, lean, the same shapes on WB + urgency queue alone):
    the schedule invariants and the per-tenant counts hold."""
    from tests import cases
    wl = cases.random_workload(seed, lean)
    tr = wl.traces[0]
    p = oracle.prep(tr, wl.cluster)
    for pt_i in range(wl.grid.n_points):
        res, log, ext = oracle.simulate(tr, wl.cluster, oracle.point_of(wl.grid, pt_i), check=True, log=True,
                                        extra=True)
        assert res["status"] == 0
        check_schedule(tr, wl.cluster, res, log, reissued=int(ext["reissued"]))
        lat = log["end"][tr.call_base[1:] - 1] - tr.arrival_us
        ten = tr.tenant if tr.tenant is not None else np.zeros(tr.n_queries, np.uint8)
        for t in range(4):
            sel = ten == t
            assert int(ext["n_done"][t]) == int(sel.sum())
            assert int(ext["slo_met"][t]) == int(np.sum(lat[sel] <= p["t_slo"][sel]))
            assert int(ext["p95_us"][t]) == _p95(lat[sel])
