"""Pins of the CPU oracle against facts fixed outside the oracle itself:
hand-worked schedules, the paper's worked examples (Table 2, Fig. 3), closed
forms and the special cases the paper states for Eq. (score)."""
import numpy as np
import pytest

import oracle
from paper_2505_05286_gb300 import workloads as W
from tests import cases

HAND = sorted(cases.load_golden("hand_cases.json")["cases"].keys())


@pytest.mark.parametrize("name", HAND)
def test_hand_case(name):
    tr, cl, exp = cases.hand_case(name)
    res, log, ext = oracle.simulate(tr, cl, exp["point"], check=True, log=True, extra=True)
    assert res["status"] == 0
    assert log["inst"].tolist() == exp["inst"]
    assert log["start"].tolist() == exp["start"]
    if "budget" in exp:
        assert log["budget"].tolist() == exp["budget"]
    ends_e = log["end"][tr.call_base[1:] - 1]
    assert (ends_e - tr.arrival_us).tolist() == exp["latency"]
    assert int(res["p95_us"]) == exp["p95_us"]
    assert int(res["slo_met"]) == exp["slo_met"]
    assert int(res["makespan_us"]) == exp["makespan_us"]
    assert int(res["n_done"]) == tr.n_queries
    assert int(res["events"]) == tr.n_calls
    if "tenant_slo_met" in exp:
        assert ext["slo_met"].tolist() == exp["tenant_slo_met"]
        assert ext["n_done"].tolist() == exp["tenant_done"]
        assert int(ext["reissued"]) == exp["reissued"]
    if "tenant_p95_us" in exp:
        assert ext["p95_us"].tolist() == exp["tenant_p95_us"]


def test_table2_pick():
    """Table 2 / Sec. 5.3: PQ starts request 6 (urgency 26.9), FCFS request 1."""
    g = cases.load_golden("table2_queue.json")
    rid = g["request_id"]
    urg = [round(u * 10) for u in g["urgency"]]  # 0.1 resolution is exact in integers
    enq = [round(a * 1e6) for a in g["arrive_at_s"]]
    assert rid[oracle.pick(0, rid, urg, enq)] == g["pq_pick"]
    assert rid[oracle.pick(1, rid, urg, enq)] == g["fcfs_pick"]
    # without requests 6 and 7 the two 19.0 urgencies tie: the lower id (3) wins
    assert rid[oracle.pick(0, rid[:5], urg[:5], enq[:5])] == 3
    # order of presentation does not matter
    perm = [6, 2, 0, 5, 3, 1, 4]
    assert [rid[i] for i in perm][oracle.pick(0, [rid[i] for i in perm], [urg[i] for i in perm],
                                              [enq[i] for i in perm])] == g["pq_pick"]


def test_fig3_budget_debit():
    """Fig. 3: q_i1 is budgeted 40 ms but takes 50 ms; the 10 ms debit tightens q_i2."""
    t_slo = 100_000
    t1, t2 = 40_000, 60_000
    assert oracle.budget(t_slo, 0, t1, t1 + t2) == 40_000
    on_time = oracle.budget(t_slo, 40_000, t2, t2)
    late = oracle.budget(t_slo, 50_000, t2, t2)
    assert on_time == 60_000 and late == 50_000 and on_time - late == 10_000


def test_budget_truncates_toward_zero():
    assert oracle.budget(3000, 4000, 2000, 6000) == -333
    assert oracle.budget(3000, 2000, 2000, 6000) == 333
    assert oracle.budget(0, 0, 5, 7) == 0


def test_score_special_cases():
    """Sec. 4.1: alpha = 1 keeps only the computation cost, alpha = 0 only the
    queue term beta / t_queue; an empty queue counts as t_queue = 1."""
    beta = 9_000_000
    for q, comp in [(0, 2000), (5000, 2000), (123, 99999)]:
        assert oracle.score(W.SCALE, beta, q, comp) == -W.SCALE * comp
    assert oracle.score(0, beta, 0, 2000) == W.SCALE * beta
    assert oracle.score(0, beta, 1, 2000) == W.SCALE * beta
    assert oracle.score(0, beta, 2000, 7) == W.SCALE * 4500
    assert oracle.score(0, beta, 7, 1) == W.SCALE * (beta // 7)
    assert oracle.score(0, 1 << 50, 1, 1) == W.SCALE * ((1 << 43) - 1)  # reward cap
    # (1 - a) * beta / q - a * comp at a = 1/2: 0.5 * 4500 - 0.5 * 2000
    assert oracle.score(W.SCALE // 2, beta, 2000, 2000) == 1_250_000_000


@pytest.mark.parametrize("n", [1, 2, 3, 4, 20, 200])
def test_closed_form_fcfs_burst(n):
    """One instance, one slot, FCFS, k = 1, no corrections, every call s us, all
    n queries at t = 0: all S first, then all G, then all E, so query j
    finishes at (2n + j + 1) s and P95 = (2n + ceil(0.95 n)) s."""
    s = 1000
    tr, cl = cases.uniform_single_instance(n, [0] * n, svc_us=s)
    pt = dict(alpha_fp=W.SCALE // 2, gamma_fp=W.SCALE, beta_us2=10 ** 6, rho=0, local_policy=1,
              dispatch_policy=0)
    res, log = oracle.simulate(tr, cl, pt, check=True, log=True)
    assert res["status"] == 0
    lat = (log["end"][tr.call_base[1:] - 1] - tr.arrival_us).tolist()
    assert lat == [(2 * n + j + 1) * s for j in range(n)]
    rank = -(-95 * n // 100)
    assert int(res["p95_us"]) == (2 * n + rank) * s
    # T_slo = 3 * (3 s): met iff 2n + j + 1 <= 9
    assert int(res["slo_met"]) == sum(1 for j in range(n) if 2 * n + j + 1 <= 9)


@pytest.mark.parametrize("n,n_tenants", [(1, 2), (5, 2), (40, 2), (41, 3), (200, 4)])
def test_closed_form_fcfs_burst_per_tenant(n, n_tenants):
    """The burst above with query j in tenant j mod n_tenants: tenant t holds
    queries j = t, t + n_tenants, ... in latency order, so its P95 is the
    latency (2n + j + 1) s of its ceil(0.95 n_t)-th query, and a tenant
    without queries reports 0; SLO counts split the same way."""
    s = 1000
    tr, cl1 = cases.uniform_single_instance(n, [0] * n, svc_us=s)
    tr.tenant = (np.arange(n) % n_tenants).astype(np.uint8)
    mult = np.full(n_tenants, 3 * W.SCALE, np.int64)
    cl = W.Cluster(cl1.prefill_tok_s, cl1.decode_us_tok, cl1.slots, cl1.inst_type, cl1.ref_type, cl1.slo_mult_fp,
                   cl1.rmax, cl1.stage_ref_prompt, cl1.stage_ref_out, mult)
    pt = dict(alpha_fp=W.SCALE // 2, gamma_fp=W.SCALE, beta_us2=10 ** 6, rho=0, local_policy=1,
              dispatch_policy=0)
    res, ext = oracle.simulate(tr, cl, pt, check=True, extra=True)
    assert res["status"] == 0
    for t in range(4):
        js = [j for j in range(n) if j % n_tenants == t] if t < n_tenants else []
        if not js:
            assert int(ext["p95_us"][t]) == 0 and int(ext["n_done"][t]) == 0
            continue
        j = js[-(-95 * len(js) // 100) - 1]
        assert int(ext["p95_us"][t]) == (2 * n + j + 1) * s
        assert int(ext["n_done"][t]) == len(js)
        assert int(ext["slo_met"][t]) == sum(1 for q in js if 2 * n + q + 1 <= 9)
    # with one tenant the tenant's P95 is the simulation's
    tr.tenant = None
    res1, ext1 = oracle.simulate(tr, cl1, pt, extra=True)
    assert int(ext1["p95_us"][0]) == int(res1["p95_us"]) and ext1["p95_us"][1:].tolist() == [0, 0, 0]


@pytest.mark.parametrize("policy", [0, 1])
def test_closed_form_spaced(policy):
    """Arrivals >= 3 s apart on one instance never queue: every latency is 3 s."""
    s = 1000
    n = 25
    gaps = [3 * s + (j * 7) % 5 for j in range(n)]
    tr, cl = cases.uniform_single_instance(n, np.cumsum(gaps) - gaps[0], svc_us=s)
    pt = dict(alpha_fp=0, gamma_fp=W.SCALE, beta_us2=10 ** 6, rho=0, local_policy=policy,
              dispatch_policy=0)
    res, log = oracle.simulate(tr, cl, pt, check=True, log=True)
    lat = log["end"][tr.call_base[1:] - 1] - tr.arrival_us
    assert (lat == 3 * s).all()
    assert int(res["p95_us"]) == 3 * s and int(res["slo_met"]) == n


def test_p95_nearest_rank():
    """P95 of latencies 1..n (in units of s) is ceil(0.95 n): spaced single-call
    queries whose service times are 1..n units."""
    for n in [1, 3, 19, 20, 21, 99, 100, 101]:
        q = [{"arrival": 10 ** 7 * i, "k": 1,
              "calls": [["S", 0, 0, 1, 0, 0], ["G", 0, 0, 1, 0, 0], ["E", 0, 0, 1, (i * 37) % n + 1, 0]]}
             for i in range(n)]
        tr = cases.trace_from({"queries": q})
        # prefill 1e6 tok/s: a 1-token prompt costs 1 us; decode 1000 us per output token
        cl = W.Cluster(np.array([1_000_000], np.int32), np.array([1000], np.int32), np.array([1], np.int32),
                       np.array([0], np.uint8), 0, W.SCALE, 0, np.ones(4, np.int32), np.zeros(4, np.int32))
        pt = dict(alpha_fp=0, gamma_fp=W.SCALE, beta_us2=1, rho=0, local_policy=0, dispatch_policy=0)
        res = oracle.simulate(tr, cl, pt, check=True)
        assert sorted((i * 37) % n + 1 for i in range(n)) == list(range(1, n + 1))
        rank = -(-95 * n // 100)
        assert int(res["p95_us"]) == 3 + 1000 * rank


def test_alpha1_homogeneous_all_on_lowest_index():
    """alpha = 1 on identical instances: every score ties, the lowest index wins."""
    wl = W.make_workload(0, n_queries=60)
    cl = wl.cluster
    cl = W.Cluster(cl.prefill_tok_s[:1], cl.decode_us_tok[:1], cl.slots[:1], np.zeros(4, np.uint8), 0,
                   cl.slo_mult_fp, cl.rmax, cl.stage_ref_prompt, cl.stage_ref_out)
    pt = oracle.point_of(wl.grid, wl.grid.n_points - 1)
    assert pt["alpha_fp"] == W.SCALE
    res, log = oracle.simulate(wl.traces[0], cl, pt, check=True, log=True)
    assert res["status"] == 0 and (log["inst"] == 0).all()


def test_alpha1_picks_fastest_type():
    """alpha = 1 on the two-type cluster of recipe 0: type A (12000 tok/s,
    15 us/tok) is faster for every call, so only instance 0 is used."""
    wl = W.make_workload(0, n_queries=40)
    pt = oracle.point_of(wl.grid, wl.grid.n_points - 1)
    res, log = oracle.simulate(wl.traces[0], wl.cluster, pt, check=True, log=True)
    assert res["status"] == 0 and (log["inst"] == 0).all()


def test_round_robin_balanced():
    wl = W.make_workload(1, n_traces=1, n_queries=100)
    pt = oracle.point_of(wl.grid, 3)
    pt["dispatch_policy"] = W.DISPATCH_RR
    res, log = oracle.simulate(wl.traces[0], wl.cluster, pt, check=True, log=True)
    counts = np.bincount(log["inst"], minlength=wl.cluster.n_inst)
    assert res["status"] == 0 and counts.max() - counts.min() <= 1


def test_prep_closed_forms():
    """Eq. (comp), its mean over instances, the stage reference costs and the
    SLO (a multiple of S + slowest chain + E on the reference type)."""
    g = cases.load_golden("hand_cases.json")
    tr = cases.trace_from(g["traces"]["one_query_two_chains"])
    cl = cases.cluster_from(g["clusters"]["two_inst"], 3 * W.SCALE)
    cl = W.Cluster(cl.prefill_tok_s, cl.decode_us_tok, cl.slots, cl.inst_type, cl.ref_type, cl.slo_mult_fp, 2,
                   cl.stage_ref_prompt, cl.stage_ref_out)
    p = oracle.prep(tr, cl)
    assert (p["est"] == [[2000, 4000]] * 6).all() and (p["svc"] == p["est"]).all()
    assert (p["tbar"] == 3000).all() and (p["stage_ref_cost"] == 3000).all()
    assert p["t_slo"].tolist() == [3 * (2000 + 3 * 2000 + 2000)]
    # ceil on the prefill term: 1 token at 3 tok/s = 333333.33 us -> 333334
    cl3 = W.Cluster(np.array([3, 7], np.int32), np.array([5, 0], np.int32), np.array([1, 1], np.int32),
                    np.array([0, 1, 1], np.uint8), 1, 2 * W.SCALE, 2, np.ones(4, np.int32), np.zeros(4, np.int32))
    p3 = oracle.prep(tr, cl3)
    assert p3["est"][0].tolist() == [333334 + 5, 142858]
    assert p3["tbar"][0] == (333339 + 2 * 142858) // 3
    # out (true) 1 token vs out_est 1 token: same here; change out_est
    tr.out_est[:] = 4
    p4 = oracle.prep(tr, cl3)
    assert p4["est"][0].tolist() == [333334 + 20, 142858] and p4["svc"][0].tolist() == [333339, 142858]
    assert p4["t_slo"][0] == 2 * 5 * 142858  # S + three-call chain 0 + E on type 1


def test_best_point_rules():
    """Sec. 4.3 argmin of P95 over the grid; ties to the lower point index;
    the constrained objective keeps points with >= 95% SLO attainment."""
    R = oracle.RESULT_DTYPE
    res = np.zeros(6, R)  # 2 traces x 3 points
    res["p95_us"] = [50, 40, 40, 10, 30, 30]
    res["slo_met"] = [100, 94, 100, 95, 96, 100]
    res["n_done"] = 100
    gp, gs, per = oracle.best(res, 2, 3, [100, 100], W.OBJ_P95)
    assert per.tolist() == [1, 0] and gp == 0 and gs == 60
    gp, gs, per = oracle.best(res, 2, 3, [100, 100], W.OBJ_P95_SLO95)
    # trace 0: points 0 and 2 feasible -> p95 40 at point 2; trace 1: all feasible -> point 0
    assert per.tolist() == [2, 0]
    # global sums: p0 (60, slo 195) p1 (70, slo 190 = exactly 95%) p2 (70, slo 200)
    assert gp == 0 and gs == 60
    res["slo_met"] = [10, 20, 20, 10, 10, 5]  # nothing feasible: most SLO hits, then P95
    gp, gs, per = oracle.best(res, 2, 3, [100, 100], W.OBJ_P95_SLO95)
    assert per.tolist() == [1, 0] and gp == 1
    res["status"][1] = 2  # a failed simulation never wins
    gp, gs, per = oracle.best(res, 2, 3, [100, 100], W.OBJ_P95)
    assert per.tolist() == [2, 0] and gp == 0


@pytest.mark.parametrize("alpha_index", [1, 3, 5])
def test_wb_moves_work_to_fast_instances(alpha_index):
    """Table 1 / Sec. 5.3, qualitatively: round robin spreads every stage over
    the instances evenly, while workload-balanced dispatch sends a larger share
    of each stage to the fastest instance type and a smaller one to the
    slowest (recipe 1: 4 A, 2 B = slowest, 2 C = fastest)."""
    wl = W.make_workload(1, n_traces=1, n_queries=500)
    tr, cl = wl.traces[0], wl.cluster
    pt = oracle.point_of(wl.grid, alpha_index * 8 + 3)
    assert 0 < pt["alpha_fp"] < W.SCALE
    rr = dict(pt, dispatch_policy=W.DISPATCH_RR)
    _, wb_log = oracle.simulate(tr, cl, pt, log=True)
    _, rr_log = oracle.simulate(tr, cl, rr, log=True)
    inst_share = np.bincount(cl.inst_type, minlength=3) / cl.n_inst
    fast, slow = 2, 1
    for st in range(4):
        sel = tr.stage == st
        wb = np.bincount(cl.inst_type[wb_log["inst"][sel]], minlength=3) / sel.sum()
        rrs = np.bincount(cl.inst_type[rr_log["inst"][sel]], minlength=3) / sel.sum()
        assert np.abs(rrs - inst_share).max() < 0.05, (st, rrs)
        assert wb[fast] > rrs[fast] + 0.1 and wb[slow] < rrs[slow] - 0.1, (st, wb, rrs)
