"""CUDA path vs the CPU oracle, bit for bit, through the C ABI.

Everything here is integer work, so the bar is exact equality: per-call
instance, dispatch time, SLO budget and start time (full logs), and per
simulation P95, makespan, completed calls, digest, SLO count and status; the
best points of Sec. 4.3 likewise.  Small cases compare every simulation;
the full-size workloads compare a seeded sample of simulations plus
properties that hold at any size.
"""
import os

import numpy as np
import pytest

import oracle
from paper_2505_05286_gb300 import build as B
from paper_2505_05286_gb300 import hxsim as H
from paper_2505_05286_gb300 import workloads as W
from tests import cases

pytestmark = pytest.mark.gpu

NPROC = max(1, min(16, os.cpu_count() or 1))
FIELDS = ["p95_us", "makespan_us", "events", "digest", "slo_met", "n_done", "status"]


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()
    H.load()


def gpu(wl, record=(), **kw):
    sim = H.Sim(wl.traces, wl.cluster, wl.grid, record_sims=record, **kw)
    sim.run()
    return sim


def assert_same(g, o, what=""):
    for f in FIELDS:
        bad = np.nonzero(g[f] != o[f])[0]
        assert bad.size == 0, f"{what} field {f} differs at {bad[:8].tolist()}: gpu {g[f][bad[:4]]} oracle {o[f][bad[:4]]}"


def assert_logs(sim, wl, j):
    s = sim.record_sims[j]
    P = wl.grid.n_points
    tr = wl.traces[s // P]
    _, lo = oracle.simulate(tr, wl.cluster, oracle.point_of(wl.grid, s % P), log=True)
    lg = sim.records(j)
    for f in ("inst", "enq", "budget", "start", "end"):
        bad = np.nonzero(lg[f] != lo[f])[0]
        assert bad.size == 0, f"sim {s}: {f} differs first at call {bad[:5].tolist()}"


def oracle_results(wl, sims):
    return oracle.run(wl, sims, procs=NPROC)


def check_best(sim, wl, res):
    nq = [t.n_queries for t in wl.traces]
    for obj in (W.OBJ_P95, W.OBJ_P95_SLO95):
        gp, gs, per = oracle.best(res, len(wl.traces), wl.grid.n_points, nq, obj)
        bp, bs, _, bper = sim.best(obj)
        assert (bp, bs) == (gp, gs) and bper.tolist() == per.tolist(), f"objective {obj}"


# ------------------------------------------------------------------ hand cases
@pytest.mark.parametrize("name", sorted(cases.load_golden("hand_cases.json")["cases"].keys()))
def test_hand_case(name):
    tr, cl, exp = cases.hand_case(name)
    grid = cases.grid_from_points([exp["point"]])
    wl = W.Workload(name, [tr], cl, grid, W.OBJ_P95)
    sim = gpu(wl, record=[0])
    r = sim.results()[0]
    lg = sim.records(0)
    assert r["status"] == 0
    assert lg["inst"].tolist() == exp["inst"]
    assert lg["start"].tolist() == exp["start"]
    if "budget" in exp:
        assert lg["budget"].tolist() == exp["budget"]
    assert int(r["p95_us"]) == exp["p95_us"] and int(r["slo_met"]) == exp["slo_met"]
    assert int(r["makespan_us"]) == exp["makespan_us"]
    if "tenant_slo_met" in exp:
        e = sim.extras()[0]
        assert e["slo_met"].tolist() == exp["tenant_slo_met"] and e["n_done"].tolist() == exp["tenant_done"]
        assert int(e["reissued"]) == exp["reissued"]
    sim.close()


# ---------------------------------------------------------------- preparation
@pytest.mark.parametrize("cfg,nt,nq", [(0, None, None), (2, 2, 300), (3, 1, 500), (4, 2, 300)])
def test_prep_matches_oracle(cfg, nt, nq):
    wl = W.make_workload(cfg, n_traces=nt, n_queries=nq)
    sim = gpu(wl)
    T = wl.cluster.n_types
    for t, tr in enumerate(wl.traces):
        g = sim.prep(t)
        o = oracle.prep(tr, wl.cluster)
        assert (g["est"][:, :T] == o["est"]).all() and (g["svc"][:, :T] == o["svc"]).all()
        assert (g["tbar"] == o["tbar"]).all()
        qid = np.repeat(np.arange(tr.n_queries), np.diff(tr.call_base))
        assert (g["deadline"] == tr.arrival_us[qid] + o["t_slo"][qid]).all()
    sim.close()


# ------------------------------------------------------------- small, complete
def test_recipe0_every_sim_and_every_call():
    wl = W.make_workload(0)
    sim = gpu(wl, record=range(wl.n_sims))
    g = sim.results()
    o = oracle_results(wl, range(wl.n_sims))
    assert_same(g, o, "recipe 0")
    for j in range(wl.n_sims):
        assert_logs(sim, wl, j)
    check_best(sim, wl, o)
    golden = cases.load_golden("cfg0_oracle.json")
    assert [int(x) for x in g["digest"]] == [r["digest"] for r in golden["results"]]
    sim.close()


REDUCED = [
    (1, 2, 400, 6),
    (2, 2, 300, 6),
    (3, 1, 300, 6),
    (4, 1, 200, 6),
]


@pytest.mark.parametrize("cfg,nt,nq,nrec", REDUCED)
def test_reduced_recipes_every_sim(cfg, nt, nq, nrec):
    wl = W.make_workload(cfg, n_traces=nt, n_queries=nq)
    rng = np.random.default_rng(cfg)
    rec = sorted(rng.choice(wl.n_sims, size=nrec, replace=False).tolist() + [wl.n_sims - 1])
    rec = sorted(set(rec))
    sim = gpu(wl, record=rec)
    g = sim.results()
    o = oracle_results(wl, range(wl.n_sims))
    assert_same(g, o, f"recipe {cfg}")
    for j in range(len(rec)):
        assert_logs(sim, wl, j)
    check_best(sim, wl, o)
    sim.close()


@pytest.mark.parametrize("local,dispatch", [(W.POLICY_FCFS, W.DISPATCH_WB), (W.POLICY_PQ, W.DISPATCH_RR),
                                            (W.POLICY_FCFS, W.DISPATCH_RR), (W.POLICY_LLF, W.DISPATCH_WB),
                                            (W.POLICY_LLF, W.DISPATCH_RR)])
def test_policy_variants(local, dispatch):
    wl = W.make_workload(1, n_traces=2, n_queries=300)
    g0 = wl.grid
    wl.grid = W.Grid(g0.alpha_fp, g0.gamma_fp, g0.rho, g0.beta_us2, np.full(g0.n_points, local, np.uint8),
                     np.full(g0.n_points, dispatch, np.uint8))
    sim = gpu(wl, record=[0, 77])
    o = oracle_results(wl, range(wl.n_sims))
    assert_same(sim.results(), o, "policies")
    assert_logs(sim, wl, 0)
    assert_logs(sim, wl, 1)
    sim.close()


def test_overload_long_queues():
    """alpha near 1 on recipe 4 routes nearly everything to one instance: its
    local queue grows to thousands and its heap is re-homed many times."""
    wl = W.make_workload(4, n_traces=1, n_queries=3000)
    pts = list(range(1024 - 16, 1024)) + list(range(896 - 8, 896)) + [0, 5, 300]
    wl.grid = W.subset_grid(wl.grid, pts)
    sim = gpu(wl, record=[0, len(pts) - 4])
    o = oracle_results(wl, range(wl.n_sims))
    assert_same(sim.results(), o, "overload")
    assert_logs(sim, wl, 0)
    assert_logs(sim, wl, 1)
    sim.close()


def test_ragged_traces_and_empty():
    r = W.RECIPES[2]
    traces = [W.make_trace(r, 2, 0, n_queries=0), W.make_trace(r, 2, 1, n_queries=1),
              W.make_trace(r, 2, 2, n_queries=3), W.make_trace(r, 2, 3, n_queries=700),
              W.make_trace(r, 2, 4, n_queries=0), W.make_trace(r, 2, 5, n_queries=37)]
    wl = W.Workload("ragged", traces, W.make_cluster(r), W.subset_grid(W.make_grid(r), list(range(0, 256, 9))),
                    W.OBJ_P95)
    P = wl.grid.n_points
    sim = gpu(wl, record=[P * 1, P * 2 + 3, P * 3 + 5, P * 5 + 7])
    g = sim.results()
    o = oracle_results(wl, range(wl.n_sims))
    assert_same(g, o, "ragged")
    assert (g["p95_us"][:P] == 0).all() and (g["n_done"][:P] == 0).all()
    for j in range(4):
        assert_logs(sim, wl, j)
    check_best(sim, wl, o)
    sim.close()


def test_largest_shapes():
    """64 instances of 16 slots (1024 slots per simulation), k = 8 candidates,
    up to 15 corrections per chain."""
    r = W.RECIPES[2]
    r2 = W.Recipe("maxshape", 2, 120, "poisson", [3.0], 0.0, [8, 8], 0.85, 15, r.prompt, r.out, r.out_est,
                  r.ref_prompt, [W.TYPE_C, W.TYPE_A], [64, 0], 1, 3 * W.SCALE, 4, [W.SCALE, 4 * W.SCALE], [0, 15],
                  [(1, 1)], 300_000, W.OBJ_P95)
    traces = [W.make_trace(r2, 9, s) for s in range(2)]
    assert max(int(t.retry.max()) for t in traces) == 15
    wl = W.Workload("maxshape", traces, W.make_cluster(r2), W.make_grid(r2), W.OBJ_P95)
    sim = gpu(wl, record=[1, 13])
    o = oracle_results(wl, range(wl.n_sims))
    assert_same(sim.results(), o, "max shapes")
    assert_logs(sim, wl, 0)
    assert_logs(sim, wl, 1)
    sim.close()


def test_repeat_runs_and_upload():
    wl = W.make_workload(1, n_traces=2, n_queries=300)
    sim = gpu(wl)
    a = sim.results()
    sim.run()
    b = sim.results()
    assert_same(a, b, "repeat")
    # same shapes, different tokens and arrivals: upload in place == fresh handle
    alt = []
    for t in wl.traces:
        u = W.Trace(*[getattr(t, f).copy() for f in ("arrival_us", "k", "call_base", "prompt", "out", "out_est",
                                                      "stage", "cand", "retry")])
        u.prompt[:] = u.prompt[::-1].copy()
        u.arrival_us[:] = u.arrival_us * 3 // 4
        alt.append(u)
    sim.upload(alt)
    sim.run()
    c = sim.results()
    wl2 = W.Workload("alt", alt, wl.cluster, wl.grid, wl.objective)
    fresh = gpu(wl2)
    assert_same(c, fresh.results(), "upload")
    o = oracle_results(wl2, range(wl2.n_sims))
    assert_same(c, o, "upload vs oracle")
    sim.close()
    fresh.close()


def test_upload_with_tenants():
    # two-tenant traces: re-uploading them reproduces every result; uploading
    # them without tenant arrays makes every query tenant 0
    wl = W.make_workload("two-tenant", n_traces=2, n_queries=300)
    sim = gpu(wl)
    a, ea = sim.results(), sim.extras()
    fields = ("arrival_us", "k", "call_base", "prompt", "out", "out_est", "stage", "cand", "retry", "tenant")
    sim.upload([W.Trace(*[None if getattr(t, f) is None else getattr(t, f).copy() for f in fields])
                for t in wl.traces])
    sim.run()
    assert_same(sim.results(), a, "upload with tenants")
    assert np.array_equal(sim.extras(), ea)
    plain = [W.Trace(*[getattr(t, f) for f in fields[:-1]]) for t in wl.traces]
    sim.upload(plain)
    sim.run()
    b, eb = sim.results(), sim.extras()
    o, oe = oracle.run(W.Workload("no tenants", plain, wl.cluster, wl.grid, wl.objective), range(wl.n_sims),
                       procs=NPROC, extra=True)
    assert_same(b, o, "upload without tenants")
    assert_extras(eb, oe, "upload without tenants")
    assert (eb["n_done"][:, 1] == 0).all()
    sim.close()


# ------------------------------------------------------------------ full size
def stratified_sims(wl, per_alpha, alpha1_trace, seed):
    """Simulations drawn evenly over the grid's alpha values (per_alpha of
    each, trace and the other axes at random, without repeats), plus every
    alpha = 1 point of one trace: the points whose local queues grow longest
    and whose simulations cost the oracle the most."""
    g = wl.grid
    P, T = g.n_points, len(wl.traces)
    rng = np.random.default_rng(seed)
    sims = set()
    for a in np.unique(g.alpha_fp):
        pts = np.nonzero(g.alpha_fp == a)[0]
        pick = rng.choice(T * pts.size, size=min(per_alpha, T * pts.size), replace=False)
        sims.update((pick // pts.size * P + pts[pick % pts.size]).tolist())
    a1 = np.nonzero(g.alpha_fp == W.SCALE)[0]
    sims.update((alpha1_trace * P + a1).tolist())
    return sorted(sims)


def test_recipe1_full_every_sim():
    wl = W.make_workload(1)
    sim = gpu(wl)
    g = sim.results()
    o = oracle_results(wl, range(wl.n_sims))
    assert_same(g, o, "recipe 1")
    check_best(sim, wl, o)
    sim.close()


@pytest.mark.parametrize("cfg", [2, 3, 4])
def test_full_size_stratified(cfg):
    """A full recipe (config 4 is the benchmarked workload: 256 traces x
    20000 queries x 1024 points) in the benchmark's launch configuration:
    every simulation completes; a sample stratified over alpha (32 per alpha
    value, over all traces) plus every alpha = 1 point of one full-length
    trace matches the oracle exactly; the best-point kernel agrees with the
    oracle's rule applied to the GPU's whole table; and five full-length
    simulations (alpha = 0, two interior points, two at alpha = 1) have
    per-call logs equal to the oracle's."""
    wl = W.make_workload(cfg)
    sim = gpu(wl)
    assert sim.info()["generic_kernel"] == 0
    g = sim.results()
    P = wl.grid.n_points
    nq = np.repeat([t.n_queries for t in wl.traces], P)
    nc = np.repeat([t.n_calls for t in wl.traces], P)
    assert (g["status"] == 0).all() and (g["n_done"] == nq).all() and (g["events"] == nc).all()
    T = len(wl.traces)
    sims = stratified_sims(wl, 32, T - 1, 100 + cfg)
    assert len(sims) >= 256 and (wl.grid.alpha_fp[np.asarray(sims) % P] == W.SCALE).sum() >= P // 8
    o = oracle_results(wl, sims)
    assert_same(g[sims], o, f"recipe {cfg} stratified sample")
    nqt = [t.n_queries for t in wl.traces]
    for obj in (W.OBJ_P95, W.OBJ_P95_SLO95):
        gp, gs, per = oracle.best(g, T, P, nqt, obj)
        bp, bs, _, bper = sim.best(obj)
        assert (bp, bs) == (gp, gs) and bper.tolist() == per.tolist()
    sim.close()
    # full per-call logs of five full-length simulations (run alone as a subset)
    a1 = np.nonzero(wl.grid.alpha_fp == W.SCALE)[0]
    inner = np.nonzero((wl.grid.alpha_fp > 0) & (wl.grid.alpha_fp < W.SCALE))[0]
    rng = np.random.default_rng(7 + cfg)
    logged = sorted({0 * P + 0, 3 * P + int(rng.choice(inner)), (T // 2) * P + int(rng.choice(inner)),
                     1 * P + int(a1[0]), (T - 2) * P + int(a1[-1])})
    rec = gpu(wl, record=logged, subset=logged)
    assert_same(rec.results()[logged], g[logged], f"recipe {cfg} logged runs vs the full run")
    for j in range(len(logged)):
        assert_logs(rec, wl, j)
    rec.close()


def test_point_sums_and_best_of_sums():
    """Traces split over two handles (as over two ranks): the per-point sums
    add up to one handle's, and the best point of the sums is its best."""
    wl = W.make_workload(3, n_traces=4, n_queries=400)
    wl.grid = W.subset_grid(wl.grid, list(range(0, 512, 3)))
    whole = gpu(wl)
    halves = [gpu(W.Workload("h", wl.traces[i:i + 2], wl.cluster, wl.grid, wl.objective)) for i in (0, 2)]
    sums = [h.point_sums() for h in halves]
    tot = [sums[0][k] + sums[1][k] for k in range(3)]
    ref = whole.point_sums()
    for k in range(3):
        assert np.array_equal(tot[k], ref[k])
    nq = sum(t.n_queries for t in wl.traces)
    for obj in (W.OBJ_P95, W.OBJ_P95_SLO95):
        bp, bs, bslo, _ = whole.best(obj)
        assert H.best_of_sums(tot[0], tot[1], tot[2], nq, obj) == (bp, bs, bslo)
    for h in [whole] + halves:
        h.close()


@pytest.mark.parametrize("name,nt,nq", [("paper-shaped", 3, 150), ("noisy-estimate", 2, 300)])
def test_extra_recipes_every_sim(name, nt, nq):
    """~20 calls per query with up to 10 refinement rounds, and a noisy
    output-length estimate: every simulation and two full logs."""
    wl = W.make_workload(name, n_traces=nt, n_queries=nq)
    sim = gpu(wl, record=[1, wl.n_sims - 2])
    o = oracle_results(wl, range(wl.n_sims))
    assert_same(sim.results(), o, name)
    assert_logs(sim, wl, 0)
    assert_logs(sim, wl, 1)
    check_best(sim, wl, o)
    sim.close()


def test_lean_and_generic_kernels_agree():
    """The simulation kernel built for uniform WB + urgency-queue grids without
    logs gives exactly what the general one gives."""
    wl = W.make_workload(4, n_traces=2, n_queries=400)
    lean = gpu(wl)
    full = gpu(wl, force_generic=True)
    assert_same(lean.results(), full.results(), "lean vs generic")
    o = oracle_results(wl, list(range(0, wl.n_sims, 37)) + [wl.n_sims - 1])
    assert_same(lean.results()[list(range(0, wl.n_sims, 37)) + [wl.n_sims - 1]], o, "lean vs oracle")
    lean.close()
    full.close()


def assert_extras(g, o, what=""):
    for f in ("slo_met", "n_done", "reissued", "p95_us"):
        bad = np.nonzero((g[f] != o[f]).reshape(len(g), -1).any(axis=1))[0]
        assert bad.size == 0, f"{what} extra field {f} differs at {bad[:8].tolist()}"


@pytest.mark.parametrize("name,nt,nq", [("two-tenant", 2, 400), ("competing-25", 2, 300), ("competing-50", 1, 300),
                                        ("faulty", 1, 1400)])
def test_tenants_single_shots_faults_every_sim(name, nt, nq):
    """Two tenants with their own SLOs, competing single-shot requests, and
    instances that slow down or stop (timeout and re-issue): every
    simulation, the per-tenant counts and re-issues, and two full logs."""
    wl = W.make_workload(name, n_traces=nt, n_queries=nq)
    sim = gpu(wl, record=[0, wl.n_sims - 1])
    assert sim.info()["generic_kernel"] == 1
    o, oe = oracle.run(wl, range(wl.n_sims), procs=NPROC, extra=True)
    assert_same(sim.results(), o, name)
    assert_extras(sim.extras(), oe, name)
    if name == "faulty":
        assert int(oe["reissued"].sum()) > 0
    assert_logs(sim, wl, 0)
    assert_logs(sim, wl, 1)
    check_best(sim, wl, o)
    sim.close()


def test_single_shots_on_the_lean_kernel():
    """Single-shot requests (k = 0) of one tenant run on the lean kernel."""
    src = W.make_workload("competing-25", n_traces=2, n_queries=300)
    traces = [W.Trace(*[getattr(t, f) for f in ("arrival_us", "k", "call_base", "prompt", "out", "out_est",
                                                "stage", "cand", "retry")]) for t in src.traces]
    c = src.cluster
    cl = W.Cluster(c.prefill_tok_s, c.decode_us_tok, c.slots, c.inst_type, c.ref_type, c.slo_mult_fp, c.rmax,
                   c.stage_ref_prompt, c.stage_ref_out)
    wl = W.Workload("competing-25 one tenant", traces, cl, src.grid, src.objective)
    assert (traces[0].k == 0).any()
    sim = gpu(wl)
    assert sim.info()["generic_kernel"] == 0
    o = oracle_results(wl, range(wl.n_sims))
    assert_same(sim.results(), o, "lean single shots")
    e = sim.extras()
    assert (e["n_done"][:, 0] == o["n_done"]).all() and (e["n_done"][:, 1:] == 0).all()
    sim.close()


def _fault_cluster(c, faults, timeout_fp, tmult=None):
    f = np.zeros(len(faults), W.FAULT_DTYPE)
    for j, x in enumerate(faults):
        f[j] = (x[0], 0, x[1], x[2], x[3])
    return W.Cluster(c.prefill_tok_s, c.decode_us_tok, c.slots, c.inst_type, c.ref_type, c.slo_mult_fp, c.rmax,
                     c.stage_ref_prompt, c.stage_ref_out, tmult, timeout_fp, f)


def test_fault_edge_cases():
    """Overlapping windows (the first listed applies), a window stopping two
    instances at once, round robin stepping past the failed instance, and a
    one-instance cluster where a re-issue returns to the same instance."""
    src = W.make_workload(1, n_traces=1, n_queries=400)
    tr, c, g = src.traces[0], src.cluster, src.grid
    faults = [(0, 10_000_000, 40_000_000, 2 * W.SCALE), (0, 0, 60_000_000, 0), (1, 5_000_000, 70_000_000, 0),
              (6, 20_000_000, 30_000_000, 0), (2, 0, 100_000_000, 3 * W.SCALE // 2)]
    cl = _fault_cluster(c, faults, 2 * W.SCALE)
    pts = [0, 9, 27, 63]
    lp = np.zeros(len(pts), np.uint8)
    dp = np.array([0, 1, 0, 1], np.uint8)
    grid = W.Grid(g.alpha_fp[pts], g.gamma_fp[pts], g.rho[pts], g.beta_us2[pts], lp, dp)
    wl = W.Workload("fault edges", [tr], cl, grid, W.OBJ_P95)
    sim = gpu(wl, record=[1, 2])
    o, oe = oracle.run(wl, range(wl.n_sims), procs=NPROC, extra=True)
    assert_same(sim.results(), o, "fault edges")
    assert_extras(sim.extras(), oe, "fault edges")
    assert int(oe["reissued"].sum()) > 0
    assert_logs(sim, wl, 0)
    assert_logs(sim, wl, 1)
    sim.close()
    # one instance: a re-issue goes back to it
    one = W.Cluster(c.prefill_tok_s[:1], c.decode_us_tok[:1], c.slots[:1], np.zeros(1, np.uint8), 0, c.slo_mult_fp,
                    c.rmax, c.stage_ref_prompt, c.stage_ref_out, None, 3 * W.SCALE,
                    np.array([(0, 0, 0, 2_000_000, 0)], W.FAULT_DTYPE))
    tr1 = W.make_workload(0, n_queries=40).traces[0]
    wl1 = W.Workload("one instance", [tr1], one, grid, W.OBJ_P95)
    sim = gpu(wl1)
    o, oe = oracle.run(wl1, range(wl1.n_sims), extra=True)
    assert_same(sim.results(), o, "one instance")
    assert_extras(sim.extras(), oe, "one instance")
    sim.close()


def test_four_tenants_and_only_single_shots():
    """Four tenants with random assignment, and a trace made only of
    single-shot requests."""
    src = W.make_workload(1, n_traces=2, n_queries=300)
    c = src.cluster
    cl = W.Cluster(c.prefill_tok_s, c.decode_us_tok, c.slots, c.inst_type, c.ref_type, c.slo_mult_fp, c.rmax,
                   c.stage_ref_prompt, c.stage_ref_out, np.array([W.SCALE, 2 * W.SCALE, 3 * W.SCALE, 16 * W.SCALE]))
    rng = np.random.default_rng(5)
    traces = []
    for t in src.traces:
        t2 = W.Trace(*[getattr(t, f) for f in ("arrival_us", "k", "call_base", "prompt", "out", "out_est", "stage",
                                               "cand", "retry")], rng.integers(0, 4, t.n_queries).astype(np.uint8))
        traces.append(t2)
    # single shots only: one E call per query
    n = 500
    arr = np.cumsum(rng.integers(0, 400_000, n)).astype(np.int64)
    singles = W.Trace(arr, np.zeros(n, np.uint8), np.arange(n + 1, dtype=np.int32),
                      rng.integers(100, 5000, n).astype(np.int32), rng.integers(10, 400, n).astype(np.int32),
                      np.full(n, 200, np.int32), np.full(n, W.STAGE_E, np.uint8), np.zeros(n, np.uint8),
                      np.zeros(n, np.uint8), rng.integers(0, 4, n).astype(np.uint8))
    traces.append(singles)
    wl = W.Workload("tenants", traces, cl, W.subset_grid(src.grid, [0, 20, 45, 63]), W.OBJ_P95_SLO95)
    sim = gpu(wl, record=[wl.n_sims - 1])
    o, oe = oracle.run(wl, range(wl.n_sims), procs=NPROC, extra=True)
    assert_same(sim.results(), o, "tenants")
    assert_extras(sim.extras(), oe, "tenants")
    assert_logs(sim, wl, 0)
    check_best(sim, wl, o)
    sim.close()


def test_per_tenant_p95_from_records():
    """Per-tenant P95 from a recorded simulation's call end times equals the
    oracle's and the device's own per-tenant P95, also when fault windows
    stretch services."""
    from paper_2505_05286_gb300 import tenants as T
    for name, nq in (("two-tenant", 400), ("faulty", 1400)):
        wl = W.make_workload(name, n_traces=1, n_queries=nq)
        tr = wl.traces[0]
        sim = gpu(wl, record=[5, 40])
        ex = sim.extras()
        for j, s in enumerate([5, 40]):
            _, lo = oracle.simulate(tr, wl.cluster, oracle.point_of(wl.grid, s), log=True)
            lat_g = T.query_latencies(tr, sim.records(j))
            lat_o = lo["end"][tr.call_base[1:] - 1] - tr.arrival_us
            assert (lat_g == lat_o).all()
            nt = wl.cluster.n_tenants
            assert T.tenant_p95(lat_g, tr.tenant, nt) == T.tenant_p95(lat_o, tr.tenant, nt)
            assert [int(x) for x in ex["p95_us"][s][:nt]] == [x or 0 for x in T.tenant_p95(lat_o, tr.tenant, nt)]
        sim.close()


def test_per_tenant_p95_on_the_grid_without_records():
    """The device's per-tenant P95 on every simulation of the two-tenant and
    competing recipes (no per-call logs), against the oracle's."""
    for name, nt, nq in (("two-tenant", 2, 500), ("competing-50", 1, 400)):
        wl = W.make_workload(name, n_traces=nt, n_queries=nq)
        sim = gpu(wl)
        o, oe = oracle.run(wl, range(wl.n_sims), procs=NPROC, extra=True)
        assert_same(sim.results(), o, name)
        ex = sim.extras()
        assert_extras(ex, oe, name)
        assert (ex["p95_us"][:, :2] > 0).all() and (ex["p95_us"][:, 2:] == 0).all()
        sim.close()


def test_results_as_tensors():
    wl = W.make_workload(0)
    sim = gpu(wl)
    r = sim.results()
    t = sim.results_tensors()
    assert set(t) == set(H.RESULT_DTYPE.names)
    assert (t["p95_us"].numpy() == r["p95_us"]).all() and (t["digest"].numpy().view(np.uint64) == r["digest"]).all()
    sim.close()


@pytest.mark.parametrize("seed", range(24))
def test_random_small_workloads(seed):
    """Random clusters, traces and grids: every simulation, the per-tenant
    counts and a full log equal the oracle's (odd seeds with the per-event
    invariant checks on)."""
    wl = cases.random_workload(seed)
    sim = gpu(wl, record=[wl.n_sims - 1], checked=bool(seed % 2))
    o, oe = oracle.run(wl, range(wl.n_sims), extra=True)
    assert (o["status"] == 0).all()
    assert_same(sim.results(), o, wl.name)
    assert_extras(sim.extras(), oe, wl.name)
    assert_logs(sim, wl, 0)
    check_best(sim, wl, o)
    sim.close()


@pytest.mark.parametrize("seed", range(24))
def test_random_small_workloads_lean(seed):
    """The same random shapes (any instance count and slots, k from 0 to 8)
    on WB + the urgency queue alone, so that the benchmark's lean kernel runs
    them: every simulation and the best points equal the oracle's."""
    wl = cases.random_workload(seed, lean=True)
    sim = gpu(wl)
    assert sim.info()["generic_kernel"] == 0
    o = oracle_results(wl, range(wl.n_sims))
    assert (o["status"] == 0).all()
    assert_same(sim.results(), o, wl.name)
    check_best(sim, wl, o)
    sim.close()


def test_command_line(capsys):
    import json
    from paper_2505_05286_gb300 import __main__ as cli
    assert cli.main(["--recipe", "0"]) == 0
    out = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    wl = W.make_workload(0)
    o = oracle_results(wl, range(wl.n_sims))
    gp, gs, _ = oracle.best(o, 1, wl.grid.n_points, [wl.traces[0].n_queries], W.OBJ_P95)
    assert out["best_point"] == gp and out["sum_p95_us"] == gs and out["failed"] == 0


# ------------------------------------------------------------ subset, checked
@pytest.mark.parametrize("generic", [False, True])
def test_subset_runs_only_the_listed_simulations(generic):
    wl = W.make_workload(1, n_traces=2, n_queries=300)  # 2 traces x 64 points
    sub = [5, 64 + 63, 0, 64 + 7, 40, 63]
    sim = gpu(wl, subset=sub, force_generic=generic)
    r = sim.results()
    inside = np.zeros(wl.n_sims, bool)
    inside[sub] = True
    o = oracle_results(wl, sub)
    assert_same(r[np.sort(sub)], o[np.argsort(sub)], "subset")
    assert (r["status"][~inside] == H.HX_SKIPPED).all() and (r["p95_us"][~inside] == -1).all()
    assert (r["events"][~inside] == 0).all() and (r["n_done"][~inside] == 0).all()
    if generic:
        e = sim.extras()
        assert (e["n_done"][~inside] == 0).all() and (e["n_done"][inside].sum(axis=1) == 300).all()
    # the best-point reduction counts the skipped simulations as failed
    check_best(sim, wl, r)
    sim.run()
    assert_same(sim.results(), r, "subset re-run")
    sim.close()


@pytest.mark.parametrize("generic", [False, True])
def test_costliest_first_order_changes_no_result(generic):
    # 4 traces x 64 points on 64 resident warps: four waves, records far
    # below L2, so every trace's workload-balanced alpha = 1 points go first
    wl = W.make_workload(1, n_traces=4, n_queries=300)
    sim = gpu(wl, max_resident_warps=64, force_generic=generic)
    assert sim.info()["work_order"] == 2
    r = sim.results()
    assert_same(r, oracle_results(wl, range(wl.n_sims)), "costliest first")
    check_best(sim, wl, r)
    sim.close()
    # one wave: the default order; a subset: its own; eight waves: only the
    # last trace (two waves of 32 warps) takes its alpha = 1 points first
    for kw, order in (({}, 0), ({"subset": list(range(0, wl.n_sims, 3)), "max_resident_warps": 64}, 1),
                      ({"max_resident_warps": 32}, 3)):
        s2 = gpu(wl, force_generic=generic, **kw)
        assert s2.info()["work_order"] == order
        if order == 3:
            assert_same(s2.results(), r, "last traces' alpha = 1 points first")
        s2.close()


@pytest.mark.parametrize("name,nt,nq", [(1, 2, 300), ("faulty", 1, 1400), ("competing-50", 1, 300)])
def test_checked_mode_changes_nothing(name, nt, nq):
    """With the per-event invariant checks on (generic kernel), every
    simulation still matches the oracle, status included."""
    wl = W.make_workload(name, n_traces=nt, n_queries=nq)
    if name == 1:
        # mixed policies over the points
        g = wl.grid
        lp = np.array([W.POLICY_PQ, W.POLICY_FCFS, W.POLICY_LLF, W.POLICY_PQ], np.uint8)[np.arange(g.n_points) % 4]
        dp = np.array([W.DISPATCH_WB, W.DISPATCH_WB, W.DISPATCH_WB, W.DISPATCH_RR], np.uint8)[np.arange(g.n_points) % 4]
        wl = W.Workload(wl.name, wl.traces, wl.cluster, W.Grid(g.alpha_fp, g.gamma_fp, g.rho, g.beta_us2, lp, dp),
                        wl.objective)
    sim = gpu(wl, checked=True)
    assert sim.info()["generic_kernel"] == 1
    o = oracle_results(wl, range(wl.n_sims))
    assert_same(sim.results(), o, f"checked {name}")
    sim.close()


def _arena_need(log, n_inst):
    """Lower and upper bounds of the arena entries one simulation takes: per
    instance the heap of its largest queue, grown by doubling from 16 (16 +
    32 + ...); the lower bound counts requests strictly waiting after an
    event, the upper one also those queued and started in the same event."""
    def alloc(s):
        c = tot = 16 if s else 0
        while s and c < s:
            c *= 2
            tot += c
        return tot
    lo = hi = 0
    for m in range(n_inst):
        sel = log["inst"] == m
        enq, st = log["enq"][sel], log["start"][sel]
        cur = top = 0
        for _, _, d in sorted([(e, 0, 1) for e in enq] + [(s, 1, -1) for s in st]):
            cur += d
            top = max(top, cur)
        hi += alloc(top)
        w = st > enq
        cur = top = 0
        for _, _, d in sorted([(e, 1, 1) for e in enq[w]] + [(s, 0, -1) for s in st[w]]):
            cur += d
            top = max(top, cur)
        lo += alloc(top)
    return lo, hi


@pytest.mark.parametrize("generic", [False, True])
def test_small_arena_reports_capacity(generic):
    """A local-queue arena too small for the alpha = 1 queues: those
    simulations stop with HX_ERR_CAPACITY (no truncation, no fault), the others
    still match the oracle."""
    wl = W.make_workload(4, n_traces=1, n_queries=1500)
    pts = list(range(0, 1024, 64)) + list(range(1024 - 128, 1024, 16))
    wl = W.Workload(wl.name, wl.traces, wl.cluster, W.subset_grid(wl.grid, pts), wl.objective)
    arena = 1024
    sim = gpu(wl, arena_entries=arena, force_generic=generic)
    r = sim.results()
    o = oracle_results(wl, range(wl.n_sims))
    n_cap = n_ok = 0
    for p in range(wl.n_sims):
        _, log = oracle.simulate(wl.traces[0], wl.cluster, oracle.point_of(wl.grid, p), log=True)
        lo, hi = _arena_need(log, wl.cluster.n_inst)
        if hi <= arena:
            n_ok += 1
            assert r["status"][p] == H.HX_OK, p
        if lo > arena:
            n_cap += 1
            assert r["status"][p] == H.HX_ERR_CAPACITY and r["p95_us"][p] == -1, p
        if r["status"][p] == H.HX_OK:
            assert_same(r[p:p + 1], o[p:p + 1], f"point {p}")
        else:
            assert r["status"][p] == H.HX_ERR_CAPACITY
    assert n_cap >= 4 and n_ok >= 8
    sim.close()


def test_step_limit_on_endless_reissues():
    """One instance stopped with a timeout of 1x: every attempt fails after
    its 2 ms estimate and goes out again to the same instance.  A 20 ms
    window (10 re-issues) matches the oracle; a 100 s window needs 50000
    re-issues, more events than the bound (n_calls + n_queries + 8 +
    16 n_calls + 4096), so the simulation stops with HX_ERR_STEP_LIMIT."""
    g = cases.load_golden("hand_cases.json")
    tr = cases.trace_from(g["traces"]["T10_one_query"])
    pt = dict(alpha_fp=W.SCALE // 2, gamma_fp=W.SCALE, beta_us2=9_000_000, rho=0, local_policy=0, dispatch_policy=0)

    def workload(t1):
        f = np.zeros(1, W.FAULT_DTYPE)
        f[0] = (0, 0, 0, t1, 0)
        cl = W.Cluster(np.array([1000], np.int32), np.array([1000], np.int32), np.array([1], np.int32),
                       np.zeros(1, np.uint8), 0, 3 * W.SCALE, 0, np.ones(4, np.int32), np.ones(4, np.int32),
                       None, W.SCALE, f)
        return W.Workload("stopped", [tr], cl, cases.grid_from_points([pt]), W.OBJ_P95)
    short = workload(20_000)
    s = gpu(short)
    o, oe = oracle.run(short, [0], extra=True)
    assert int(oe["reissued"][0]) == 10
    assert_same(s.results(), o, "20 ms window")
    assert_extras(s.extras(), oe, "20 ms window")
    s.close()
    long_ = workload(100_000_000)
    s = gpu(long_)
    r = s.results()[0]
    assert r["status"] == H.HX_ERR_STEP_LIMIT and r["p95_us"] == -1
    s.close()
