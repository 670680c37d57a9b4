"""Builders for small hand-made inputs used by the tests."""
import json
import os

import numpy as np

from paper_2505_05286_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
_STAGE = {"S": W.STAGE_S, "G": W.STAGE_G, "C": W.STAGE_C, "E": W.STAGE_E}


def load_golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def cluster_from(d, slo_mult_fp=None):
    faults = None
    if d.get("faults"):
        faults = np.zeros(len(d["faults"]), W.FAULT_DTYPE)
        for j, (m, t0, t1, slow) in enumerate(d["faults"]):
            faults[j] = (m, 0, t0, t1, slow)
    tm = d.get("tenant_slo_mult_fp")
    return W.Cluster(np.array(d["prefill_tok_s"], np.int32), np.array(d["decode_us_tok"], np.int32),
                     np.array(d["slots"], np.int32), np.array(d["inst_type"], np.uint8), int(d["ref_type"]),
                     int(d["slo_mult_fp"] if slo_mult_fp is None else slo_mult_fp), int(d["rmax"]),
                     np.array(d["stage_ref_prompt"], np.int32), np.array(d["stage_ref_out"], np.int32),
                     None if tm is None else np.array(tm, np.int64), int(d.get("timeout_mult_fp", 0)), faults)


def trace_from(d):
    arrival, k, base = [], [], [0]
    cols = {n: [] for n in ("stage", "cand", "retry", "prompt", "out", "out_est")}
    for q in d["queries"]:
        arrival.append(q["arrival"])
        k.append(q["k"])
        for c in q["calls"]:
            cols["stage"].append(_STAGE[c[0]])
            cols["cand"].append(c[1])
            cols["retry"].append(c[2])
            cols["prompt"].append(c[3])
            cols["out"].append(c[4])
            cols["out_est"].append(c[5])
        base.append(base[-1] + len(q["calls"]))
    tenant = None
    if any("tenant" in q for q in d["queries"]):
        tenant = np.array([q.get("tenant", 0) for q in d["queries"]], np.uint8)
    return W.Trace(np.array(arrival, np.int64), np.array(k, np.uint8), np.array(base, np.int32),
                   np.array(cols["prompt"], np.int32), np.array(cols["out"], np.int32),
                   np.array(cols["out_est"], np.int32), np.array(cols["stage"], np.uint8),
                   np.array(cols["cand"], np.uint8), np.array(cols["retry"], np.uint8), tenant)


def grid_from_points(points):
    f = lambda key, dt: np.array([p[key] for p in points], dt)
    return W.Grid(f("alpha_fp", np.int64), f("gamma_fp", np.int64), f("rho", np.int32),
                  f("beta_us2", np.int64), f("local_policy", np.uint8), f("dispatch_policy", np.uint8))


def hand_case(name):
    g = load_golden("hand_cases.json")
    c = g["cases"][name]
    cl = cluster_from(g["clusters"][c["cluster"]], c.get("slo_mult_fp"))
    tr = trace_from(g["traces"][c["trace"]])
    return tr, cl, c


def uniform_single_instance(n, arrivals, svc_us=1000, slots=1):
    """n queries (k = 1, no corrections) on one instance where every call costs svc_us:
    prefill 1e6 tok/s with a 1-token prompt (1 us) plus one output token at svc_us - 1 us."""
    q = [{"arrival": int(a), "k": 1, "calls": [["S", 0, 0, 1, 1, 1], ["G", 0, 0, 1, 1, 1],
                                             ["E", 0, 0, 1, 1, 1]]} for a in arrivals[:n]]
    tr = trace_from({"queries": q})
    cl = W.Cluster(np.array([1_000_000], np.int32), np.array([svc_us - 1], np.int32),
                   np.array([slots], np.int32), np.array([0], np.uint8), 0, 3 * W.SCALE, 0,
                   np.ones(4, np.int32), np.ones(4, np.int32))
    return tr, cl


def random_workload(seed, lean=False):
    """A small random but valid workload: any cluster shape, k from 0 to 8,
    retries up to R, tenants, fault windows, mixed policies.  `lean` keeps
    the shapes but drops tenants and fault windows and puts every point on
    WB + the urgency queue (the domain of the benchmark's kernel)."""
    rng = np.random.default_rng(1000 + seed)
    T = int(rng.integers(1, 5))
    N = int(rng.integers(1, 65))
    prefill = rng.integers(500, 30000, T).astype(np.int32)
    decode = rng.integers(1, 60, T).astype(np.int32)
    slots = rng.integers(1, 17, T).astype(np.int32)
    inst_type = np.sort(rng.integers(0, T, N)).astype(np.uint8)
    rmax = int(rng.integers(0, 5))
    n_ten = int(rng.integers(1, 5))
    tmult = rng.integers(W.SCALE, 6 * W.SCALE, n_ten).astype(np.int64) if n_ten > 1 else None
    faults = None
    timeout = 0
    if rng.random() < 0.5:
        timeout = int(rng.integers(W.SCALE, 4 * W.SCALE))
        nf = int(rng.integers(1, 5))
        faults = np.zeros(nf, W.FAULT_DTYPE)
        for j in range(nf):
            t0 = int(rng.integers(0, 60_000_000))
            faults[j] = (int(rng.integers(0, N)), 0, t0, t0 + int(rng.integers(0, 30_000_000)),
                         0 if rng.random() < 0.4 else int(rng.integers(W.SCALE // 2, 4 * W.SCALE)))
    cl = W.Cluster(prefill, decode, slots, inst_type, int(rng.integers(0, T)), int(rng.integers(W.SCALE, 5 * W.SCALE)),
                   rmax, rng.integers(100, 3000, 4).astype(np.int32), rng.integers(10, 300, 4).astype(np.int32),
                   tmult, timeout, faults)
    nq = int(rng.integers(1, 120))
    arrival = np.sort(rng.integers(0, 80_000_000, nq)).astype(np.int64)
    ks, base, stage, cand, retry = [], [0], [], [], []
    for _ in range(nq):
        k = int(rng.integers(0, 9))
        ks.append(k)
        if k == 0:
            stage.append(W.STAGE_E); cand.append(0); retry.append(0)
        else:
            stage.append(W.STAGE_S); cand.append(0); retry.append(0)
            for cidx in range(k):
                stage.append(W.STAGE_G); cand.append(cidx); retry.append(0)
            for cidx in range(k):
                for r in range(1, int(rng.integers(0, rmax + 1)) + 1):
                    stage.append(W.STAGE_C); cand.append(cidx); retry.append(r)
            stage.append(W.STAGE_E); cand.append(0); retry.append(0)
        base.append(len(stage))
    nc = len(stage)
    tr = W.Trace(arrival, np.array(ks, np.uint8), np.array(base, np.int32),
                 rng.integers(1, 8000, nc).astype(np.int32), rng.integers(0, 600, nc).astype(np.int32),
                 rng.integers(0, 600, nc).astype(np.int32), np.array(stage, np.uint8), np.array(cand, np.uint8),
                 np.array(retry, np.uint8), rng.integers(0, n_ten, nq).astype(np.uint8) if n_ten > 1 else None)
    P = 6
    grid = W.Grid(rng.integers(0, W.SCALE + 1, P).astype(np.int64), rng.integers(0, 4 * W.SCALE + 1, P).astype(np.int64),
                  rng.integers(0, 4, P).astype(np.int32), rng.integers(0, 10 ** 12, P).astype(np.int64),
                  rng.integers(0, 3, P).astype(np.uint8), rng.integers(0, 2, P).astype(np.uint8))
    grid.alpha_fp[0], grid.alpha_fp[1] = 0, W.SCALE
    objective = int(rng.integers(0, 2))
    if lean:
        cl = W.Cluster(cl.prefill_tok_s, cl.decode_us_tok, cl.slots, cl.inst_type, cl.ref_type, cl.slo_mult_fp,
                       cl.rmax, cl.stage_ref_prompt, cl.stage_ref_out)
        tr.tenant = None
        grid.local_policy[:] = W.POLICY_PQ
        grid.dispatch_policy[:] = W.DISPATCH_WB
        return W.Workload(f"random lean {seed}", [tr], cl, grid, objective)
    return W.Workload(f"random {seed}", [tr], cl, grid, objective)
