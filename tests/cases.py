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
