"""Writes tests/golden/cfg0_oracle.json: the recipe-0 trace digest and the
oracle's result for every point of recipe 0.  Calls only the input generator
and the CPU oracle (never the CUDA library).

    python tests/golden/make_golden.py
"""
import hashlib
import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle  # noqa: E402
from paper_2505_05286_gb300 import workloads as W  # noqa: E402


def main():
    wl = W.make_workload(0)
    tr = wl.traces[0]
    h = hashlib.sha256()
    for f in ("arrival_us", "k", "call_base", "prompt", "out", "out_est", "stage", "cand", "retry"):
        h.update(np.ascontiguousarray(getattr(tr, f)).tobytes())
    res = oracle.run(wl, check=True)
    gp, gs, per = oracle.best(res, 1, wl.grid.n_points, [tr.n_queries], wl.objective)
    out = {
        "_source": "CPU oracle on recipe 0 (1 trace x 200 queries, 4 instances, 4 alpha x 4 gamma)",
        "trace_sha256": h.hexdigest(),
        "results": [{k: int(r[k]) for k in ("p95_us", "makespan_us", "events", "digest", "slo_met",
                                             "n_done", "status")} for r in res],
        "best": {"global_point": gp, "global_sum_p95": gs, "per_trace_point": per.tolist()},
    }
    with open(os.path.join(HERE, "cfg0_oracle.json"), "w") as f:
        json.dump(out, f, indent=1)


if __name__ == "__main__":
    main()
