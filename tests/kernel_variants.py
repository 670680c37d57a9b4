"""Kernel variants: source edits of the simulation kernel, built beside the
library and timed against it on the same workload, each required to give
bit-identical results.  This is how the alternatives the design notes
mention were measured (GPU only).

    python -m tests.kernel_variants prefetch [--traces 64] [--reps 3] [--out FILE]

Variants `prefetch`:
  arrival_l1 / arrival_l2  at a query's arrival, prefetch its call records
                           (up to 10 records, 5 lines of 128 bytes) into L1 / L2;
  start_l1 / start_l2      when a request is dispatched, prefetch the records
                           that follow its own (its successors) into L1 / L2.
Every prefetch stays inside the trace's records.
"""
from __future__ import annotations

import argparse
import json
import os
import shutil
import subprocess
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

CSRC = os.path.join(ROOT, "paper_2505_05286_gb300", "csrc")
OUT = os.path.join(ROOT, "paper_2505_05286_gb300", "_variants")
NVCC = ["nvcc", "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-lineinfo", "-std=c++17", "-Xcompiler",
        "-fPIC", "-I", os.path.join(ROOT, "include")]

_ARRIVAL = ("""        rel_first = (int32_t)(a.qcall[qbase + qa] - W->cb);""",
            """        rel_first = (int32_t)(a.qcall[qbase + qa] - W->cb);
        {
          const char* pa = reinterpret_cast<const char*>(rec + rel_first) + 128 * lane;
          if (lane < 5 && (int64_t)rel_first * 64 + 128 * lane < (int64_t)nc * 64)
            asm volatile("prefetch.global.LVL [%0];" ::"l"(pa));
        }""")
_START = ("""        HX_BOUND(rid < nc)
        const CallRec* r = rec + rid;""",
          """        HX_BOUND(rid < nc)
        const CallRec* r = rec + rid;
        {
          const char* pa = reinterpret_cast<const char*>(r + 1) + 128 * lane;
          if (lane < 4 && (int64_t)(rid + 1) * 64 + 128 * lane < (int64_t)nc * 64)
            asm volatile("prefetch.global.LVL [%0];" ::"l"(pa));
        }""")

VARIANTS = {
    "prefetch": {f"{w}_{lvl.lower()}": [(e[0], e[1].replace("LVL", lvl))]
                 for w, e in (("arrival", _ARRIVAL), ("start", _START)) for lvl in ("L1", "L2")},
}


def make_variant(name, edits):
    """Copy the library sources, apply the edits to hx_kernels.cu, build a .so."""
    d = os.path.join(OUT, name)
    shutil.rmtree(d, ignore_errors=True)
    shutil.copytree(CSRC, os.path.join(d, "csrc"))
    p = os.path.join(d, "csrc", "hx_kernels.cu")
    s = open(p).read()
    for a, b in edits:
        if a not in s:
            raise RuntimeError(f"variant {name}: anchor not found in hx_kernels.cu: {a[:60]!r}")
        s = s.replace(a, b)
    open(p, "w").write(s)
    objs = []
    for src in ("hx_kernels.cu", "hx_api.cu"):
        o = os.path.join(d, src.replace(".cu", ".o"))
        subprocess.check_call(NVCC + ["-I", os.path.join(d, "csrc"), "-c", os.path.join(d, "csrc", src), "-o", o])
        objs.append(o)
    lib = os.path.join(d, "libhxsim.so")
    subprocess.check_call(NVCC[:3] + ["-shared", "-o", lib] + objs)
    return lib


def time_lib(lib_path, wl, reps, **sim_options):
    """Median simulation-kernel milliseconds over `reps` runs after one
    warm-up, and the results, with the library at lib_path (Sim options
    passed through)."""
    from paper_2505_05286_gb300 import hxsim as H
    saved = H._lib
    H._lib = H.load(lib_path)
    try:
        sim = H.Sim(wl.traces, wl.cluster, wl.grid, timing=True, **sim_options)
        sim.run()
        ms = []
        for _ in range(reps):
            sim.run()
            ms.append(sim.timings()[1])
        r = sim.results()
        sim.close()
    finally:
        H._lib = saved
    return float(np.median(ms)), ms, r


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("family", choices=sorted(VARIANTS))
    ap.add_argument("--traces", type=int, default=64)
    ap.add_argument("--reps", type=int, default=3)
    ap.add_argument("--out", default=None)
    args = ap.parse_args(argv)
    import torch

    from paper_2505_05286_gb300 import build as B
    from paper_2505_05286_gb300 import hxsim as H
    from paper_2505_05286_gb300 import workloads as W
    B.build()
    torch.cuda.set_device(0)
    wl = W.make_workload(4, n_traces=args.traces)
    fields = ("p95_us", "makespan_us", "events", "digest", "slo_met", "n_done", "status")
    base_ms, base_all, base = time_lib(H.LIB_PATH, wl, args.reps)
    out = {"workload": f"{wl.name} cut to {args.traces} traces", "sims": wl.n_sims, "library_ms": base_ms,
           "library_all_ms": base_all, "variants": {}}
    print("library", base_ms, base_all, flush=True)
    for name, edits in VARIANTS[args.family].items():
        ms, all_ms, r = time_lib(make_variant(name, edits), wl, args.reps)
        same = all(np.array_equal(r[f], base[f]) for f in fields)
        out["variants"][name] = {"ms": ms, "all_ms": all_ms, "same_results": same, "speedup": base_ms / ms}
        print(name, ms, all_ms, same, round(base_ms / ms, 4), flush=True)
    again, again_all, _ = time_lib(H.LIB_PATH, wl, args.reps)
    out["library_again_ms"] = again
    print("library again", again, again_all, flush=True)
    if args.out:
        with open(args.out, "w") as f:
            json.dump(out, f, indent=1)
    return 0 if all(v["same_results"] for v in out["variants"].values()) else 1


if __name__ == "__main__":
    sys.exit(main())
