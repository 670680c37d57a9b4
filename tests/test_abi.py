"""The C ABI without a GPU: the library builds for sm_103a, loads, exports
every function include/hxsim.h declares, its structs match the binding's
layout, and malformed inputs are rejected before any device work."""
import ctypes
import os
import subprocess

import numpy as np
import pytest

from paper_2505_05286_gb300 import build as B
from paper_2505_05286_gb300 import hxsim as H
from paper_2505_05286_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    B.build()
    return H.load()


def test_exports_every_declared_function(lib):
    names = H.declared_functions()
    assert len(names) >= 11
    for n in names:
        assert hasattr(lib, n), f"{n} declared in include/hxsim.h but not exported"


def test_bounds_checked_build_exports_the_same_functions(lib):
    chk = H.load_checked()
    for n in H.declared_functions():
        assert hasattr(chk, n), f"{n} missing from the bounds-checked build"
    assert os.path.getsize(H.LIB_CHECKED_PATH) > 0 and chk is not lib


_PROBE = r"""
#include <stdio.h>
#include <stddef.h>
#include "hxsim.h"
#define F(T, f) printf(#T "." #f " %zu %zu\n", offsetof(T, f), sizeof(((T*)0)->f));
#define S(T) printf(#T " %zu\n", sizeof(T));
int main(void) {
  S(hx_trace) F(hx_trace, n_queries) F(hx_trace, arrival_us) F(hx_trace, retry) F(hx_trace, tenant)
  S(hx_cluster) F(hx_cluster, n_inst) F(hx_cluster, inst_type) F(hx_cluster, slo_mult_fp) F(hx_cluster, rmax)
  F(hx_cluster, stage_ref_out) F(hx_cluster, n_faults) F(hx_cluster, tenant_slo_mult_fp)
  F(hx_cluster, timeout_mult_fp) F(hx_cluster, faults)
  S(hx_fault) F(hx_fault, t0_us) F(hx_fault, slow_fp)
  S(hx_extra) F(hx_extra, n_done) F(hx_extra, reissued) F(hx_extra, p95_us)
  S(hx_grid) F(hx_grid, alpha_fp) F(hx_grid, dispatch_policy)
  S(hx_options) F(hx_options, record_sims) F(hx_options, timing) F(hx_options, force_generic)
  F(hx_options, n_subset) F(hx_options, sim_subset) F(hx_options, checked) F(hx_options, arena_entries)
  S(hx_result) F(hx_result, digest) F(hx_result, status) F(hx_result, cycles_k)
  S(hx_best) F(hx_best, global_sum_p95) F(hx_best, per_trace_point)
  S(hx_info) F(hx_info, resident_warps) F(hx_info, smem_per_block) F(hx_info, generic_kernel)
  return 0;
}
"""


def test_struct_layout_matches_binding(tmp_path):
    src = tmp_path / "probe.c"
    src.write_text(_PROBE)
    exe = tmp_path / "probe"
    subprocess.check_call(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)])
    got = {}
    for line in subprocess.check_output([str(exe)], text=True).splitlines():
        parts = line.split()
        got[parts[0]] = tuple(int(x) for x in parts[1:])
    structs = {"hx_trace": H.hx_trace, "hx_cluster": H.hx_cluster, "hx_grid": H.hx_grid,
               "hx_options": H.hx_options, "hx_best": H.hx_best, "hx_info": H.hx_info, "hx_fault": H.hx_fault}
    for key, val in got.items():
        if "." in key:
            sname, field = key.split(".")
            if sname == "hx_result":
                assert H.RESULT_DTYPE.fields[field][1] == val[0]
                continue
            if sname == "hx_extra":
                assert H.EXTRA_DTYPE.fields[field][1] == val[0]
                continue
            ct = structs[sname]
            assert getattr(ct, field).offset == val[0], key
            assert getattr(ct, field).size == val[1], key
        elif key == "hx_result":
            assert H.RESULT_DTYPE.itemsize == val[0]
        elif key == "hx_extra":
            assert H.EXTRA_DTYPE.itemsize == val[0]
        else:
            assert ctypes.sizeof(structs[key]) == val[0], key


def _create(lib, traces, cluster, grid, opt=None):
    t = H._Traces(traces)
    hc, keep = H._cluster_struct(cluster)
    g = grid
    gc = [np.ascontiguousarray(g.alpha_fp, np.int64), np.ascontiguousarray(g.gamma_fp, np.int64),
          np.ascontiguousarray(g.rho, np.int32), np.ascontiguousarray(g.beta_us2, np.int64),
          np.ascontiguousarray(g.local_policy, np.uint8), np.ascontiguousarray(g.dispatch_policy, np.uint8)]
    hg = H.hx_grid(len(gc[0]), *[H._p(x) for x in gc])
    h = ctypes.c_void_p()
    rc = lib.hx_sim_create(t.arr, len(traces), ctypes.byref(hc), ctypes.byref(hg),
                           None if opt is None else ctypes.byref(opt), ctypes.byref(h))
    return rc, lib.hx_last_error().decode(), h


def _copy_trace(tr):
    return W.Trace(*[getattr(tr, f).copy() for f in ("arrival_us", "k", "call_base", "prompt", "out", "out_est",
                                                      "stage", "cand", "retry")])


def test_rejects_malformed_inputs_without_device_work(lib):
    wl = W.make_workload(0, n_queries=20)
    tr = wl.traces[0]
    cases = []
    t1 = _copy_trace(tr)
    t1.arrival_us[3] = t1.arrival_us[2] - 1
    cases.append(("unsorted arrivals", [t1], wl.cluster, wl.grid, "sorted"))
    t2 = _copy_trace(tr)
    t2.stage[1] = W.STAGE_E
    cases.append(("broken workflow", [t2], wl.cluster, wl.grid, "S must be followed"))
    t3 = _copy_trace(tr)
    t3.prompt[0] = 0
    cases.append(("zero prompt", [t3], wl.cluster, wl.grid, "token"))
    t4 = _copy_trace(tr)
    t4.k[0] = 9
    cases.append(("k > 8", [t4], wl.cluster, wl.grid, "k must be"))
    g = W.Grid(wl.grid.alpha_fp.copy(), wl.grid.gamma_fp.copy(), wl.grid.rho.copy(), wl.grid.beta_us2.copy(),
               wl.grid.local_policy.copy(), wl.grid.dispatch_policy.copy())
    g.alpha_fp[0] = W.SCALE + 1
    cases.append(("alpha > 1", [tr], wl.cluster, g, "alpha"))
    c = wl.cluster
    c2 = W.Cluster(c.prefill_tok_s, c.decode_us_tok, np.array([8, 17], np.int32), c.inst_type, c.ref_type,
                   c.slo_mult_fp, c.rmax, c.stage_ref_prompt, c.stage_ref_out)
    cases.append(("17 slots", [tr], c2, wl.grid, "slots"))
    c3 = W.Cluster(c.prefill_tok_s, c.decode_us_tok, c.slots, np.zeros(65, np.uint8), c.ref_type, c.slo_mult_fp,
                   c.rmax, c.stage_ref_prompt, c.stage_ref_out)
    cases.append(("65 instances", [tr], c3, wl.grid, "n_inst"))
    t5 = _copy_trace(tr)
    t5.arrival_us[:] += 1 << 40
    cases.append(("horizon", [t5], wl.cluster, wl.grid, "horizon"))
    t6 = _copy_trace(tr)
    t6.tenant = np.full(tr.n_queries, 2, np.uint8)
    c6 = W.Cluster(c.prefill_tok_s, c.decode_us_tok, c.slots, c.inst_type, c.ref_type, c.slo_mult_fp, c.rmax,
                   c.stage_ref_prompt, c.stage_ref_out, np.array([W.SCALE, 2 * W.SCALE], np.int64))
    cases.append(("tenant 2 of 2", [t6], c6, wl.grid, "tenant out of range"))
    t7 = _copy_trace(tr)
    t7.k[0] = 0
    cases.append(("k = 0 with a whole workflow", [t7], wl.cluster, wl.grid, "single E call"))

    def faulty(faults, timeout):
        f = np.zeros(len(faults), W.FAULT_DTYPE)
        for j, x in enumerate(faults):
            f[j] = (x[0], 0, x[1], x[2], x[3])
        return W.Cluster(c.prefill_tok_s, c.decode_us_tok, c.slots, c.inst_type, c.ref_type, c.slo_mult_fp, c.rmax,
                         c.stage_ref_prompt, c.stage_ref_out, None, timeout, f)
    cases.append(("stopped without timeout", [tr], faulty([(0, 0, 100, 0)], 0), wl.grid, "needs a timeout"))
    cases.append(("fault instance", [tr], faulty([(4, 0, 100, W.SCALE)], 0), wl.grid, "fault instance"))
    cases.append(("fault window", [tr], faulty([(0, 100, 50, W.SCALE)], 0), wl.grid, "fault window"))
    cases.append(("timeout < 1", [tr], faulty([(0, 0, 100, 0)], W.SCALE // 2), wl.grid, "timeout_mult_fp"))
    for name, trs, cl, gr, msg in cases:
        rc, err, h = _create(lib, trs, cl, gr)
        assert rc == H.HX_ERR_INVALID, name
        assert msg in err, (name, err)
        assert not h.value


def test_parallel_validation_names_the_first_bad_trace(lib):
    # about half a million calls: the traces are validated on several host
    # threads, and the error still names the lowest-numbered bad trace
    wl = W.make_workload(4, n_traces=8, n_queries=8000)
    trs = [_copy_trace(t) for t in wl.traces]
    trs[5].prompt[3] = 0
    trs[2].arrival_us[4] = trs[2].arrival_us[3] - 1
    trs[7].k[1] = 9
    rc, err, h = _create(lib, trs, wl.cluster, wl.grid)
    assert rc == H.HX_ERR_INVALID and err.startswith("trace 2:") and "sorted" in err, err
    assert not h.value
    trs[2] = _copy_trace(wl.traces[2])
    rc, err, h = _create(lib, trs, wl.cluster, wl.grid)
    assert rc == H.HX_ERR_INVALID and err.startswith("trace 5:") and "token" in err, err


def test_horizon_limit_is_exact(lib):
    # without fault windows the horizon is the sum over calls of
    # ceil(prompt * 10^6 / min prefill rate) + max(out, out_est) * max decode
    # time, plus the last arrival; 2^39 us is allowed, one more is not
    wl = W.make_workload(0, n_queries=20)
    c, tr = wl.cluster, wl.traces[0]
    mp, md = int(np.min(c.prefill_tok_s)), int(np.max(c.decode_us_tok))
    hz = sum(-(-int(p) * 10 ** 6 // mp) + max(int(o), int(oe)) * md
             for p, o, oe in zip(tr.prompt, tr.out, tr.out_est))
    for extra, accepted in ((0, True), (1, False)):
        t = _copy_trace(tr)
        t.arrival_us += (1 << 39) - hz - int(tr.arrival_us[-1]) + extra
        rc, err, h = _create(lib, [t], c, wl.grid)
        if accepted:
            assert rc != H.HX_ERR_INVALID, err  # validation passed (HX_ERR_CUDA without a GPU)
            if h.value:
                lib.hx_sim_destroy(h)
        else:
            assert rc == H.HX_ERR_INVALID and "horizon" in err, err


def test_rejects_bad_options(lib):
    wl = W.make_workload(0, n_queries=20)  # 1 trace x 16 points

    def opt(subset=None, n=None, checked=0, arena=0, record=None, n_record=None):
        arr = np.asarray(subset if subset else [0], np.int32)
        rec = np.asarray(record if record else [0], np.int32)
        o = H.hx_options(len(record or []) if n_record is None else n_record,
                         None if record is None else H._p(rec), 0, 0, 0,
                         len(subset or []) if n is None else n,
                         None if subset is None else H._p(arr), checked, arena)
        return o, (arr, rec)
    for name, (o, keep), msg in [("out of range", opt([3, 16]), "out of range"),
                                 ("negative index", opt([-1]), "out of range"),
                                 ("twice", opt([5, 2, 5]), "twice"),
                                 ("negative count", opt([1], n=-1), "n_subset"),
                                 ("NULL subset", opt(None, n=2), "NULL"),
                                 ("checked = 2", opt(None, n=0, checked=2), "checked"),
                                 ("negative arena", opt(None, n=0, arena=-1), "arena_entries"),
                                 ("record out of range", opt(None, n=0, record=[16]), "record_sims"),
                                 ("record twice", opt(None, n=0, record=[3, 3]), "record_sims"),
                                 ("negative n_record", opt(None, n=0, n_record=-1), "n_record")]:
        rc, err, h = _create(lib, wl.traces, wl.cluster, wl.grid, o)
        assert rc == H.HX_ERR_INVALID, name
        assert msg in err, (name, err)
        assert not h.value


def test_null_safety(lib):
    assert lib.hx_sim_destroy(None) == H.HX_OK
    assert lib.hx_sim_run(None, None) == H.HX_ERR_INVALID
    assert lib.hx_sim_results(None, None, 0) == H.HX_ERR_INVALID
    assert lib.hx_last_error().decode() != ""


def test_missing_library_fails_loudly(tmp_path):
    with pytest.raises(ImportError):
        H.load(str(tmp_path / "nope.so"))
