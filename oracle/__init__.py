"""CPU oracle of the batched HexGen-Flow scheduler simulation.

TEST INFRASTRUCTURE ONLY: the plain single-threaded C simulator in
`hx_oracle.c`, loaded through ctypes.  It is what the CUDA library is checked
against, bit for bit.  Only the tests, `__graft_entry__.smoke()` and the CPU
baseline leg of `bench.py` may import it; the library itself never does.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Dict, Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "hx_oracle.c")
_LIB = os.path.join(_HERE, "libhxoracle.so")

RESULT_DTYPE = np.dtype([("p95_us", "<i8"), ("makespan_us", "<i8"), ("events", "<i8"),
                         ("digest", "<u8"), ("slo_met", "<i4"), ("n_done", "<i4"),
                         ("status", "<i4"), ("pad", "<i4")])
EXTRA_DTYPE = np.dtype([("slo_met", "<i4", (4,)), ("n_done", "<i4", (4,)), ("reissued", "<i4"), ("pad", "<i4"),
                        ("p95_us", "<i8", (4,))])
FAULT_DTYPE = np.dtype([("inst", "<i4"), ("pad", "<i4"), ("t0_us", "<i8"), ("t1_us", "<i8"), ("slow_fp", "<i8")])


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (plain C, no vector or fast-math flags)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < max(
            os.path.getmtime(_SRC), os.path.getmtime(os.path.join(_HERE, "hx_oracle.h"))):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off",
                               "-Wall", "-o", tmp, _SRC])
        os.replace(tmp, _LIB)
    return _LIB


class _Trace(ctypes.Structure):
    _fields_ = [("n_queries", ctypes.c_int32), ("n_calls", ctypes.c_int32),
                ("arrival_us", ctypes.c_void_p), ("k", ctypes.c_void_p), ("call_base", ctypes.c_void_p),
                ("prompt", ctypes.c_void_p), ("out", ctypes.c_void_p), ("out_est", ctypes.c_void_p),
                ("stage", ctypes.c_void_p), ("cand", ctypes.c_void_p), ("retry", ctypes.c_void_p),
                ("tenant", ctypes.c_void_p)]


class _Cluster(ctypes.Structure):
    _fields_ = [("n_types", ctypes.c_int32), ("prefill_tok_s", ctypes.c_void_p),
                ("decode_us_tok", ctypes.c_void_p), ("slots", ctypes.c_void_p),
                ("n_inst", ctypes.c_int32), ("inst_type", ctypes.c_void_p), ("ref_type", ctypes.c_int32),
                ("slo_mult_fp", ctypes.c_int64), ("rmax", ctypes.c_int32),
                ("stage_ref_prompt", ctypes.c_void_p), ("stage_ref_out", ctypes.c_void_p),
                ("n_tenants", ctypes.c_int32), ("n_faults", ctypes.c_int32),
                ("tenant_slo_mult_fp", ctypes.c_void_p), ("timeout_mult_fp", ctypes.c_int64),
                ("faults", ctypes.c_void_p)]


class _Log(ctypes.Structure):
    _fields_ = [("inst", ctypes.c_void_p), ("enq", ctypes.c_void_p), ("budget", ctypes.c_void_p),
                ("start", ctypes.c_void_p), ("end", ctypes.c_void_p)]


class _Point(ctypes.Structure):
    _fields_ = [("alpha_fp", ctypes.c_int64), ("gamma_fp", ctypes.c_int64), ("beta_us2", ctypes.c_int64),
                ("rho", ctypes.c_int32), ("local_policy", ctypes.c_int32),
                ("dispatch_policy", ctypes.c_int32)]


_lib = None


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        lib.hxo_prep.restype = ctypes.c_int
        lib.hxo_simulate.restype = ctypes.c_int
        lib.hxo_budget.restype = ctypes.c_int64
        lib.hxo_budget.argtypes = [ctypes.c_int64] * 4
        lib.hxo_score.restype = ctypes.c_int64
        lib.hxo_score.argtypes = [ctypes.c_int64] * 4
        lib.hxo_pick.restype = ctypes.c_int32
        lib.hxo_pick.argtypes = [ctypes.c_int32, ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p,
                                 ctypes.c_void_p]
        lib.hxo_best.restype = ctypes.c_int
        _lib = lib
    return _lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


class _Marshal:
    """Keeps the contiguous copies alive while the C structs point at them."""

    def __init__(self, trace, cluster):
        t = trace
        self.t = [_c(t.arrival_us, np.int64), _c(t.k, np.uint8), _c(t.call_base, np.int32),
                  _c(t.prompt, np.int32), _c(t.out, np.int32), _c(t.out_est, np.int32),
                  _c(t.stage, np.uint8), _c(t.cand, np.uint8), _c(t.retry, np.uint8)]
        ten = getattr(t, "tenant", None)
        self.tenant = None if ten is None else _c(ten, np.uint8)
        self.trace = _Trace(int(self.t[0].shape[0]), int(self.t[3].shape[0]), *[_ptr(a) for a in self.t],
                            None if self.tenant is None else _ptr(self.tenant))
        c = cluster
        self.c = [_c(c.prefill_tok_s, np.int32), _c(c.decode_us_tok, np.int32), _c(c.slots, np.int32),
                  _c(c.inst_type, np.uint8), _c(c.stage_ref_prompt, np.int32), _c(c.stage_ref_out, np.int32)]
        tm = getattr(c, "tenant_slo_mult_fp", None)
        self.tmult = None if tm is None else _c(tm, np.int64)
        fl = getattr(c, "faults", None)
        self.faults = np.zeros(0, FAULT_DTYPE) if fl is None else np.ascontiguousarray(fl, dtype=FAULT_DTYPE)
        self.cluster = _Cluster(int(self.c[0].shape[0]), _ptr(self.c[0]), _ptr(self.c[1]), _ptr(self.c[2]),
                                int(self.c[3].shape[0]), _ptr(self.c[3]), int(c.ref_type),
                                int(c.slo_mult_fp), int(c.rmax), _ptr(self.c[4]), _ptr(self.c[5]),
                                1 if self.tmult is None else int(self.tmult.shape[0]), int(self.faults.shape[0]),
                                None if self.tmult is None else _ptr(self.tmult),
                                int(getattr(c, "timeout_mult_fp", 0)),
                                _ptr(self.faults) if self.faults.shape[0] else None)


def point_of(grid, p: int) -> Dict[str, int]:
    return dict(alpha_fp=int(grid.alpha_fp[p]), gamma_fp=int(grid.gamma_fp[p]),
                beta_us2=int(grid.beta_us2[p]), rho=int(grid.rho[p]),
                local_policy=int(grid.local_policy[p]), dispatch_policy=int(grid.dispatch_policy[p]))


def prep(trace, cluster) -> Dict[str, np.ndarray]:
    """Eq. (comp) per call and type, t-bar per call, SLO per query, stage reference costs."""
    lib = _load()
    m = _Marshal(trace, cluster)
    T = cluster.n_types
    nc, nq = trace.n_calls, trace.n_queries
    est = np.zeros(max(nc, 1) * T, np.int64)
    svc = np.zeros(max(nc, 1) * T, np.int64)
    tbar = np.zeros(max(nc, 1), np.int64)
    tslo = np.zeros(max(nq, 1), np.int64)
    cref = np.zeros(4, np.int64)
    st = lib.hxo_prep(ctypes.byref(m.trace), ctypes.byref(m.cluster), _ptr(est), _ptr(svc), _ptr(tbar),
                      _ptr(tslo), _ptr(cref))
    if st != 0:
        raise ValueError(f"oracle prep rejected the input (status {st})")
    return dict(est=est[:nc * T].reshape(nc, T), svc=svc[:nc * T].reshape(nc, T), tbar=tbar[:nc],
                t_slo=tslo[:nq], stage_ref_cost=cref)


def simulate(trace, cluster, point: Dict[str, int], check: bool = False, log: bool = False,
             extra: bool = False):
    """One simulation.  Returns the result record, then the per-call logs if
    `log`, then the per-tenant counts and re-issues (EXTRA_DTYPE) if `extra`."""
    lib = _load()
    m = _Marshal(trace, cluster)
    pt = _Point(point["alpha_fp"], point["gamma_fp"], point["beta_us2"], point["rho"],
                point["local_policy"], point["dispatch_policy"])
    res = np.zeros(1, RESULT_DTYPE)
    ext = np.zeros(1, EXTRA_DTYPE)
    if not log:
        lib.hxo_simulate(ctypes.byref(m.trace), ctypes.byref(m.cluster), ctypes.byref(pt), int(check),
                         _ptr(res), None, _ptr(ext))
        return (res[0], ext[0]) if extra else res[0]
    nc = max(trace.n_calls, 1)
    arrs = dict(inst=np.full(nc, -1, np.int32), enq=np.full(nc, -1, np.int64),
                budget=np.zeros(nc, np.int64), start=np.full(nc, -1, np.int64),
                end=np.full(nc, -1, np.int64))
    lg = _Log(*[_ptr(arrs[k]) for k in ("inst", "enq", "budget", "start", "end")])
    lib.hxo_simulate(ctypes.byref(m.trace), ctypes.byref(m.cluster), ctypes.byref(pt), int(check),
                     _ptr(res), ctypes.byref(lg), _ptr(ext))
    n = trace.n_calls
    logs = {k: v[:n] for k, v in arrs.items()}
    return (res[0], logs, ext[0]) if extra else (res[0], logs)


def _run_one(args):
    trace, cluster, point, check, extra = args
    return simulate(trace, cluster, point, check=check, extra=extra)


def run(workload, sims: Optional[Sequence[int]] = None, procs: int = 1, check: bool = False,
        extra: bool = False):
    """Simulate the listed sims (index = trace * P + point) of a workload;
    with `extra`, also return their per-tenant counts (EXTRA_DTYPE).

    With procs > 1 the sims run in a process pool started with `spawn`.
    """
    P = workload.grid.n_points
    if sims is None:
        sims = range(len(workload.traces) * P)
    jobs = [(workload.traces[s // P], workload.cluster, point_of(workload.grid, s % P), check, extra) for s in sims]
    if procs <= 1 or len(jobs) <= 1:
        out = [_run_one(j) for j in jobs]
    else:
        import multiprocessing as mp
        ctx = mp.get_context("spawn")
        with ctx.Pool(procs) as pool:
            out = pool.map(_run_one, jobs, chunksize=max(1, len(jobs) // (4 * procs)))
    res = np.zeros(len(jobs), RESULT_DTYPE)
    ext = np.zeros(len(jobs), EXTRA_DTYPE)
    for i, r in enumerate(out):
        if extra:
            res[i], ext[i] = r
        else:
            res[i] = r
    return (res, ext) if extra else res


def budget(t_slo: int, elapsed: int, tbar: int, remaining: int) -> int:
    return int(_load().hxo_budget(t_slo, elapsed, tbar, remaining))


def score(alpha_fp: int, beta_us2: int, t_queue: int, t_comp: int) -> int:
    return int(_load().hxo_score(alpha_fp, beta_us2, t_queue, t_comp))


def pick(policy: int, rid: Sequence[int], urgency_fp: Sequence[int], enq_us: Sequence[int]) -> int:
    r = _c(rid, np.int32)
    u = _c(urgency_fp, np.int64)
    e = _c(enq_us, np.int64)
    return int(_load().hxo_pick(int(policy), int(r.shape[0]), _ptr(r), _ptr(u), _ptr(e)))


def best(results: np.ndarray, n_traces: int, n_points: int, n_queries: Sequence[int], objective: int):
    """(global point, global sum of P95, per-trace points) of Sec. 4.3's argmin."""
    lib = _load()
    res = np.ascontiguousarray(results)
    if res.dtype != RESULT_DTYPE:
        if res.dtype.itemsize != RESULT_DTYPE.itemsize:
            raise ValueError("result records must be 48 bytes")
        res = res.view(RESULT_DTYPE)
    nq = _c(n_queries, np.int32)
    gp = ctypes.c_int32(0)
    gs = ctypes.c_int64(0)
    per = np.zeros(max(n_traces, 1), np.int32)
    st = lib.hxo_best(_ptr(res), ctypes.c_int32(n_traces), ctypes.c_int32(n_points), _ptr(nq),
                      ctypes.c_int32(objective), ctypes.byref(gp), ctypes.byref(gs), _ptr(per))
    if st != 0:
        raise ValueError(f"oracle best rejected the input (status {st})")
    return int(gp.value), int(gs.value), per[:n_traces].copy()
