"""Python binding of libhxsim.so (include/hxsim.h): argument marshalling only.

Every step of the simulation runs in the library's CUDA kernels; this module
packs numpy arrays into the C structs, passes a CUDA stream, and unpacks the
results.  There is no CPU fallback: if the library is missing, loading fails.

    sim = Sim(traces, cluster, grid)
    sim.run()                      # on torch's current CUDA stream
    res = sim.results()            # numpy structured array, one row per sim
    point, sum_p95, slo, per_trace = sim.best(OBJ_P95)
"""
from __future__ import annotations

import ctypes
import os
import re
from typing import Optional, Sequence

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libhxsim.so")
# the same library built with every simulation-kernel index range-checked
# (-DHX_CHECKED): a failed check is the per-simulation status HX_ERR_BOUNDS
LIB_CHECKED_PATH = os.path.join(_PKG, "libhxsim_checked.so")
HEADER = os.path.join(os.path.dirname(_PKG), "include", "hxsim.h")

(HX_OK, HX_ERR_INVALID, HX_ERR_CUDA, HX_ERR_OOM, HX_ERR_CAPACITY, HX_ERR_STEP_LIMIT, HX_ERR_STATE,
 HX_ERR_INVARIANT, HX_SKIPPED, HX_ERR_BOUNDS) = range(10)
OBJ_P95, OBJ_P95_SLO95 = 0, 1

RESULT_DTYPE = np.dtype([("p95_us", "<i8"), ("makespan_us", "<i8"), ("events", "<i8"),
                         ("digest", "<u8"), ("slo_met", "<i4"), ("n_done", "<i4"),
                         ("status", "<i4"), ("cycles_k", "<i4")])
EXTRA_DTYPE = np.dtype([("slo_met", "<i4", (4,)), ("n_done", "<i4", (4,)), ("reissued", "<i4"), ("pad", "<i4"),
                        ("p95_us", "<i8", (4,))])


class HxError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"hxsim error {code}: {msg}")
        self.code = code


class hx_trace(ctypes.Structure):
    _fields_ = [("n_queries", ctypes.c_int32), ("n_calls", ctypes.c_int32),
                ("arrival_us", ctypes.c_void_p), ("k", ctypes.c_void_p), ("call_base", ctypes.c_void_p),
                ("prompt", ctypes.c_void_p), ("out", ctypes.c_void_p), ("out_est", ctypes.c_void_p),
                ("stage", ctypes.c_void_p), ("cand", ctypes.c_void_p), ("retry", ctypes.c_void_p),
                ("tenant", ctypes.c_void_p)]


class hx_fault(ctypes.Structure):
    _fields_ = [("inst", ctypes.c_int32), ("pad", ctypes.c_int32), ("t0_us", ctypes.c_int64),
                ("t1_us", ctypes.c_int64), ("slow_fp", ctypes.c_int64)]


class hx_cluster(ctypes.Structure):
    _fields_ = [("n_types", ctypes.c_int32), ("prefill_tok_s", ctypes.c_void_p),
                ("decode_us_tok", ctypes.c_void_p), ("slots", ctypes.c_void_p), ("n_inst", ctypes.c_int32),
                ("inst_type", ctypes.c_void_p), ("ref_type", ctypes.c_int32), ("slo_mult_fp", ctypes.c_int64),
                ("rmax", ctypes.c_int32), ("stage_ref_prompt", ctypes.c_void_p),
                ("stage_ref_out", ctypes.c_void_p), ("n_tenants", ctypes.c_int32), ("n_faults", ctypes.c_int32),
                ("tenant_slo_mult_fp", ctypes.c_void_p), ("timeout_mult_fp", ctypes.c_int64),
                ("faults", ctypes.c_void_p)]


class hx_grid(ctypes.Structure):
    _fields_ = [("n_points", ctypes.c_int32), ("alpha_fp", ctypes.c_void_p), ("gamma_fp", ctypes.c_void_p),
                ("rho", ctypes.c_void_p), ("beta_us2", ctypes.c_void_p), ("local_policy", ctypes.c_void_p),
                ("dispatch_policy", ctypes.c_void_p)]


class hx_options(ctypes.Structure):
    _fields_ = [("n_record", ctypes.c_int32), ("record_sims", ctypes.c_void_p),
                ("max_resident_warps", ctypes.c_int32), ("timing", ctypes.c_int32),
                ("force_generic", ctypes.c_int32), ("n_subset", ctypes.c_int32), ("sim_subset", ctypes.c_void_p),
                ("checked", ctypes.c_int32), ("arena_entries", ctypes.c_int32)]


class hx_best(ctypes.Structure):
    _fields_ = [("global_point", ctypes.c_int32), ("pad", ctypes.c_int32), ("global_sum_p95", ctypes.c_int64),
                ("global_slo_met", ctypes.c_int64), ("per_trace_point", ctypes.c_void_p)]


class hx_info(ctypes.Structure):
    _fields_ = [("n_sims", ctypes.c_int64), ("n_calls_total", ctypes.c_int64),
                ("n_queries_total", ctypes.c_int64), ("scratch_bytes", ctypes.c_int64),
                ("device_bytes", ctypes.c_int64), ("resident_warps", ctypes.c_int32),
                ("warps_per_block", ctypes.c_int32), ("blocks", ctypes.c_int32),
                ("smem_per_block", ctypes.c_int32), ("generic_kernel", ctypes.c_int32),
                ("work_order", ctypes.c_int32)]


_lib = None


def declared_functions() -> list:
    """Names of the functions include/hxsim.h declares."""
    with open(HEADER) as f:
        text = f.read()
    return sorted(set(re.findall(r"^\s*(?:int|const char\s*\*)\s+(hx_\w+)\s*\(", text, re.M)))


_lib_checked = None


def load_checked():
    """Load the bounds-checked build libhxsim_checked.so; raises if it has not been built."""
    global _lib_checked
    if _lib_checked is None:
        _lib_checked = load(LIB_CHECKED_PATH)
    return _lib_checked


def load(path: Optional[str] = None):
    """Load libhxsim.so (or the library at `path`); raises if it has not been built."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise ImportError(f"{p} is missing: build it with `python -m paper_2505_05286_gb300.build`")
    lib = ctypes.CDLL(p)
    vp, i32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
    lib.hx_last_error.restype = ctypes.c_char_p
    lib.hx_last_error.argtypes = []
    for name, args in [("hx_sim_create", [vp, i32, vp, vp, vp, vp]), ("hx_sim_upload", [vp, vp, i32, vp]),
                       ("hx_sim_run", [vp, vp]), ("hx_sim_results", [vp, vp, sz]),
                       ("hx_sim_best", [vp, i32, vp]), ("hx_sim_records", [vp, i32, vp, vp, vp, vp, vp, sz]),
                       ("hx_sim_prep", [vp, i32, vp, vp, vp, vp, sz]), ("hx_sim_timings", [vp, vp, vp, vp]),
                       ("hx_sim_timings_back", [vp, i32, vp, vp, vp]),
                       ("hx_sim_info", [vp, vp]), ("hx_sim_destroy", [vp]),
                       ("hx_sim_run_static", [vp, vp, vp, i32, vp, vp, vp]),
                       ("hx_selftest_div", [vp, vp, vp, vp, sz]),
                       ("hx_sim_point_sums", [vp, vp, vp, vp, sz]), ("hx_sim_extras", [vp, vp, sz]),
                       ("hx_best_of_sums", [vp, vp, vp, i32, ctypes.c_int64, i32, vp])]:
        fn = getattr(lib, name)
        fn.restype = ctypes.c_int
        fn.argtypes = args
    if path is None:
        _lib = lib
    return lib


def _check(lib, code: int):
    if code != HX_OK:
        raise HxError(code, lib.hx_last_error().decode())


def _p(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


def _stream_handle(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


class _Traces:
    """Contiguous copies of the trace arrays and the hx_trace array pointing at them."""

    def __init__(self, traces):
        self.keep = []
        self.arr = (hx_trace * len(traces))()
        for i, t in enumerate(traces):
            cols = [_c(t.arrival_us, np.int64), _c(t.k, np.uint8), _c(t.call_base, np.int32),
                    _c(t.prompt, np.int32), _c(t.out, np.int32), _c(t.out_est, np.int32),
                    _c(t.stage, np.uint8), _c(t.cand, np.uint8), _c(t.retry, np.uint8)]
            ten = getattr(t, "tenant", None)
            cols.append(None if ten is None else _c(ten, np.uint8))
            self.keep.append(cols)
            self.arr[i] = hx_trace(int(cols[0].shape[0]), int(cols[3].shape[0]), *[_p(x) for x in cols])


def selftest_div(n: np.ndarray, d: np.ndarray):
    """(library quotients, compiler quotients) of n // d on the current device."""
    lib = load()
    n = _c(n, np.uint64)
    d = _c(d, np.uint64)
    q = np.zeros_like(n)
    qr = np.zeros_like(n)
    _check(lib, lib.hx_selftest_div(_p(n), _p(d), _p(q), _p(qr), int(n.shape[0])))
    return q, qr


def best_of_sums(sum_p95, sum_slo_met, n_failed, n_queries_total: int, objective: int = OBJ_P95):
    """Best point from per-point sums gathered over several handles or ranks."""
    lib = load()
    a, b, c = _c(sum_p95, np.int64), _c(sum_slo_met, np.int64), _c(n_failed, np.int32)
    best = hx_best(0, 0, 0, 0, None)
    _check(lib, lib.hx_best_of_sums(_p(a), _p(b), _p(c), int(a.shape[0]), int(n_queries_total), int(objective),
                                    ctypes.byref(best)))
    return int(best.global_point), int(best.global_sum_p95), int(best.global_slo_met)


def _cluster_struct(c):
    cols = [_c(c.prefill_tok_s, np.int32), _c(c.decode_us_tok, np.int32), _c(c.slots, np.int32),
            _c(c.inst_type, np.uint8), _c(c.stage_ref_prompt, np.int32), _c(c.stage_ref_out, np.int32)]
    tm = getattr(c, "tenant_slo_mult_fp", None)
    tm = None if tm is None else _c(tm, np.int64)
    fl = getattr(c, "faults", None)
    n_f = 0 if fl is None else len(fl)
    faults = (hx_fault * max(n_f, 1))()
    for j in range(n_f):
        f = fl[j]
        faults[j] = hx_fault(int(f["inst"]), 0, int(f["t0_us"]), int(f["t1_us"]), int(f["slow_fp"]))
    cols += [tm, faults]
    st = hx_cluster(int(cols[0].shape[0]), _p(cols[0]), _p(cols[1]), _p(cols[2]), int(cols[3].shape[0]),
                    _p(cols[3]), int(c.ref_type), int(c.slo_mult_fp), int(c.rmax), _p(cols[4]), _p(cols[5]),
                    0 if tm is None else int(tm.shape[0]), n_f, _p(tm), int(getattr(c, "timeout_mult_fp", 0)),
                    ctypes.cast(faults, ctypes.c_void_p) if n_f else None)
    return st, cols


def _grid_struct(g):
    cols = [_c(g.alpha_fp, np.int64), _c(g.gamma_fp, np.int64), _c(g.rho, np.int32), _c(g.beta_us2, np.int64),
            _c(g.local_policy, np.uint8), _c(g.dispatch_policy, np.uint8)]
    return hx_grid(int(cols[0].shape[0]), *[_p(x) for x in cols]), cols


def run_static(trace, cluster, grid, objective: int = OBJ_P95, stream=None):
    """hx_sim_run_static: one trace through the whole path with no memory
    allocation (the library's fixed device array holds every intermediate).
    Returns (results, (best point, its P95, its SLO count))."""
    lib = load()
    tr = _Traces([trace])
    hc, keep_c = _cluster_struct(cluster)
    hg, keep_g = _grid_struct(grid)
    res = np.zeros(int(grid.alpha_fp.shape[0]), RESULT_DTYPE)
    best = hx_best(0, 0, 0, 0, None)
    _check(lib, lib.hx_sim_run_static(ctypes.cast(tr.arr, ctypes.c_void_p), ctypes.byref(hc), ctypes.byref(hg),
                                      int(objective), _p(res), ctypes.byref(best), _stream_handle(stream)))
    return res, (int(best.global_point), int(best.global_sum_p95), int(best.global_slo_met))


class Sim:
    """A set of (trace x point) simulations resident on the current CUDA device."""

    def __init__(self, traces, cluster, grid, record_sims: Sequence[int] = (), timing: bool = False,
                 max_resident_warps: int = 0, force_generic: bool = False, subset: Optional[Sequence[int]] = None,
                 checked: bool = False, arena_entries: int = 0, bounds_checked: bool = False):
        """`subset`: run only these simulations (index trace * P + point); the
        others report HX_SKIPPED.  `checked`: also check the scheduler's
        invariants after every event (per-sim status HX_ERR_INVARIANT).
        `arena_entries` (testing) caps each warp's local-queue arena.
        `bounds_checked`: run on the bounds-checked build of the library
        (per-sim status HX_ERR_BOUNDS if an index check fails)."""
        self.lib = load_checked() if bounds_checked else load()
        self.n_traces = len(traces)
        self.n_points = int(grid.alpha_fp.shape[0])
        self.n_calls = [int(t.prompt.shape[0]) for t in traces]
        self.n_queries = [int(t.arrival_us.shape[0]) for t in traces]
        tr = _Traces(traces)
        hc, keep_c = _cluster_struct(cluster)
        hg, keep_g = _grid_struct(grid)
        self.record_sims = [int(s) for s in record_sims]
        rs = _c(self.record_sims if self.record_sims else [0], np.int32)
        self.subset = None if subset is None else [int(s) for s in subset]
        ss = _c(self.subset if self.subset else [0], np.int32)
        opt = hx_options(len(self.record_sims), _p(rs), int(max_resident_warps), int(bool(timing)),
                         int(bool(force_generic)), len(self.subset or []), _p(ss), int(bool(checked)),
                         int(arena_entries))
        h = ctypes.c_void_p()
        _check(self.lib, self.lib.hx_sim_create(tr.arr, self.n_traces, ctypes.byref(hc), ctypes.byref(hg),
                                                ctypes.byref(opt), ctypes.byref(h)))
        self.h = h

    @property
    def n_sims(self) -> int:
        return self.n_traces * self.n_points

    def upload(self, traces, stream=None):
        tr = _Traces(traces)
        _check(self.lib, self.lib.hx_sim_upload(self.h, tr.arr, len(traces), _stream_handle(stream)))

    def run(self, stream=None):
        _check(self.lib, self.lib.hx_sim_run(self.h, _stream_handle(stream)))

    def results(self, out: Optional[np.ndarray] = None) -> np.ndarray:
        """One RESULT_DTYPE row per simulation; `out` (e.g. pinned host memory)
        receives them when given."""
        if out is None:
            out = np.zeros(self.n_sims, RESULT_DTYPE)
        elif out.dtype != RESULT_DTYPE or out.shape[0] < self.n_sims or not out.flags["C_CONTIGUOUS"]:
            raise ValueError("out must be a contiguous RESULT_DTYPE array with a row per simulation")
        _check(self.lib, self.lib.hx_sim_results(self.h, _p(out), self.n_sims))
        return out

    def results_tensors(self) -> dict:
        """The results as one torch tensor per field (int64 / int32 / the
        digest's 64 bits as int64), indexed by simulation."""
        import torch
        r = self.results()
        return {f: torch.from_numpy(np.ascontiguousarray(r[f]).view(np.int64) if f == "digest"
                                    else np.ascontiguousarray(r[f])) for f in RESULT_DTYPE.names}

    def extras(self) -> np.ndarray:
        """Per-tenant SLO hits and completed queries, and re-issued attempts, one row per sim."""
        out = np.zeros(self.n_sims, EXTRA_DTYPE)
        _check(self.lib, self.lib.hx_sim_extras(self.h, _p(out), self.n_sims))
        return out

    def best(self, objective: int = OBJ_P95):
        per = np.zeros(self.n_traces, np.int32)
        b = hx_best(0, 0, 0, 0, _p(per))
        _check(self.lib, self.lib.hx_sim_best(self.h, int(objective), ctypes.byref(b)))
        return int(b.global_point), int(b.global_sum_p95), int(b.global_slo_met), per

    def point_sums(self):
        """(summed P95, summed SLO hits, failed simulations) per point over this handle's traces."""
        a = np.zeros(self.n_points, np.int64)
        b = np.zeros(self.n_points, np.int64)
        c = np.zeros(self.n_points, np.int32)
        _check(self.lib, self.lib.hx_sim_point_sums(self.h, _p(a), _p(b), _p(c), self.n_points))
        return a, b, c

    def records(self, rec_index: int) -> dict:
        t = self.record_sims[rec_index] // self.n_points
        n = self.n_calls[t]
        out = dict(inst=np.zeros(n, np.int32), enq=np.zeros(n, np.int64), budget=np.zeros(n, np.int64),
                   start=np.zeros(n, np.int64), end=np.zeros(n, np.int64))
        _check(self.lib, self.lib.hx_sim_records(self.h, int(rec_index), _p(out["inst"]), _p(out["enq"]),
                                                 _p(out["budget"]), _p(out["start"]), _p(out["end"]), n))
        return out

    def prep(self, trace_index: int) -> dict:
        n = self.n_calls[trace_index]
        out = dict(est=np.zeros((n, 4), np.int32), svc=np.zeros((n, 4), np.int32), tbar=np.zeros(n, np.int32),
                   deadline=np.zeros(n, np.int64))
        _check(self.lib, self.lib.hx_sim_prep(self.h, int(trace_index), _p(out["est"]), _p(out["svc"]),
                                              _p(out["tbar"]), _p(out["deadline"]), n))
        return out

    def timings(self, back: int = 0):
        """(prep, simulate, best) milliseconds of the last run, or of the run
        `back` runs before it (the handle keeps its last 64 runs)."""
        a, b, c = ctypes.c_float(), ctypes.c_float(), ctypes.c_float()
        _check(self.lib, self.lib.hx_sim_timings_back(self.h, int(back), ctypes.byref(a), ctypes.byref(b),
                                                      ctypes.byref(c)))
        return float(a.value), float(b.value), float(c.value)

    def info(self) -> dict:
        i = hx_info()
        _check(self.lib, self.lib.hx_sim_info(self.h, ctypes.byref(i)))
        return {f: getattr(i, f) for f, _ in hx_info._fields_}

    def close(self):
        if getattr(self, "h", None):
            self.lib.hx_sim_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()
