"""Online alpha tuning (Sec. 4.3) on top of the batched simulator.

The serving system starts with alpha* = 0 (cold start), watches the tail
latency of completed queries in sliding windows of at least `min_queries`
queries, and compares each window with the previous one by a one-sided
two-sample t-test (H1: the new window's latencies are larger).  When the
p-value falls below `p_threshold` it replays the most recent window through
the simulator for every alpha in {0, 0.1, ..., 1} and adopts the alpha with
the lowest simulated P95 (alpha* = argmin_alpha T_0.95(alpha)).

The live system is emulated: window w's "observed" latencies are those of a
simulation of window w's queries under the alpha in force at that time,
started from an idle cluster (queues are not carried across windows).  The
simulation backend is a function so the same loop can run on the CUDA
library (`gpu_backend`) or on any other implementation of the simulation.
"""
from __future__ import annotations

import time
from dataclasses import dataclass, field
from typing import Callable, List, Optional, Sequence, Tuple

import numpy as np

from . import workloads as W


@dataclass
class WindowReport:
    index: int
    t0_us: int
    t1_us: int
    n_queries: int
    alpha_fp: int             # alpha in force during the window
    p95_us: int               # observed nearest-rank P95 of the window
    p_value: Optional[float]  # one-sided t-test against the previous window
    triggered: bool
    new_alpha_fp: int         # alpha after the window (changed only when triggered)
    sweep_p95_us: List[int] = field(default_factory=list)
    tune_ms: float = 0.0      # wall time of the sweep (upload, simulate, best point)


def slice_queries(trace: W.Trace, i0: int, i1: int) -> W.Trace:
    """Queries [i0, i1) of a trace as a trace of their own, arrivals measured
    from the first of them."""
    b0, b1 = int(trace.call_base[i0]), int(trace.call_base[i1])
    arr = trace.arrival_us[i0:i1]
    t0 = int(arr[0]) if i1 > i0 else 0
    return W.Trace(arr - t0, trace.k[i0:i1].copy(), (trace.call_base[i0:i1 + 1] - b0).astype(np.int32),
                   trace.prompt[b0:b1].copy(), trace.out[b0:b1].copy(), trace.out_est[b0:b1].copy(),
                   trace.stage[b0:b1].copy(), trace.cand[b0:b1].copy(), trace.retry[b0:b1].copy())


def windows(trace: W.Trace, window_us: int, min_queries: int) -> List[Tuple[int, int]]:
    """Query ranges of consecutive windows of `window_us`; a window holding
    fewer than `min_queries` queries is extended by the next one."""
    arr = trace.arrival_us
    out = []
    i = 0
    n = trace.n_queries
    while i < n:
        end_t = int(arr[i]) // window_us * window_us + window_us
        j = int(np.searchsorted(arr, end_t, side="left"))
        while j - i < min_queries and j < n:
            end_t += window_us
            j = int(np.searchsorted(arr, end_t, side="left"))
        if j - i < min_queries and out:
            a, _ = out.pop()
            i = a
        out.append((i, j))
        i = j
    return out


def nearest_rank_p95(lat: np.ndarray) -> int:
    s = np.sort(np.asarray(lat))
    return int(s[(95 * len(s) + 99) // 100 - 1]) if len(s) else 0


def welch_greater(new: np.ndarray, ref: np.ndarray) -> float:
    """p-value of the one-sided Welch t-test H1: mean(new) > mean(ref)."""
    from scipy import stats
    if len(new) < 2 or len(ref) < 2:
        return 1.0
    r = stats.ttest_ind(np.asarray(new, np.float64), np.asarray(ref, np.float64), equal_var=False,
                        alternative="greater")
    p = float(r.pvalue)
    return 1.0 if np.isnan(p) else p


# A backend simulates one trace under several points and returns
# (per-point results with a "p95_us" field, per-query latencies of point 0).
Backend = Callable[[W.Trace, W.Cluster, W.Grid], Tuple[np.ndarray, np.ndarray]]


def gpu_backend(trace: W.Trace, cluster: W.Cluster, grid: W.Grid):
    """The CUDA library: one handle per call (upload, run, read back)."""
    from . import hxsim as H
    sim = H.Sim([trace], cluster, grid, record_sims=[0])
    try:
        sim.run()
        res = sim.results()
        rec = sim.records(0)
        # a query ends when its evaluation call (its last call) ends
        lat = rec["end"][trace.call_base[1:] - 1] - trace.arrival_us
        return res, lat
    finally:
        sim.close()


class OnlineTuner:
    def __init__(self, cluster: W.Cluster, backend: Backend = gpu_backend, alphas_fp: Optional[Sequence[int]] = None,
                 gamma_fp: int = W.SCALE, rho: Optional[int] = None, beta_us2: int = 300_000 ** 2,
                 window_us: int = 100_000_000, min_queries: int = 5, p_threshold: float = 0.01):
        self.cluster = cluster
        self.backend = backend
        self.alphas = list(alphas_fp) if alphas_fp is not None else [i * W.SCALE // 10 for i in range(11)]
        self.gamma_fp = gamma_fp
        self.rho = cluster.rmax if rho is None else rho
        self.beta = beta_us2
        self.window_us = window_us
        self.min_queries = min_queries
        self.p_threshold = p_threshold

    def grid_of(self, alphas: Sequence[int]) -> W.Grid:
        """Grid of the given alpha values with this tuner's gamma, rho and beta."""
        n = len(alphas)
        return W.Grid(np.asarray(alphas, np.int64), np.full(n, self.gamma_fp, np.int64),
                      np.full(n, self.rho, np.int32), np.full(n, self.beta, np.int64),
                      np.zeros(n, np.uint8), np.zeros(n, np.uint8))

    def run(self, trace: W.Trace) -> List[WindowReport]:
        alpha = 0  # cold start: queue-length minimisation
        reports: List[WindowReport] = []
        ref_lat = None
        for w, (i0, i1) in enumerate(windows(trace, self.window_us, self.min_queries)):
            win = slice_queries(trace, i0, i1)
            _, lat = self.backend(win, self.cluster, self.grid_of([alpha]))
            p = welch_greater(lat, ref_lat) if ref_lat is not None else None
            trig = p is not None and p < self.p_threshold
            rep = WindowReport(w, int(trace.arrival_us[i0]), int(trace.arrival_us[i1 - 1]), i1 - i0, alpha,
                               nearest_rank_p95(lat), p, trig, alpha)
            if trig:
                t0 = time.perf_counter()
                res, _ = self.backend(win, self.cluster, self.grid_of(self.alphas))
                p95 = res["p95_us"].astype(np.int64)
                ok = res["status"] == 0
                best = int(np.argmin(np.where(ok, p95, np.iinfo(np.int64).max)))  # ties: lowest alpha
                rep.tune_ms = 1000 * (time.perf_counter() - t0)
                rep.sweep_p95_us = [int(x) for x in p95]
                alpha = self.alphas[best]
                rep.new_alpha_fp = alpha
            reports.append(rep)
            ref_lat = lat
        return reports


def shift_trace(rates_qps: Sequence[float], seconds: Sequence[float], recipe: int = 0, seed: int = 0) -> W.Trace:
    """A trace whose Poisson rate steps through `rates_qps`, each for the
    matching number of seconds (the 5 -> 20 -> 5 QPS shift of Sec. 5.1)."""
    r = W.RECIPES[recipe]
    parts = []
    t_off = 0
    for j, (rate, sec) in enumerate(zip(rates_qps, seconds)):
        n = max(1, int(rate * sec))
        rj = W.Recipe(**{**r.__dict__, "rate_qps": [rate], "arrival": "poisson"})
        tr = W.make_trace(rj, 100 + recipe, seed * 16 + j, n_queries=n)
        tr.arrival_us = tr.arrival_us + t_off
        t_off = max(int(t_off + sec * 1e6), int(tr.arrival_us[-1]) + 1)
        parts.append(tr)
    # concatenate
    cb = [np.zeros(1, np.int32)]
    off = 0
    for tr in parts:
        cb.append(tr.call_base[1:] + off)
        off += tr.n_calls
    cat = lambda f: np.concatenate([getattr(tr, f) for tr in parts])
    return W.Trace(cat("arrival_us"), cat("k"), np.concatenate(cb).astype(np.int32), cat("prompt"), cat("out"),
                   cat("out_est"), cat("stage"), cat("cand"), cat("retry"))
