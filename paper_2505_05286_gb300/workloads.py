"""Seeded synthetic workloads for the batched HexGen-Flow scheduler simulation.

This module only *generates inputs*: request traces (the agentic Text-to-SQL
workflow of Sec. 2.1 - schema linking, k parallel SQL candidates, per-candidate
self-correction retries, evaluation), heterogeneous clusters (the per-type
performance profiles of Sec. 3.3) and hyper-parameter grids (the alpha sweep of
Sec. 4.3).  It holds none of the scheduler's arithmetic: no service-time or
cost estimate, no budget, score, urgency, deadline or percentile.  Both the
CUDA library and the CPU oracle consume its arrays; neither shares any other
code with the other.

Randomness is a counter-based splitmix64 stream (Steele, Lea & Flood, 2014):
value j of a stream with key K is mix64(K + (j + 1) * 0x9E3779B97F4A7C15).
Uniform doubles are (x >> 11) * 2^-53.  Every draw is addressed by
(stream, index), so traces are reproducible independently of generation
order.

The five workload recipes (`RECIPES`) stand in for the paper's BIRD / Spider
derived traces (Sec. 5.1), which are not available: Poisson or two-state MMPP
query arrivals, per-stage token-length distributions (uniform or clipped
lognormal), candidate counts k, error probability p and retry limit R.  The
`EXTRA` recipes add Sec. 5's other settings: ~20 calls per query, a noisy
output-length predictor, two tenants with different SLOs, competing
single-shot requests, and instances that slow down or stop for a while.
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass, field
from typing import List, Optional, Sequence

import numpy as np

# Stage codes of the workflow (Sec. 2.1).
STAGE_S = 0  # schema linking
STAGE_G = 1  # SQL candidate generation
STAGE_C = 2  # self-correction
STAGE_E = 3  # evaluation

POLICY_PQ = 0    # local queue: urgency priority queue (Sec. 4.2)
POLICY_FCFS = 1  # local queue: first come first served (ablation, Sec. 5.1)
POLICY_LLF = 2   # local queue: least laxity first, no per-request budget (baseline, Sec. 5.1)
DISPATCH_WB = 0  # global dispatch: workload balanced (Sec. 4.1)
DISPATCH_RR = 1  # global dispatch: round robin (ablation, Sec. 5.1)

OBJ_P95 = 0        # argmin P95 (Sec. 4.3)
OBJ_P95_SLO95 = 1  # argmin P95 among points with >= 95% SLO attainment

SCALE = 1_000_000  # fixed-point scale of alpha, gamma and the SLO multiplier

# A fault window: attempts that start on `inst` in [t0_us, t1_us) run
# slow_fp / SCALE times longer; slow_fp = 0 stops them (they time out).
FAULT_DTYPE = np.dtype([("inst", "<i4"), ("pad", "<i4"), ("t0_us", "<i8"), ("t1_us", "<i8"), ("slow_fp", "<i8")])

_M64 = (1 << 64) - 1
_GOLD = 0x9E3779B97F4A7C15


# ----------------------------------------------------------------------------
# Containers (plain arrays; the library and the oracle marshal them separately)
# ----------------------------------------------------------------------------
@dataclass
class Trace:
    """One request trace.

    Queries are sorted by arrival.  Calls of query i occupy
    [call_base[i], call_base[i+1]) in the order S, G_0..G_{k-1}, then the
    self-correction calls C_{c,r} by (candidate c, retry r) ascending, then E.
    `retry` is r (1-based) for C calls and 0 otherwise; `cand` is c for G and
    C calls and 0 otherwise.  `out_est` is the output length the scheduler
    believes (the predictor of Sec. 4.1 replaced by the stage mean); `out`
    is the true output length that decides the service time.
    """

    arrival_us: np.ndarray  # int64 [nq]
    k: np.ndarray           # uint8 [nq]
    call_base: np.ndarray   # int32 [nq + 1]
    prompt: np.ndarray      # int32 [nc]
    out: np.ndarray         # int32 [nc]
    out_est: np.ndarray     # int32 [nc]
    stage: np.ndarray       # uint8 [nc]
    cand: np.ndarray        # uint8 [nc]
    retry: np.ndarray       # uint8 [nc]
    tenant: Optional[np.ndarray] = None  # uint8 [nq] tenant of each query (None: all tenant 0)

    @property
    def n_queries(self) -> int:
        return int(self.arrival_us.shape[0])

    @property
    def n_calls(self) -> int:
        return int(self.prompt.shape[0])


@dataclass
class Cluster:
    """Heterogeneous instances: per-type profile + instance -> type map."""

    prefill_tok_s: np.ndarray   # int32 [T]   prefill throughput, tokens / s
    decode_us_tok: np.ndarray   # int32 [T]   decode cost, microseconds / token
    slots: np.ndarray           # int32 [T]   concurrent batch slots per instance
    inst_type: np.ndarray       # uint8 [N]
    ref_type: int               # type whose exclusive latency defines the SLO
    slo_mult_fp: int            # SLO multiplier, fixed point (SCALE)
    rmax: int                   # configured retry bound R of the workflow
    stage_ref_prompt: np.ndarray  # int32 [4] reference prompt length per stage
    stage_ref_out: np.ndarray     # int32 [4] reference output length per stage
    tenant_slo_mult_fp: Optional[np.ndarray] = None  # int64 [n_tenants] per-tenant SLO multipliers
    timeout_mult_fp: int = 0      # attempt timeout as a multiple of its estimate (0: none)
    faults: Optional[np.ndarray] = None  # FAULT_DTYPE [n_faults] instance slow-down / outage windows

    @property
    def n_tenants(self) -> int:
        return 1 if self.tenant_slo_mult_fp is None else int(len(self.tenant_slo_mult_fp))

    @property
    def n_types(self) -> int:
        return int(self.prefill_tok_s.shape[0])

    @property
    def n_inst(self) -> int:
        return int(self.inst_type.shape[0])


@dataclass
class Grid:
    """Hyper-parameter points, row-major with alpha outermost."""

    alpha_fp: np.ndarray         # int64 [P]  alpha * SCALE, in [0, SCALE]
    gamma_fp: np.ndarray         # int64 [P]  urgency ageing weight * SCALE
    rho: np.ndarray              # int32 [P]  assumed remaining corrections bound
    beta_us2: np.ndarray         # int64 [P]  beta = C_ref * Q_ref, microseconds^2
    local_policy: np.ndarray     # uint8 [P]  POLICY_PQ / POLICY_FCFS / POLICY_LLF
    dispatch_policy: np.ndarray  # uint8 [P]  DISPATCH_WB / DISPATCH_RR

    @property
    def n_points(self) -> int:
        return int(self.alpha_fp.shape[0])


@dataclass
class Workload:
    name: str
    traces: List[Trace]
    cluster: Cluster
    grid: Grid
    objective: int

    @property
    def n_sims(self) -> int:
        return len(self.traces) * self.grid.n_points

    @property
    def n_calls(self) -> int:
        return sum(t.n_calls for t in self.traces)


# ----------------------------------------------------------------------------
# Counter-based splitmix64
# ----------------------------------------------------------------------------
def _mix64_int(z: int) -> int:
    z &= _M64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _M64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _M64
    return z ^ (z >> 31)


def _mix64_arr(z: np.ndarray) -> np.ndarray:
    z = z ^ (z >> np.uint64(30))
    z = z * np.uint64(0xBF58476D1CE4E5B9)
    z = z ^ (z >> np.uint64(27))
    z = z * np.uint64(0x94D049BB133111EB)
    return z ^ (z >> np.uint64(31))


def stream_key(*parts: int) -> int:
    """Key of a random stream addressed by integer parts (config, seed, name)."""
    k = 0x243F6A8885A308D3
    for p in parts:
        k = _mix64_int(k ^ _mix64_int((int(p) + _GOLD) & _M64))
    return k


def stream_u64(key: int, n: int, start: int = 0) -> np.ndarray:
    idx = np.arange(start + 1, start + n + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return _mix64_arr(np.uint64(key) + idx * np.uint64(_GOLD))


def stream_uniform(key: int, n: int, start: int = 0) -> np.ndarray:
    """Doubles in [0, 1)."""
    return (stream_u64(key, n, start) >> np.uint64(11)).astype(np.float64) * (2.0 ** -53)


_STREAM_ARRIVAL, _STREAM_DWELL, _STREAM_K, _STREAM_ERR, _STREAM_PROMPT, _STREAM_OUT, _STREAM_EST = range(1, 8)
_STREAM_TENANT, _STREAM_SINGLE = 8, 9


# ----------------------------------------------------------------------------
# Recipes
# ----------------------------------------------------------------------------
@dataclass
class TokenDist:
    kind: str          # "uniform" (inclusive [a, b]) or "lognormal" (mu, sigma, clip [a, b])
    a: float
    b: float
    mu: float = 0.0
    sigma: float = 0.0


@dataclass
class Recipe:
    name: str
    n_traces: int
    n_queries: int
    arrival: str                 # "poisson" or "mmpp"
    rate_qps: Sequence[float]    # one rate (poisson) or the two MMPP state rates
    mmpp_dwell_s: float
    k_range: Sequence[int]       # inclusive [kmin, kmax]
    p_err: float
    rmax: int
    prompt: Sequence[TokenDist]  # per stage S, G, C, E
    out: Sequence[TokenDist]
    out_est: Sequence[int]       # scheduler's output-length belief per stage
    ref_prompt: Sequence[int]    # reference tokens per stage (stage means)
    types: Sequence[Sequence[int]]   # (prefill tok/s, decode us/tok, slots)
    inst_counts: Sequence[int]
    ref_type: int
    slo_mult_fp: int
    alpha_n: int
    gamma_fp: Sequence[int]
    rho: Optional[Sequence[int]]
    beta_mult: Sequence[Sequence[int]]  # (num, den) multipliers of c_ref^2
    c_ref_us: int                # reference computation / queueing time (beta = c_ref^2)
    objective: int
    trace_seeds: Optional[Sequence[int]] = None
    est_noise_sigma: float = 0.0  # lognormal noise of the believed output length (0: the stage mean)
    tenant_slo_mult_fp: Optional[Sequence[int]] = None  # per-tenant SLO multipliers (None: one tenant)
    tenant_share: Optional[Sequence[float]] = None      # tenant probabilities of the workflow queries
    single_frac: float = 0.0      # single-shot requests added, as a fraction of the workflow's calls
    single_tenant: int = 0        # tenant of the single-shot requests
    timeout_mult: float = 0.0     # attempt timeout as a multiple of its estimate (0: none)
    faults: Optional[Sequence[Sequence[float]]] = None  # (instance, t0 s, t1 s, slow-down; 0 = stopped)


def _u(a, b):
    return TokenDist("uniform", a, b)


def _ln(mu, sigma, a, b):
    return TokenDist("lognormal", a, b, mu, sigma)


_UNIF_PROMPT = [_u(2000, 6000), _u(1500, 4000), _u(1000, 3000), _u(2000, 5000)]
_UNIF_OUT = [_u(50, 200), _u(100, 400), _u(100, 300), _u(50, 150)]
# Stage means floor((a + b) / 2) of the uniform recipes above.
_UNIF_OUT_EST = [125, 250, 200, 100]
_UNIF_REF_PROMPT = [4000, 2750, 2000, 3500]
_LN_PROMPT = [_ln(8.0, 0.6, 256, 32000)] * 4
_LN_OUT = [_ln(5.0, 0.7, 16, 2048)] * 4
# Lognormal means floor(exp(mu + sigma^2 / 2)): exp(8.18) = 3568.7, exp(5.245) = 189.6.
_LN_OUT_EST = [189] * 4
_LN_REF_PROMPT = [3568] * 4

TYPE_A = (12000, 15, 8)
TYPE_B = (5000, 35, 4)
TYPE_C = (20000, 10, 16)
TYPES_4 = [(5000, 35, 4), (9000, 22, 8), (12000, 15, 8), (20000, 10, 16)]

_GAMMA4 = [SCALE // 2, SCALE, 3 * SCALE // 2, 2 * SCALE]
_GAMMA8 = [(i + 1) * SCALE // 4 for i in range(8)]

RECIPES: List[Recipe] = [
    Recipe("tiny-1x200q-4inst-16pt", 1, 200, "poisson", [2.0], 0.0, [4, 4], 0.3, 2,
           _UNIF_PROMPT, _UNIF_OUT, _UNIF_OUT_EST, _UNIF_REF_PROMPT,
           [TYPE_A, TYPE_B], [2, 2], 0, 3 * SCALE,
           4, _GAMMA4, None, [(1, 1)], 400_000, OBJ_P95),
    Recipe("small-8x2000q-8inst-64pt", 8, 2000, "poisson", [4.0], 0.0, [4, 4], 0.3, 2,
           _UNIF_PROMPT, _UNIF_OUT, _UNIF_OUT_EST, _UNIF_REF_PROMPT,
           [TYPE_A, TYPE_B, TYPE_C], [4, 2, 2], 0, 3 * SCALE,
           8, _GAMMA8, None, [(1, 1)], 300_000, OBJ_P95),
    Recipe("bursty-32x5000q-16inst-256pt", 32, 5000, "mmpp", [1.0, 12.0], 60.0, [2, 8], 0.5, 3,
           _UNIF_PROMPT, _UNIF_OUT, _UNIF_OUT_EST, _UNIF_REF_PROMPT,
           [TYPE_A, TYPE_B, TYPE_C], [8, 4, 4], 0, 3 * SCALE,
           8, _GAMMA8, [0, 1, 2, 3], [(1, 1)], 300_000, OBJ_P95),
    Recipe("hetero-64x10000q-32inst-512pt", 64, 10000, "poisson", [10.0], 0.0, [4, 4], 0.3, 2,
           _LN_PROMPT, _LN_OUT, _LN_OUT_EST, _LN_REF_PROMPT,
           TYPES_4, [8, 8, 8, 8], 2, 5 * SCALE // 2,
           8, _GAMMA8, None, [(1, 16), (1, 8), (1, 4), (1, 2), (1, 1), (2, 1), (4, 1), (8, 1)],
           400_000, OBJ_P95),
    Recipe("ceiling-256x20000q-64inst-1024pt", 256, 20000, "poisson", [16.0], 0.0, [4, 4], 0.3, 2,
           _LN_PROMPT, _LN_OUT, _LN_OUT_EST, _LN_REF_PROMPT,
           TYPES_4, [26, 19, 13, 6], 2, 5 * SCALE // 2,
           8, _GAMMA8, [0, 1, 2, 3], [(1, 4), (1, 2), (1, 1), (2, 1)], 500_000, OBJ_P95_SLO95),
]

# Extra recipes beyond the five benchmark ones (Sec. 5.1's workload shapes):
#  - "paper-shaped": ~20 calls per query (k = 8 candidates, error probability
#    0.55, up to 10 refinement rounds) at 1 query/s on a 2A + 2B cluster;
#  - "noisy-estimate": recipe 1 with the output-length predictor replaced by
#    the true length times lognormal(0, 0.5) noise;
#  - "two-tenant": recipe 1 with two tenants, SLO 2x and 4x, half the
#    queries each (the multi-tenant evaluation);
#  - "competing-25" / "competing-50": recipe 1 plus single-shot requests
#    numbering 25% / 50% of the workflow's calls, with generation-stage token
#    lengths and their own tenant and SLO (5x);
#  - "faulty": recipe 1 with a 3x-estimate timeout, instance 0 (type A)
#    stopped for 60 s, instance 4 (type B) 3x slower for 120 s and instance
#    6 (type C) stopped for 30 s (timeout and re-issue, Sec. 3.3).
_SMALL = dict(n_traces=8, n_queries=2000, arrival="poisson", rate_qps=[4.0], mmpp_dwell_s=0.0, k_range=[4, 4],
              p_err=0.3, rmax=2, prompt=_UNIF_PROMPT, out=_UNIF_OUT, out_est=_UNIF_OUT_EST,
              ref_prompt=_UNIF_REF_PROMPT, types=[TYPE_A, TYPE_B, TYPE_C], inst_counts=[4, 2, 2], ref_type=0,
              slo_mult_fp=3 * SCALE, alpha_n=8, gamma_fp=_GAMMA8, rho=None, beta_mult=[(1, 1)], c_ref_us=300_000,
              objective=OBJ_P95)
EXTRA: dict = {
    "paper-shaped": Recipe("paper-shaped-8x400q-4inst-16pt", 8, 400, "poisson", [1.0], 0.0, [8, 8], 0.55, 10,
                           _UNIF_PROMPT, _UNIF_OUT, _UNIF_OUT_EST, _UNIF_REF_PROMPT,
                           [TYPE_A, TYPE_B], [2, 2], 0, 3 * SCALE,
                           4, _GAMMA4, None, [(1, 1)], 400_000, OBJ_P95),
    "noisy-estimate": Recipe("noisy-estimate-8x2000q-8inst-64pt", 8, 2000, "poisson", [4.0], 0.0, [4, 4], 0.3, 2,
                             _UNIF_PROMPT, _UNIF_OUT, _UNIF_OUT_EST, _UNIF_REF_PROMPT,
                             [TYPE_A, TYPE_B, TYPE_C], [4, 2, 2], 0, 3 * SCALE,
                             8, _GAMMA8, None, [(1, 1)], 300_000, OBJ_P95, est_noise_sigma=0.5),
    "two-tenant": Recipe("two-tenant-8x2000q-8inst-64pt", **_SMALL, tenant_slo_mult_fp=[2 * SCALE, 4 * SCALE],
                         tenant_share=[0.5, 0.5]),
    "competing-25": Recipe("competing25-8x2000q-8inst-64pt", **_SMALL, tenant_slo_mult_fp=[3 * SCALE, 5 * SCALE],
                           single_frac=0.25, single_tenant=1),
    "competing-50": Recipe("competing50-8x2000q-8inst-64pt", **_SMALL, tenant_slo_mult_fp=[3 * SCALE, 5 * SCALE],
                           single_frac=0.5, single_tenant=1),
    "faulty": Recipe("faulty-8x2000q-8inst-64pt", **_SMALL, timeout_mult=3.0,
                     faults=[(0, 100.0, 160.0, 0.0), (4, 200.0, 320.0, 3.0), (6, 300.0, 330.0, 0.0)]),
}
# Random-stream ids of the extra recipes (fixed, so adding one changes no other trace).
EXTRA_ID = {"noisy-estimate": 16, "paper-shaped": 17, "two-tenant": 18, "competing-25": 19, "competing-50": 20,
            "faulty": 21}


# ----------------------------------------------------------------------------
# Generators
# ----------------------------------------------------------------------------
def _group_arange(counts: np.ndarray) -> np.ndarray:
    """concat(arange(c) for c in counts) without a Python loop."""
    counts = np.asarray(counts, dtype=np.int64)
    total = int(counts.sum())
    starts = np.cumsum(counts) - counts
    return np.arange(total, dtype=np.int64) - np.repeat(starts, counts)


def _poisson_arrivals(key: int, n: int, rate: float) -> np.ndarray:
    u = stream_uniform(stream_key(key, _STREAM_ARRIVAL), n)
    gaps = np.floor(-np.log(1.0 - u) / rate * 1e6).astype(np.int64)
    return np.cumsum(gaps, dtype=np.int64)


def _mmpp_arrivals(key: int, n: int, rates: Sequence[float], dwell_s: float) -> np.ndarray:
    """Two-state Markov-modulated Poisson arrivals starting in state 0."""
    ka, kd = stream_key(key, _STREAM_ARRIVAL), stream_key(key, _STREAM_DWELL)
    ua = stream_uniform(ka, 8 * n + 64)
    ud = stream_uniform(kd, 8 * n + 64)
    ia = idd = 0
    t = 0
    state = 0
    switch_at = int(np.floor(-np.log(1.0 - ud[idd]) * dwell_s * 1e6))
    idd += 1
    out = np.empty(n, dtype=np.int64)
    i = 0
    while i < n:
        gap = int(np.floor(-np.log(1.0 - ua[ia]) / rates[state] * 1e6))
        ia += 1
        if t + gap > switch_at:
            # memoryless: move to the switch, change state, redraw the gap
            t = switch_at
            state ^= 1
            switch_at = t + int(np.floor(-np.log(1.0 - ud[idd]) * dwell_s * 1e6))
            idd += 1
            continue
        t += gap
        out[i] = t
        i += 1
    return out


def _draw_tokens(key: int, stage: np.ndarray, dists: Sequence[TokenDist]) -> np.ndarray:
    n = stage.shape[0]
    u = stream_uniform(key, 2 * n).reshape(n, 2)
    res = np.zeros(n, dtype=np.int64)
    for s, d in enumerate(dists):
        sel = stage == s
        if not sel.any():
            continue
        us = u[sel]
        if d.kind == "uniform":
            a, b = int(d.a), int(d.b)
            v = a + np.floor(us[:, 0] * (b - a + 1)).astype(np.int64)
        else:
            z = np.sqrt(-2.0 * np.log(1.0 - us[:, 0])) * np.cos(2.0 * np.pi * us[:, 1])
            v = np.floor(np.exp(d.mu + d.sigma * z) + 0.5).astype(np.int64)
            v = np.clip(v, int(d.a), int(d.b))
        res[sel] = v
    return res.astype(np.int32)


def make_trace(recipe: Recipe, cfg_id: int, seed: int, n_queries: Optional[int] = None) -> Trace:
    nq = recipe.n_queries if n_queries is None else int(n_queries)
    key = stream_key(cfg_id, seed)
    if nq == 0:
        z32 = np.zeros(0, np.int32)
        z8 = np.zeros(0, np.uint8)
        return Trace(np.zeros(0, np.int64), z8, np.zeros(1, np.int32), z32, z32.copy(), z32.copy(),
                     z8.copy(), z8.copy(), z8.copy())
    if recipe.arrival == "poisson":
        arrival = _poisson_arrivals(key, nq, recipe.rate_qps[0])
    else:
        arrival = _mmpp_arrivals(key, nq, recipe.rate_qps, recipe.mmpp_dwell_s)

    kmin, kmax = recipe.k_range
    if kmin == kmax:
        k = np.full(nq, kmin, dtype=np.int64)
    else:
        uk = stream_uniform(stream_key(key, _STREAM_K), nq)
        k = kmin + np.floor(uk * (kmax - kmin + 1)).astype(np.int64)

    R = recipe.rmax
    KMAX = 8
    if R > 0:
        ue = stream_uniform(stream_key(key, _STREAM_ERR), nq * KMAX * R).reshape(nq, KMAX, R)
        err = ue < recipe.p_err
        # a chain keeps erring (and retrying) while consecutive draws err, up to R retries
        r = np.cumprod(err, axis=2).sum(axis=2).astype(np.int64)
    else:
        r = np.zeros((nq, KMAX), dtype=np.int64)
    r[np.arange(KMAX)[None, :] >= k[:, None]] = 0
    ncorr = r.sum(axis=1)
    ncalls = 2 + k + ncorr
    call_base = np.zeros(nq + 1, dtype=np.int64)
    call_base[1:] = np.cumsum(ncalls)
    nc = int(call_base[-1])

    stage = np.full(nc, STAGE_C, dtype=np.uint8)
    cand = np.zeros(nc, dtype=np.uint8)
    retry = np.zeros(nc, dtype=np.uint8)
    stage[call_base[:-1]] = STAGE_S
    stage[call_base[1:] - 1] = STAGE_E
    # G_0..G_{k-1}
    qg = np.repeat(np.arange(nq), k)
    cg = _group_arange(k)
    pg = call_base[:-1][qg] + 1 + cg
    stage[pg] = STAGE_G
    cand[pg] = cg
    # C_{c,1..r_c} by (c, r)
    valid = np.arange(KMAX)[None, :] < k[:, None]
    qc = np.repeat(np.arange(nq), k)          # one entry per (query, candidate)
    rc = r[valid]                              # r_c in (query, candidate) order
    cc = cg
    pref = np.cumsum(rc) - rc                  # global exclusive prefix over (q, c)
    qfirst = np.cumsum(k) - k                  # index of each query's first candidate
    pref_in_q = pref - pref[qfirst][qc]
    qcc = np.repeat(qc, rc)
    ccc = np.repeat(cc, rc)
    rr = _group_arange(rc) + 1
    pc = call_base[:-1][qcc] + 1 + k[qcc] + np.repeat(pref_in_q, rc) + (rr - 1)
    stage[pc] = STAGE_C
    cand[pc] = ccc
    retry[pc] = rr

    prompt = _draw_tokens(stream_key(key, _STREAM_PROMPT), stage, recipe.prompt)
    out = _draw_tokens(stream_key(key, _STREAM_OUT), stage, recipe.out)
    out_est = np.asarray(recipe.out_est, dtype=np.int32)[stage]
    if recipe.est_noise_sigma > 0:
        # an output-length predictor with multiplicative lognormal error around the truth
        ue = stream_uniform(stream_key(key, _STREAM_EST), 2 * nc).reshape(nc, 2)
        z = np.sqrt(-2.0 * np.log(1.0 - ue[:, 0])) * np.cos(2.0 * np.pi * ue[:, 1])
        est = np.floor(out.astype(np.float64) * np.exp(recipe.est_noise_sigma * z) + 0.5)
        out_est = np.clip(est, 0, 1 << 20).astype(np.int32)
    tr = Trace(arrival.astype(np.int64), k.astype(np.uint8), call_base.astype(np.int32),
               prompt, out, out_est.astype(np.int32), stage, cand, retry)
    if recipe.tenant_share is not None:
        ut = stream_uniform(stream_key(key, _STREAM_TENANT), nq)
        cum = np.cumsum(np.asarray(recipe.tenant_share, np.float64))
        tr.tenant = np.minimum(np.searchsorted(cum / cum[-1], ut, side="right"), len(cum) - 1).astype(np.uint8)
    if recipe.single_frac > 0:
        tr = _add_single_shots(tr, recipe, key)
    return tr


def _add_single_shots(tr: Trace, recipe: Recipe, key: int) -> Trace:
    """Merge independent single-shot requests (a query of one evaluation-stage
    call, k = 0) into a trace: single_frac x its calls of them, Poisson over
    the trace's span, generation-stage token lengths, tenant single_tenant."""
    ns = int(np.floor(recipe.single_frac * tr.n_calls + 0.5))
    if ns == 0 or tr.n_queries == 0:
        return tr
    ks = stream_key(key, _STREAM_SINGLE)
    span_s = max(int(tr.arrival_us[-1]), 1) / 1e6
    arr = _poisson_arrivals(ks, ns, ns / span_s)
    gen = np.full(ns, STAGE_G, np.uint8)
    s_prompt = _draw_tokens(stream_key(ks, _STREAM_PROMPT), gen, recipe.prompt)
    s_out = _draw_tokens(stream_key(ks, _STREAM_OUT), gen, recipe.out)
    s_est = np.full(ns, recipe.out_est[STAGE_G], np.int32)
    if recipe.est_noise_sigma > 0:
        ue = stream_uniform(stream_key(ks, _STREAM_EST), 2 * ns).reshape(ns, 2)
        z = np.sqrt(-2.0 * np.log(1.0 - ue[:, 0])) * np.cos(2.0 * np.pi * ue[:, 1])
        s_est = np.clip(np.floor(s_out * np.exp(recipe.est_noise_sigma * z) + 0.5), 0, 1 << 20).astype(np.int32)
    nq0, nc0 = tr.n_queries, tr.n_calls
    # by arrival, workflow queries first at equal times
    arr_all = np.concatenate([tr.arrival_us, arr])
    single = np.concatenate([np.zeros(nq0, np.int64), np.ones(ns, np.int64)])
    order = np.lexsort((np.arange(nq0 + ns), single, arr_all))
    cnt = np.concatenate([np.diff(tr.call_base).astype(np.int64), np.ones(ns, np.int64)])[order]
    call_base = np.zeros(nq0 + ns + 1, np.int64)
    call_base[1:] = np.cumsum(cnt)
    src = np.concatenate([tr.call_base[:-1].astype(np.int64), nc0 + np.arange(ns, dtype=np.int64)])[order]
    idx = np.repeat(src - call_base[:-1], cnt) + np.arange(int(call_base[-1]), dtype=np.int64)
    cat = lambda base, extra: np.concatenate([base, extra])[idx]
    z8 = np.zeros(ns, np.uint8)
    ten0 = tr.tenant if tr.tenant is not None else np.zeros(nq0, np.uint8)
    return Trace(arr_all[order].astype(np.int64), np.concatenate([tr.k, z8])[order].astype(np.uint8),
                 call_base.astype(np.int32), cat(tr.prompt, s_prompt).astype(np.int32),
                 cat(tr.out, s_out).astype(np.int32), cat(tr.out_est, s_est).astype(np.int32),
                 cat(tr.stage, np.full(ns, STAGE_E, np.uint8)), cat(tr.cand, z8), cat(tr.retry, z8),
                 np.concatenate([ten0, np.full(ns, recipe.single_tenant, np.uint8)])[order].astype(np.uint8))


def make_cluster(recipe: Recipe) -> Cluster:
    t = np.asarray(recipe.types, dtype=np.int64)
    inst = np.repeat(np.arange(len(recipe.types)), recipe.inst_counts).astype(np.uint8)
    faults = None
    if recipe.faults:
        faults = np.zeros(len(recipe.faults), FAULT_DTYPE)
        for j, (m, t0, t1, slow) in enumerate(recipe.faults):
            faults[j] = (int(m), 0, int(round(t0 * 1e6)), int(round(t1 * 1e6)), int(round(slow * SCALE)))
    tmult = None if recipe.tenant_slo_mult_fp is None else np.asarray(recipe.tenant_slo_mult_fp, np.int64)
    return Cluster(t[:, 0].astype(np.int32), t[:, 1].astype(np.int32), t[:, 2].astype(np.int32), inst,
                   int(recipe.ref_type), int(recipe.slo_mult_fp), int(recipe.rmax),
                   np.asarray(recipe.ref_prompt, dtype=np.int32),
                   np.asarray(recipe.out_est, dtype=np.int32), tmult,
                   int(round(recipe.timeout_mult * SCALE)), faults)


def make_grid(recipe: Recipe, local_policy: int = POLICY_PQ, dispatch_policy: int = DISPATCH_WB) -> Grid:
    na = recipe.alpha_n
    alphas = [(i * SCALE) // (na - 1) for i in range(na)] if na > 1 else [0]
    gammas = list(recipe.gamma_fp)
    rhos = list(recipe.rho) if recipe.rho is not None else [recipe.rmax]
    c2 = recipe.c_ref_us * recipe.c_ref_us
    betas = [c2 * num // den for (num, den) in recipe.beta_mult]
    A, G, Rh, B = np.meshgrid(np.array(alphas, np.int64), np.array(gammas, np.int64),
                              np.array(rhos, np.int64), np.array(betas, np.int64), indexing="ij")
    P = A.size
    return Grid(A.ravel().astype(np.int64), G.ravel().astype(np.int64), Rh.ravel().astype(np.int32),
                B.ravel().astype(np.int64), np.full(P, local_policy, np.uint8),
                np.full(P, dispatch_policy, np.uint8))


def make_workload(cfg_id, n_traces: Optional[int] = None, n_queries: Optional[int] = None,
                  first_trace: int = 0) -> Workload:
    """Workload of recipe `cfg_id` (an index of RECIPES or a key of EXTRA),
    optionally with fewer traces or queries."""
    r = RECIPES[cfg_id] if isinstance(cfg_id, int) else EXTRA[cfg_id]
    if not isinstance(cfg_id, int):
        cfg_id = EXTRA_ID[cfg_id]
    nt = r.n_traces if n_traces is None else int(n_traces)
    traces = [make_trace(r, cfg_id, first_trace + j, n_queries) for j in range(nt)]
    name = r.name if (n_traces is None and n_queries is None) else (
        f"{r.name}[traces={nt},queries={traces[0].n_queries if traces else 0}]")
    return Workload(name, traces, make_cluster(r), make_grid(r), r.objective)


def subset_grid(grid: Grid, points: Sequence[int]) -> Grid:
    idx = np.asarray(points, dtype=np.int64)
    return Grid(*[getattr(grid, f.name)[idx] for f in dataclasses.fields(Grid)])


def concat_traces(traces: Sequence[Trace]) -> dict:
    """Flatten traces into one set of arrays plus per-trace query/call offsets."""
    nq = np.array([t.n_queries for t in traces], dtype=np.int64)
    nc = np.array([t.n_calls for t in traces], dtype=np.int64)
    q_off = np.zeros(len(traces) + 1, np.int64)
    q_off[1:] = np.cumsum(nq)
    c_off = np.zeros(len(traces) + 1, np.int64)
    c_off[1:] = np.cumsum(nc)
    return dict(q_off=q_off, c_off=c_off)
