"""The seeded input generator: structure, statistics and determinism."""
import hashlib
import json
import os

import numpy as np
import pytest

from paper_2505_05286_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def trace_digest(tr):
    h = hashlib.sha256()
    for f in ("arrival_us", "k", "call_base", "prompt", "out", "out_est", "stage", "cand", "retry"):
        h.update(np.ascontiguousarray(getattr(tr, f)).tobytes())
    return h.hexdigest()


@pytest.mark.parametrize("cfg", range(5))
def test_structure(cfg):
    r = W.RECIPES[cfg]
    tr = W.make_trace(r, cfg, 0, n_queries=min(r.n_queries, 3000))
    cb = tr.call_base
    assert cb[0] == 0 and cb[-1] == tr.n_calls and (np.diff(cb) >= 3).all()
    assert (np.diff(tr.arrival_us) >= 0).all()
    assert (tr.stage[cb[:-1]] == W.STAGE_S).all() and (tr.stage[cb[1:] - 1] == W.STAGE_E).all()
    for i in range(0, tr.n_queries, 97):
        st, ca, re = (a[cb[i]:cb[i + 1]] for a in (tr.stage, tr.cand, tr.retry))
        k = int(tr.k[i])
        assert (st[1:1 + k] == W.STAGE_G).all() and (ca[1:1 + k] == np.arange(k)).all()
        corr = list(zip(ca[1 + k:-1], re[1 + k:-1]))
        assert corr == sorted(corr) and all(st[1 + k:-1] == W.STAGE_C)
        for c in range(k):
            rs = [r_ for (c_, r_) in corr if c_ == c]
            assert rs == list(range(1, len(rs) + 1)) and len(rs) <= r.rmax
    assert (tr.prompt >= 1).all() and (tr.out >= 0).all()


@pytest.mark.parametrize("cfg", [0, 2, 3])
def test_calls_per_query_mean(cfg):
    """E[calls/query] = 1 + E[k] (1 + sum_{r=1..R} p^r) + 1."""
    r = W.RECIPES[cfg]
    tr = W.make_trace(r, cfg, 1, n_queries=20000)
    ek = (r.k_range[0] + r.k_range[1]) / 2
    expect = 2 + ek * (1 + sum(r.p_err ** j for j in range(1, r.rmax + 1)))
    got = tr.n_calls / tr.n_queries
    assert abs(got - expect) < 0.05 * expect


def test_poisson_rate():
    r = W.RECIPES[3]
    tr = W.make_trace(r, 3, 5, n_queries=20000)
    rate = tr.n_queries / (tr.arrival_us[-1] / 1e6)
    assert abs(rate - r.rate_qps[0]) < 0.03 * r.rate_qps[0]


def test_token_ranges():
    for cfg in (0, 3):
        r = W.RECIPES[cfg]
        tr = W.make_trace(r, cfg, 0, n_queries=2000)
        for s in range(4):
            sel = tr.stage == s
            assert tr.prompt[sel].min() >= r.prompt[s].a and tr.prompt[sel].max() <= r.prompt[s].b
            assert tr.out[sel].min() >= r.out[s].a and tr.out[sel].max() <= r.out[s].b
            assert (tr.out_est[sel] == r.out_est[s]).all()


def test_deterministic_and_seeded():
    r = W.RECIPES[1]
    a = W.make_trace(r, 1, 3, n_queries=500)
    b = W.make_trace(r, 1, 3, n_queries=500)
    c = W.make_trace(r, 1, 4, n_queries=500)
    assert trace_digest(a) == trace_digest(b) != trace_digest(c)


def test_golden_trace_digest():
    """The recipe-0 trace is byte-identical to the stored one."""
    with open(os.path.join(GOLDEN, "cfg0_oracle.json")) as f:
        g = json.load(f)
    wl = W.make_workload(0)
    assert trace_digest(wl.traces[0]) == g["trace_sha256"]


def test_grid_layout():
    g = W.make_grid(W.RECIPES[4])
    assert g.n_points == 1024
    # row-major with alpha outermost, beta multiplier innermost
    assert g.alpha_fp[0] == 0 and g.alpha_fp[-1] == W.SCALE and g.alpha_fp[128] == W.SCALE // 7
    assert g.rho[:16].tolist() == [0, 0, 0, 0, 1, 1, 1, 1, 2, 2, 2, 2, 3, 3, 3, 3]
    assert g.beta_us2[:4].tolist() == [500_000 ** 2 // 4, 500_000 ** 2 // 2, 500_000 ** 2, 2 * 500_000 ** 2]
    g0 = W.make_grid(W.RECIPES[0])
    assert g0.alpha_fp.tolist()[::4] == [0, 333333, 666666, 1000000]
    assert g0.gamma_fp.tolist()[:4] == [500000, 1000000, 1500000, 2000000]
