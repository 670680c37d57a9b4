"""The online tuning loop of Sec. 4.3 (cold start, sliding windows, one-sided
t-test, sweep over alpha) with the oracle as the simulation backend."""
import numpy as np
import pytest

from paper_2505_05286_gb300 import tuner as T
from paper_2505_05286_gb300 import workloads as W
from tests import tuner_cases as C


def test_windows_cover_and_hold_min_queries():
    tr, _, _ = C.shift_scenario()
    ws = T.windows(tr, 20_000_000, 5)
    assert ws[0][0] == 0 and ws[-1][1] == tr.n_queries
    assert all(a[1] == b[0] for a, b in zip(ws, ws[1:]))
    assert all(j - i >= 5 for i, j in ws)
    # a sparse trace: windows grow until they hold five queries
    sparse = T.slice_queries(tr, 0, 12)
    sparse.arrival_us = np.arange(12, dtype=np.int64) * 9_000_000
    ws2 = T.windows(sparse, 10_000_000, 5)
    assert all(j - i >= 5 for i, j in ws2) and ws2[-1][1] == 12


def test_slice_is_a_valid_trace():
    tr, cl, _ = C.shift_scenario()
    win = T.slice_queries(tr, 100, 140)
    assert win.arrival_us[0] == 0 and win.call_base[0] == 0 and win.call_base[-1] == win.n_calls
    res, lat = C.oracle_backend(win, cl, T.OnlineTuner(cl).grid_of([0]))
    assert res["status"][0] == 0 and len(lat) == 40 and (lat > 0).all()


def test_welch_one_sided():
    rng = np.random.default_rng(0)
    a = rng.normal(10, 1, 50)
    assert T.welch_greater(a + 3, a) < 1e-6
    assert T.welch_greater(a, a + 3) > 0.99
    assert T.welch_greater(a[:1], a) == 1.0


def test_loop_cold_start_trigger_and_argmin():
    tr, cl, kw = C.shift_scenario()
    reps = T.OnlineTuner(cl, backend=C.oracle_backend, **kw).run(tr)
    assert reps[0].alpha_fp == 0 and reps[0].p_value is None and not reps[0].triggered
    assert any(r.triggered for r in reps), "the 5 -> 20 q/s jump must trigger tuning"
    for prev, r in zip(reps, reps[1:]):
        assert r.alpha_fp == prev.new_alpha_fp
        assert r.triggered == (r.p_value < 0.01)
    for r in reps:
        if r.triggered:
            p95 = np.array(r.sweep_p95_us)
            assert len(p95) == 11
            assert r.new_alpha_fp == int(np.argmin(p95)) * W.SCALE // 10
        else:
            assert r.new_alpha_fp == r.alpha_fp


def test_command_line_tuning_host_logic(capsys, monkeypatch):
    # the command line's tuning mode, with the oracle standing in for the
    # CUDA backend: same windows and decisions as the loop driven directly
    import json
    from paper_2505_05286_gb300 import __main__ as cli
    monkeypatch.setattr(T, "gpu_backend", C.oracle_backend)
    assert cli.main(["--tune", "5,20,5", "--seconds", "60,40,60", "--window-s", "20", "--recipe", "0",
                     "--seed", "1"]) == 0
    lines = [json.loads(x) for x in capsys.readouterr().out.strip().splitlines()]
    tr, cl, kw = C.shift_scenario()
    ref = T.OnlineTuner(cl, backend=C.oracle_backend, **kw).run(tr)
    assert len(lines) == len(ref) + 1
    for w, r in zip(lines, ref):
        assert (w["window"], w["queries"], w["p95_us"], w["triggered"], w["p_value"]) == \
               (r.index, r.n_queries, r.p95_us, r.triggered, r.p_value)
        assert round(w["alpha"] * W.SCALE) == r.alpha_fp and round(w["new_alpha"] * W.SCALE) == r.new_alpha_fp
    assert lines[-1]["tunings"] == sum(r.triggered for r in ref)
    with pytest.raises(SystemExit):
        cli.main(["--tune", "5,20", "--seconds", "1,2,3"])
