"""The online tuning loop driven by the CUDA library makes exactly the
decisions it makes when driven by the oracle."""
import pytest

from paper_2505_05286_gb300 import build as B
from paper_2505_05286_gb300 import tuner as T
from tests import tuner_cases as C

pytestmark = pytest.mark.gpu


def test_gpu_loop_matches_oracle_loop():
    B.build()
    tr, cl, kw = C.shift_scenario()
    gpu = T.OnlineTuner(cl, backend=T.gpu_backend, **kw).run(tr)
    ref = T.OnlineTuner(cl, backend=C.oracle_backend, **kw).run(tr)
    assert len(gpu) == len(ref)
    for g, r in zip(gpu, ref):
        assert (g.alpha_fp, g.p95_us, g.triggered, g.new_alpha_fp, g.sweep_p95_us) == \
               (r.alpha_fp, r.p95_us, r.triggered, r.new_alpha_fp, r.sweep_p95_us)
        assert g.p_value == r.p_value
    assert any(g.triggered for g in gpu)


def test_command_line_tuning(capsys):
    import json
    from paper_2505_05286_gb300 import __main__ as cli
    from paper_2505_05286_gb300 import workloads as W
    B.build()
    # the same trace, cluster, windows and beta as the shift scenario
    assert cli.main(["--tune", "5,20,5", "--seconds", "60,40,60", "--window-s", "20", "--recipe", "0",
                     "--seed", "1"]) == 0
    lines = [json.loads(x) for x in capsys.readouterr().out.strip().splitlines()]
    wins, summary = lines[:-1], lines[-1]
    tr, cl, kw = C.shift_scenario()
    ref = T.OnlineTuner(cl, backend=C.oracle_backend, **kw).run(tr)
    assert len(wins) == len(ref) == summary["windows"] and summary["queries"] == tr.n_queries
    for w, r in zip(wins, ref):
        assert (w["queries"], w["p95_us"], w["triggered"]) == (r.n_queries, r.p95_us, r.triggered)
        assert round(w["new_alpha"] * W.SCALE) == r.new_alpha_fp
        assert (w["tune_ms"] is not None) == r.triggered
    assert summary["tunings"] == sum(r.triggered for r in ref) > 0
    assert summary["tune_ms_max"] > 0
