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
