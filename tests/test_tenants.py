"""Host-side per-tenant views: Jain's fairness index and per-tenant P95,
pinned by closed forms and the hand-worked two-tenant schedule."""
import pytest

import oracle
from paper_2505_05286_gb300 import tenants as T
from tests import cases


def test_jain_closed_forms():
    assert T.jain_index([1.0, 1.0]) == 1.0
    assert T.jain_index([0.7, 0.7, 0.7]) == pytest.approx(1.0)
    assert T.jain_index([1.0, 0.0]) == 0.5
    assert T.jain_index([1.0, 0.0, 0.0, 0.0]) == 0.25
    # (0.9 + 0.6)^2 / (2 * (0.81 + 0.36)) = 2.25 / 2.34
    assert T.jain_index([0.9, 0.6]) == pytest.approx(2.25 / 2.34)
    # scale invariance
    assert T.jain_index([0.2, 0.4, 0.8]) == pytest.approx(T.jain_index([1, 2, 4]))
    assert T.jain_index([0.0, 0.0]) == 1.0


def test_two_tenant_hand_case():
    """The hand-worked schedule: q0 (tenant 0, T_slo 6000) misses at 10000,
    q1 (tenant 1, T_slo 12000) meets at 12000: attainment (0, 1), Jain 0.5."""
    tr, cl, exp = cases.hand_case("H8_tenants")
    res, log, ext = oracle.simulate(tr, cl, exp["point"], log=True, extra=True)
    rates = T.attainment(ext, 2)
    assert rates.tolist() == [0.0, 1.0]
    assert T.jain_index(rates) == 0.5
    lat = log["end"][tr.call_base[1:] - 1] - tr.arrival_us
    assert T.tenant_p95(lat, tr.tenant, 2) == [10000, 12000]


def test_tenant_p95_nearest_rank():
    lat = list(range(1, 101)) + [1000] * 20
    ten = [0] * 100 + [1] * 20
    assert T.tenant_p95(lat, ten, 3) == [95, 1000, None]
