"""Per-tenant views of simulation results (the multi-tenant evaluation of Sec. 5).

The library counts SLO hits and completed queries per tenant for every
simulation (`Sim.extras()`); this module turns them into attainment rates
and Jain's fairness index, and gives per-tenant nearest-rank P95 from
per-query latencies (e.g. those of a recorded simulation).

Jain's index of rates x_1..x_n is (sum x)^2 / (n * sum x^2): 1 when every
tenant attains the same fraction, 1/n when one tenant has it all.
"""
from __future__ import annotations

from typing import List, Optional, Sequence

import numpy as np


def attainment(extra_row, n_tenants: int) -> np.ndarray:
    """SLO attainment rate of each of the first n_tenants tenants (0 for a
    tenant without completed queries)."""
    done = np.asarray(extra_row["n_done"][:n_tenants], np.float64)
    met = np.asarray(extra_row["slo_met"][:n_tenants], np.float64)
    return np.where(done > 0, met / np.maximum(done, 1.0), 0.0)


def jain_index(rates: Sequence[float]) -> float:
    x = np.asarray(rates, np.float64)
    if x.size == 0:
        raise ValueError("no rates")
    s2 = float(np.sum(x * x))
    return 1.0 if s2 == 0.0 else float(np.sum(x) ** 2 / (x.size * s2))


def query_latencies(trace, records) -> np.ndarray:
    """Latency of every query of a recorded simulation (`Sim.records`): the
    end of its last call (the evaluation stage) minus its arrival."""
    return np.asarray(records["end"])[np.asarray(trace.call_base)[1:] - 1] - np.asarray(trace.arrival_us)


def tenant_p95(latency_us: Sequence[int], tenant: Optional[Sequence[int]], n_tenants: int) -> List[Optional[int]]:
    """Nearest-rank P95 (sorted L[ceil(0.95 n) - 1]) of each tenant's query
    latencies; None for a tenant without queries."""
    lat = np.asarray(latency_us, np.int64)
    ten = np.zeros(lat.shape[0], np.int64) if tenant is None else np.asarray(tenant, np.int64)
    out: List[Optional[int]] = []
    for t in range(n_tenants):
        s = np.sort(lat[ten == t])
        out.append(int(s[(95 * s.size + 99) // 100 - 1]) if s.size else None)
    return out
