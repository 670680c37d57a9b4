"""The simulation kernel's integer division (trial quotient from a float
reciprocal, corrected on the exact remainder) against exact division."""
import numpy as np
import pytest

from paper_2505_05286_gb300 import build as B
from paper_2505_05286_gb300 import hxsim as H

pytestmark = pytest.mark.gpu


def _cases(rng, count):
    n = rng.integers(0, 2 ** 63, count, dtype=np.uint64)
    span = rng.integers(0, 54, count)
    d = (rng.integers(0, 2 ** 54, count, dtype=np.uint64) >> span.astype(np.uint64)) + np.uint64(1)
    # quotients near the 2^30 switch, exact multiples, remainders d - 1, d = 1, small d
    k = count // 8
    dd = rng.integers(1, 2 ** 20, k, dtype=np.uint64)
    qq = (np.uint64(2 ** 30) + rng.integers(-3, 3, k).astype(np.int64).astype(np.uint64))
    n[:k], d[:k] = dd * qq + rng.integers(0, 2 ** 20, k, dtype=np.uint64) % dd, dd
    n[k:2 * k] = (n[k:2 * k] % np.uint64(2 ** 40)) // d[k:2 * k] * d[k:2 * k]
    n[2 * k:3 * k] = (n[2 * k:3 * k] % np.uint64(2 ** 40)) // d[2 * k:3 * k] * d[2 * k:3 * k] + d[2 * k:3 * k] - np.uint64(1)
    d[3 * k:4 * k] = 1
    d[4 * k:5 * k] = rng.integers(1, 1000, k, dtype=np.uint64)
    # quotients near the 2^21 switch (one refinement step below it), small and
    # large divisors, any remainder
    d2 = (rng.integers(1, 2 ** 40, k, dtype=np.uint64) >> rng.integers(0, 40, k).astype(np.uint64)) + np.uint64(1)
    q2 = (np.uint64(2 ** 21) + rng.integers(-4, 4, k).astype(np.int64).astype(np.uint64))
    n[5 * k:6 * k], d[5 * k:6 * k] = d2 * q2 + rng.integers(0, 2 ** 62, k, dtype=np.uint64) % d2, d2
    return n, d


def test_division_matches_exact():
    B.build()
    rng = np.random.default_rng(11)
    n, d = _cases(rng, 1 << 22)
    n[:4] = [0, 2 ** 63 - 1, 2 ** 62, 12345]
    d[:4] = [1, 1, 2 ** 54 - 1, 12345]
    q, q_ref = H.selftest_div(n, d)
    want = n // d
    assert (q_ref == want).all()
    bad = np.nonzero(q != want)[0]
    assert bad.size == 0, f"{bad.size} wrong, first n={n[bad[0]]} d={d[bad[0]]} got {q[bad[0]]}"
