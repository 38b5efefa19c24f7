"""The Jensen-Shannon evaluation used by the teacher-selection kernel (Eq. 2), checked in
float64 on the CPU.

With m = (p + q)/2 and d = (p - q)/(p + q), each token contributes
  p ln(p/m) + q ln(q/m) = m phi(d),  phi(d) = (1 + d) ln(1 + d) + (1 - d) ln(1 - d),
so D_JS = 1/2 sum_n m_n phi(d_n) = 1/4 sum_n (p_n + q_n) phi(d_n).  For |d| < 1/4 phi is taken
from its even power series sum_k d^(2k) / (k (2k - 1)) cut after six terms, which avoids the
cancellation of the two logarithms when p is close to q; the cut costs below 1e-9 relative."""
import math

import numpy as np
import pytest

scipy_distance = pytest.importorskip("scipy.spatial.distance")


def _series(d, terms):
    u = d * d
    return sum(u ** k / (k * (2 * k - 1)) for k in range(1, terms + 1))


def _closed(d):
    return (1 + d) * math.log1p(d) + (1 - d) * math.log1p(-d)


def test_six_terms_are_within_1e9_relative_below_a_quarter():
    for d in np.linspace(1e-4, 0.2499, 2000):
        full = _series(d, 60)
        assert abs(_series(d, 6) - full) <= 1e-9 * full
        assert abs(_series(-d, 6) - full) <= 1e-9 * full


def test_series_is_phi():
    for d in np.linspace(0.05, 0.2499, 200):
        assert _series(d, 60) == pytest.approx(_closed(d), rel=1e-12)


def test_quarter_sum_is_the_jensen_shannon_divergence():
    rng = np.random.default_rng(0)
    for _ in range(20):
        p = rng.dirichlet(np.full(50, 0.7))
        q = rng.dirichlet(np.full(50, 0.7))
        t = p + q
        d = (p - q) / t
        phi = np.array([_series(x, 60) if abs(x) < 0.25 else _closed(x) for x in d])
        js = 0.25 * float(np.sum(t * phi))
        assert js == pytest.approx(scipy_distance.jensenshannon(p, q) ** 2, rel=1e-10)


def test_disjoint_supports_give_ln2():
    p = np.array([1.0, 0.0])
    q = np.array([0.0, 1.0])
    t = p + q
    d = (p - q) / t                                 # d = +-1: phi(+-1) = 2 ln 2
    js = 0.25 * float(np.sum(t * np.array([_closed(x) if abs(x) < 1 else 2 * math.log(2) for x in d])))
    assert js == pytest.approx(math.log(2), rel=1e-15)
