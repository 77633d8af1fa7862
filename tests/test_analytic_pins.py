"""Pins of the analytic competitive-ratio oracle (oracle/analytic.py) to what the paper and the
mathematics fix (no GPU)."""
from fractions import Fraction

import numpy as np
import pytest

from oracle import analytic as an


def _exact_AB(u):
    A = [[Fraction(min(i, j) ** 2, i * j) * (Fraction((i + j) ** 2, 2) - min(i, j) ** 2)
          for j in range(1, u + 1)] for i in range(1, u + 1)]
    B = [[Fraction(min(i, j) ** 2) for j in range(1, u + 1)] for i in range(1, u + 1)]
    return A, B


@pytest.mark.parametrize("u", [1, 2, 3, 5, 8, 12])
def test_binv_closed_form_and_trace_is_harmonic(u):
    """Section 4.1: the printed tridiagonal matrix is exactly B_u^{-1}, and
    tr(B_u^{-1} A_u) = H_u = sum_{i<=u} 1/i, in exact rational arithmetic."""
    A, B = _exact_AB(u)
    Bi = an.binv_closed(u)
    for i in range(u):
        for j in range(u):
            assert sum(Bi[i][k] * B[k][j] for k in range(u)) == (1 if i == j else 0)
    tr = sum(Bi[i][k] * A[k][i] for i in range(u) for k in range(u))
    assert tr == sum(Fraction(1, i) for i in range(1, u + 1))


@pytest.mark.parametrize("q", [0.0, 0.1, 0.3, 0.5, 0.7, 0.85])
def test_lemma_reproduces_the_lg_theorem(q):
    """The LG theorem's closed form is the lemma evaluated on P(o = k) ~ k q^(k-1), s = 0, l = 1
    (u -> infinity; truncated at u = 600, where the tail is below 1e-30)."""
    u = 600
    x = [k * q ** (k - 1) for k in range(1, u + 1)]
    assert abs(an.lemma_amin_cr(x, 1, 0.0) - an.lg_cr(q)) < 1e-12


def test_lg_endpoints():
    """1 at q = 0; 14/9 at q = 1, the theorem's bound; increasing in between."""
    assert an.lg_cr(0.0) == 1.0
    assert abs(an.lg_cr(1.0) - 14 / 9) < 1e-15
    qs = np.linspace(0, 1, 101)
    v = [an.lg_cr(q) for q in qs]
    assert all(b >= a - 1e-15 for a, b in zip(v, v[1:]))


@pytest.mark.parametrize("l,u", [(1, 2), (2, 10), (3, 7), (5, 50)])
def test_lemma_two_point_form_and_its_maximum(l, u):
    """Proof of Theorem thm:no: on x = (x_l, 0, .., 0, x_u), s = 0, the lemma equals
    1 + a(1 - a^2)t/(a^2 t^2 + 2a^2 t + 1) (a = l/u, t = x_l/x_u), whose maximum over t, reached
    at t = 1/a, is 1 + (1 - a)/2."""
    a = l / u
    for t in (0.01, 0.5, 1 / a, 2.0, 40.0):
        x = [0.0] * (u - l + 1)
        x[0], x[-1] = t, 1.0
        assert abs(an.lemma_amin_cr(x, l, 0.0) - an.two_point_cr(a, t)) < 1e-12
    ts = np.linspace(0.0, 4.0 / a, 2001)
    best = max(an.two_point_cr(a, t) for t in ts)
    assert abs(an.two_point_cr(a, 1 / a) - (1 + (1 - a) / 2)) < 1e-12
    assert best <= 1 + (1 - a) / 2 + 1e-12


def test_rayleigh_form_equals_the_lemma():
    """Corollary A/B: for s = 0 and l = 1 the lemma is the Rayleigh quotient x'A_u x / x'B_u x."""
    rng = np.random.default_rng(3)
    for u in (1, 2, 5, 17, 64):
        for _ in range(5):
            x = rng.random(u)
            assert abs(an.lemma_amin_cr(x, 1, 0.0) - an.rayleigh(x)) < 1e-12


def test_point_mass_at_l_is_one():
    """All outputs at the lower bound: A_min never cancels and runs like the hindsight rule."""
    for l, u, s in ((1, 5, 0.0), (3, 9, 2.0)):
        x = [1.0] + [0.0] * (u - l)
        assert abs(an.lemma_amin_cr(x, l, s) - 1.0) < 1e-15


@pytest.mark.parametrize("u", [2, 10, 100, 1000])
def test_rho_bounds_and_fit(u):
    """Section 4.1: the Rayleigh quotient is at most rho(B^{-1}A) <= tr = H_u; random positive
    histograms stay below rho; the figure's fit 0.2555 log(u + 0.2793) + 1.1587 is within 2 %
    for u >= 10."""
    r = an.rho(u)
    h = sum(1 / i for i in range(1, u + 1))
    assert 1.0 <= r <= h + 1e-9
    rng = np.random.default_rng(u)
    for _ in range(3):
        x = rng.random(u)
        assert an.rayleigh(x) <= r + 1e-9
    if u >= 10:
        fit = 0.2555 * np.log(u + 0.2793) + 1.1587
        assert abs(r - fit) / fit < 0.02
