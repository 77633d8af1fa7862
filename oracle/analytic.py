"""Analytic competitive-ratio formulas for A_min (CPU, double precision).

TEST INFRASTRUCTURE ONLY.  Only ``tests/`` and ``bench.py``'s CPU legs may import this module.  It
shares no code with the CUDA evaluators (``csrc/sim_analytic.cu``), which use different methods
(suffix scans; power iteration with O(u) products) on purpose.

* ``lemma_amin_cr(x, l, s)`` - Lemma thm:Amin: the large-M competitive ratio of A_min when a
  fraction x_k of the requests has output length k in [l, u] (all with prompt size s), written
  term by term from the lemma: delta(k) = s + l at k = l and 1 elsewhere; numerator
  sum_k delta(k) (sum_{i>=k} i x_i) (sum_{i>=k} delta(k) x_i/(s+i) + 2 sum_{i>k} (i-k) x_i/(s+i));
  denominator sum_k k (s+k) x_k (x_k + 2 sum_{i>k} x_i).  Plain double loops.
* ``matrices(u)`` - Corollary A/B (s = 0, l = 1): a_ij = min(i,j)^2/(ij) ((i+j)^2/2 - min(i,j)^2),
  b_ij = min(i,j)^2, and ``rayleigh(x)`` = x'Ax / x'Bx.
* ``rho(u)`` - the largest generalized eigenvalue of (A_u, B_u), i.e. the spectral radius of
  B_u^{-1} A_u that bounds the Rayleigh quotient (Section 4.1), by scipy's symmetric generalized
  eigensolver on the dense matrices.
* ``binv_closed(u)`` - the tridiagonal inverse of B_u printed in Section 4.1, as exact Fractions.
* ``lg_cr(q)`` - the closed form of the LG theorem (linearly weighted geometric outputs).
* ``two_point_cr(alpha, t)`` - the two-point form in the proof of Theorem thm:no,
  1 + alpha (1 - alpha^2) t / (alpha^2 t^2 + 2 alpha^2 t + 1), t = x_l / x_u.
"""
from __future__ import annotations

from fractions import Fraction

import numpy as np


def lemma_amin_cr(x, l: int, s: float) -> float:
    """Lemma thm:Amin; x[j] is the mass at output length l + j (u = l + len(x) - 1)."""
    x = [float(v) for v in x]
    u = l + len(x) - 1
    num = 0.0
    den = 0.0
    for k in range(l, u + 1):
        delta = (s + l) if k == l else 1.0
        s_ix = 0.0       # sum_{i>=k} i x_i
        s_frac = 0.0     # sum_{i>=k} x_i / (s + i)
        s_gap = 0.0      # sum_{i>k} (i - k) x_i / (s + i)
        s_after = 0.0    # sum_{i>k} x_i
        for i in range(k, u + 1):
            xi = x[i - l]
            s_ix += i * xi
            s_frac += xi / (s + i)
            if i > k:
                s_gap += (i - k) * xi / (s + i)
                s_after += xi
        num += delta * s_ix * (delta * s_frac + 2.0 * s_gap)
        xk = x[k - l]
        den += k * (s + k) * xk * (xk + 2.0 * s_after)
    return num / den


def matrices(u: int):
    i = np.arange(1, u + 1, dtype=np.float64)[:, None]
    j = i.T
    mn = np.minimum(i, j)
    A = mn ** 2 / (i * j) * (0.5 * (i + j) ** 2 - mn ** 2)
    B = mn ** 2
    return A, B


def rayleigh(x) -> float:
    x = np.asarray(x, dtype=np.float64)
    A, B = matrices(len(x))
    return float(x @ A @ x) / float(x @ B @ x)


def rho(u: int) -> float:
    from scipy.linalg import eigh
    A, B = matrices(u)
    return float(eigh(A, B, eigvals_only=True).max())


def binv_closed(u: int):
    """(B_u)^{-1} as printed: 4i/(4i^2-1) on the diagonal for i < u, 1/(2u-1) at (u, u),
    -1/(2 min(i,j) + 1) on the first off-diagonals, 0 elsewhere (1-based i, j)."""
    m = [[Fraction(0)] * u for _ in range(u)]
    for i in range(1, u + 1):
        m[i - 1][i - 1] = Fraction(4 * i, 4 * i * i - 1) if i < u else Fraction(1, 2 * u - 1)
        if i < u:
            m[i - 1][i] = m[i][i - 1] = Fraction(-1, 2 * i + 1)
    return m


def lg_cr(q: float) -> float:
    return ((1 + q) ** 2 * (1 + 3 * q + 6 * q ** 2 + 3 * q ** 3 + q ** 4)
            / (1 + 2 * q + 11 * q ** 2 + 8 * q ** 3 + 11 * q ** 4 + 2 * q ** 5 + q ** 6))


def two_point_cr(alpha: float, t: float) -> float:
    return 1.0 + alpha * (1.0 - alpha ** 2) * t / (alpha ** 2 * t ** 2 + 2.0 * alpha ** 2 * t + 1.0)
