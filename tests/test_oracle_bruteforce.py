"""Tiny instances checked against exhaustive optima (no GPU).

OPT_exact (every feasible non-preemptive schedule) <= OPT_perm (best order of the auxiliary
policy A_r, Algorithm random) <= TEL(H-SF) = TEL(A_r with the shortest-first order), and every
policy's TEL is at least OPT_exact: A_max and H-SF never cancel, and A_min's final runs are a
subset of what it runs at each step, so they form a feasible schedule too.
"""
import numpy as np
import pytest

from oracle import bruteforce as bf
from oracle import literal, plain


def _tiny(rng, n_max=5, o_max=5, s_max=3, arrivals=False):
    n = int(rng.integers(1, n_max + 1))
    o = rng.integers(1, o_max + 1, n)
    l = np.array([rng.integers(1, x + 1) for x in o])
    u = o + rng.integers(0, 4, n)
    s = rng.integers(1, s_max + 1, n)
    a = rng.integers(0, 3, n) if arrivals else np.zeros(n, int)
    M = int(max(s + u) + rng.integers(0, 8))
    return M, a.tolist(), s.tolist(), l.tolist(), u.tolist(), o.tolist()


@pytest.mark.parametrize("arrivals", [False, True])
def test_tel_bounds_random_tiny(arrivals):
    rng = np.random.default_rng(1234 + arrivals)
    for _ in range(60):
        M, a, s, l, u, o = _tiny(rng, arrivals=arrivals)
        opt = bf.opt_exact(M, a, s, o)
        hsf = literal.simulate(literal.HSF, M, a, s, l, u, o)
        ar_sf = bf.a_random(M, a, s, o, bf.shortest_first_perm(o))
        assert hsf["total_latency"] == ar_sf["total_latency"]
        assert hsf["completion"] == ar_sf["completion"]
        if len(o) <= 5:
            operm = bf.opt_perm(M, a, s, o)
            assert opt <= operm <= hsf["total_latency"]
        for p in (literal.AMAX, literal.AMIN, literal.HSF):
            r = literal.simulate(p, M, a, s, l, u, o)
            assert r["total_latency"] >= opt, (p, M, a, s, l, u, o)
            q = plain.run(p, M, a, s, l, u, o)
            assert q["total_latency"] == r["total_latency"]


def test_opt_exact_n7():
    rng = np.random.default_rng(77)
    for _ in range(4):
        n = 7
        o = rng.integers(1, 4, n).tolist()
        s = rng.integers(1, 3, n).tolist()
        M = int(max(np.add(s, o)) + rng.integers(2, 6))
        a = [0] * n
        opt = bf.opt_exact(M, a, s, o)
        for p in (literal.AMAX, literal.AMIN, literal.HSF):
            r = plain.run(p, M, a, s, o, o, o)
            assert r["total_latency"] >= opt


def test_opt_exact_small_closed_forms():
    # a single job: TEL = o
    assert bf.opt_exact(10, [0], [2], [5]) == 5
    # two jobs that cannot overlap at all: M = s+o of one job, run back to back
    assert bf.opt_exact(4, [0, 0], [1, 1], [3, 3]) == 3 + 6
    # arrivals: a job arriving at 5 alone: latency o
    assert bf.opt_exact(10, [5], [1], [2]) == 2
