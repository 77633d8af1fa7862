"""The auxiliary policy A_r (Algorithm random) and the promote-l policy A_ell (Algorithm
promote_l): both CPU oracles against each other, against the brute-force A_r, and against
properties the algorithms fix (no GPU)."""
import itertools
from fractions import Fraction

import numpy as np
import pytest

from oracle import bruteforce as bf
from oracle import literal, plain
from paper_2508_14544_gb300 import workloads as W
from tests import pins

AR, AELL, HSF = literal.AR, literal.AELL, literal.HSF


def _rand_case(rng, n_max=8, o_max=8, s_max=4, arrivals=True):
    n = int(rng.integers(1, n_max + 1))
    o = rng.integers(1, o_max + 1, n)
    l = np.array([rng.integers(1, x + 1) for x in o])
    u = o + rng.integers(0, 6, n)
    s = rng.integers(1, s_max + 1, n)
    a = rng.integers(0, 6, n) if arrivals else np.zeros(n, int)
    M = int(max(s + u) + rng.integers(0, 14))
    return M, a, s, l, u, o


def _same(r1, r2):
    return all(r1[k] == r2[k] for k in pins.FIELDS + ("status",)) and r1["completion"] == r2["completion"]


def test_literal_equals_plain_random():
    rng = np.random.default_rng(77)
    for trial in range(400):
        M, a, s, l, u, o = _rand_case(rng, arrivals=bool(trial % 2))
        rank = rng.permutation(len(o))
        r1 = literal.simulate(AR, M, a, s, l, u, o, rank=rank)
        r2 = plain.run(AR, M, a, s, l, u, o, completions=True, rank=rank)
        assert _same(r1, r2), ("AR", M, a.tolist(), s.tolist(), o.tolist(), rank.tolist())
        r1 = literal.simulate(AELL, M, a, s, l, u, o)
        r2 = plain.run(AELL, M, a, s, l, u, o, completions=True)
        assert _same(r1, r2), ("AELL", M, a.tolist(), s.tolist(), l.tolist(), u.tolist(), o.tolist())


def test_literal_equals_plain_c1_and_online():
    w = W.make_workload("c1")
    inst = w.instance(0)
    rank = w.ranks()
    for p in (AR, AELL):
        r1 = literal.simulate(p, inst["M"], inst["a"], inst["s"], inst["l"], inst["u"], inst["o"], rank=rank)
        r2 = plain.run(p, inst["M"], inst["a"], inst["s"], inst["l"], inst["u"], inst["o"], completions=True,
                       rank=rank)
        assert _same(r1, r2)
    rng = np.random.default_rng(19)
    n = 60
    s = rng.integers(1, 30, n)
    o = rng.integers(1, 40, n)
    l, u = W.interval_for(o, Fraction(3, 10), rng)
    a = np.floor(np.cumsum(rng.exponential(0.7, n))).astype(int)
    rank = rng.permutation(n)
    for p in (AR, AELL):
        r1 = literal.simulate(p, 400, a, s, l, u, o, rank=rank)
        r2 = plain.run(p, 400, a, s, l, u, o, completions=True, rank=rank)
        assert _same(r1, r2)


def test_ar_shortest_first_is_hsf():
    """A_r with the permutation sorted by (o, index) makes the same decisions as H-SF."""
    rng = np.random.default_rng(5)
    for _ in range(200):
        M, a, s, l, u, o = _rand_case(rng, n_max=10)
        perm = bf.shortest_first_perm(o)
        rank = np.empty(len(o), int)
        rank[perm] = np.arange(len(o))
        assert _same(plain.run(AR, M, a, s, l, u, o, completions=True, rank=rank),
                     plain.run(HSF, M, a, s, l, u, o, completions=True))


def test_ar_matches_bruteforce_every_permutation():
    """For tiny instances, every permutation: the oracles' A_r equals the brute-force module's
    A_r (an explicit per-step memory profile, no shared code), completions included; the mean
    over all n! permutations is E[TEL(A_r)] and lies between OPT_perm and the worst order."""
    rng = np.random.default_rng(31)
    for _ in range(12):
        M, a, s, l, u, o = _rand_case(rng, n_max=5, o_max=5, arrivals=bool(rng.integers(0, 2)))
        n = len(o)
        tels = []
        for perm in itertools.permutations(range(n)):
            rank = np.empty(n, int)
            rank[list(perm)] = np.arange(n)
            ref = bf.a_random(M, a, s, o, perm)
            r = literal.simulate(AR, M, a, s, l, u, o, rank=rank)
            assert r["completion"] == ref["completion"] and r["total_latency"] == ref["total_latency"]
            tels.append(r["total_latency"])
        assert bf.opt_perm(M, a, s, o) == min(tels)
        assert min(tels) <= np.mean(tels) <= max(tels)
        assert min(tels) >= bf.opt_exact(M, a, s, o)


def test_aell_counts_fixed_by_the_algorithm():
    """Each request with o > l is promoted exactly once (its estimate becomes u >= o), a request
    with o = l never is: evictions = #{o > l}, and the tokens wasted are exactly l per promoted
    request: request steps = sum o + sum_{o > l} l.  Memory stays within M; TEL >= sum o."""
    rng = np.random.default_rng(41)
    for _ in range(300):
        M, a, s, l, u, o = _rand_case(rng, n_max=12, o_max=12)
        r = plain.run(AELL, M, a, s, l, u, o, completions=True)
        assert r["status"] == 0
        longer = o > l
        assert r["evictions"] == int(longer.sum())
        assert r["request_steps"] == int(o.sum() + l[longer].sum())
        assert r["peak_memory"] <= M
        assert all(c - ai >= oi for c, ai, oi in zip(r["completion"], a, o))


def test_aell_exact_lower_bounds_is_fifo_ar():
    """With l = o nothing is ever promoted: A_ell is the FIFO queue with true lengths, i.e. A_r
    whose permutation is the order of (arrival, index)."""
    rng = np.random.default_rng(43)
    for _ in range(200):
        M, a, s, l, u, o = _rand_case(rng, n_max=10)
        order = sorted(range(len(o)), key=lambda i: (a[i], i))
        rank = np.empty(len(o), int)
        rank[order] = np.arange(len(o))
        assert _same(plain.run(AELL, M, a, s, o, u, o, completions=True),
                     plain.run(AR, M, a, s, o, u, o, completions=True, rank=rank))


def test_aell_and_ar_not_below_optimum():
    rng = np.random.default_rng(47)
    for _ in range(25):
        M, a, s, l, u, o = _rand_case(rng, n_max=5, o_max=5)
        opt = bf.opt_exact(M, a, s, o)
        assert literal.simulate(AELL, M, a, s, l, u, o)["total_latency"] >= opt
        assert literal.simulate(AR, M, a, s, l, u, o, rank=rng.permutation(len(o)))["total_latency"] >= opt


def _d2(n_l, n_u, l, u, s, M, seed):
    rng = np.random.default_rng(seed)
    o = np.array([l] * n_l + [u] * n_u)
    rng.shuffle(o)
    n = n_l + n_u
    return M, np.zeros(n, int), np.full(n, s), np.full(n, l), np.full(n, u), o


@pytest.mark.parametrize("n_l,n_u,l,u", [(2000, 2000, 20, 100), (3000, 1000, 50, 100),
                                         (1000, 3000, 10, 100), (2000, 2000, 60, 100)])
def test_aell_two_point_ratio_matches_the_fluid_formula(n_l, n_u, l, u):
    """Proof of the A_ell theorem (two-point family): TEL(A_ell)/TEL(H-SF) = 1 + (a^2 x_l x_u +
    2 a^2 x_u^2) / (a^2 x_l^2 + 2 a^2 x_l x_u + x_u^2) + O(1/M), a = l/u, x = request counts.
    4000 requests, s = 1, M = 4000: the simulated ratio is within 0.02 of the formula."""
    M, a, s, lo, up, o = _d2(n_l, n_u, l, u, 1, 4000, 1)
    al = l / u
    cr = 1 + (al ** 2 * n_l * n_u + 2 * al ** 2 * n_u ** 2) / (al ** 2 * n_l ** 2 + 2 * al ** 2 * n_l * n_u + n_u ** 2)
    sim = plain.run(AELL, M, a, s, lo, up, o)["total_latency"] / plain.run(HSF, M, a, s, lo, up, o)["total_latency"]
    assert abs(sim - cr) < 0.02, (sim, cr)
    bound = 1 + al / (2 * (1 - al)) if al <= 0.5 else 1 + 2 * al ** 2
    assert sim <= bound + 0.02


@pytest.mark.parametrize("n_l,n_u,l,u", [(2000, 2000, 20, 100), (1000, 3000, 50, 100)])
def test_ar_two_point_ratio_within_theorem_bound(n_l, n_u, l, u):
    """Theorem on A_r (worst-case realizations): E[TEL(A_r)]/TEL(H-SF) <= (1 + 1/a)/2 + O(1/M);
    three random permutations of a 4000-request two-point instance stay below the bound."""
    M, a, s, lo, up, o = _d2(n_l, n_u, l, u, 1, 4000, 2)
    hsf = plain.run(HSF, M, a, s, lo, up, o)["total_latency"]
    rng = np.random.default_rng(3)
    mean = np.mean([plain.run(AR, M, a, s, lo, up, o, rank=rng.permutation(len(o)))["total_latency"]
                    for _ in range(3)])
    assert mean / hsf <= (1 + u / l) / 2 + 0.02
