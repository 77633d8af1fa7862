"""Invariants and literal == plain agreement (no GPU)."""
import numpy as np
import pytest

from oracle import literal, plain
from paper_2508_14544_gb300 import workloads as W
from tests import pins


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
    rng = np.random.default_rng(2024)
    for trial in range(400):
        M, a, s, l, u, o = _rand_case(rng, arrivals=bool(trial % 2))
        for p in (0, 1, 2):
            r1 = literal.simulate(p, M, a, s, l, u, o, tie_seed=trial)
            r2 = plain.run(p, M, a, s, l, u, o, completions=True, tie_seed=trial)
            assert _same(r1, r2), (p, M, a.tolist(), s.tolist(), l.tolist(), u.tolist(), o.tolist())


def test_literal_equals_plain_c1():
    inst = W.make_instance("c1", 0)
    for p in (0, 1, 2):
        r1 = literal.simulate(p, inst["M"], inst["a"], inst["s"], inst["l"], inst["u"], inst["o"])
        r2 = plain.run(p, inst["M"], inst["a"], inst["s"], inst["l"], inst["u"], inst["o"], completions=True)
        assert _same(r1, r2)


def test_literal_equals_plain_scaled_online():
    """A scaled-down online instance with heterogeneous s (shape of the Poisson workloads)."""
    rng = np.random.default_rng(9)
    n = 60
    s = rng.integers(1, 30, n)
    o = rng.integers(1, 40, n)
    from fractions import Fraction
    l, u = W.interval_for(o, Fraction(3, 10), rng)
    a = np.floor(np.cumsum(rng.exponential(0.7, n))).astype(int)
    M = 400
    for p in (0, 1, 2):
        r1 = literal.simulate(p, M, a, s, l, u, o)
        r2 = plain.run(p, M, a, s, l, u, o, completions=True)
        assert _same(r1, r2)


def test_invariants_random():
    """A_max and H-SF never cancel and do exactly sum(o) tokens of work; every policy keeps the
    memory of each step within M (peak <= M); TEL >= sum(o)."""
    rng = np.random.default_rng(7)
    for _ in range(300):
        M, a, s, l, u, o = _rand_case(rng, n_max=12, o_max=12)
        for p in (0, 1, 2):
            r = plain.run(p, M, a, s, l, u, o, completions=True)
            assert r["status"] == 0
            assert r["peak_memory"] <= M
            assert r["total_latency"] >= int(np.sum(o))
            assert r["makespan"] == max(r["completion"])
            assert all(c - ai >= oi for c, ai, oi in zip(r["completion"], a, o))
            if p in (0, 2):
                assert r["evictions"] == 0
                assert r["request_steps"] == int(np.sum(o))
            else:
                assert r["request_steps"] >= int(np.sum(o))


def test_exact_intervals_make_policies_equal():
    """l = u = o: all three keys coincide and A_min never overflows, so the three policies give
    identical outputs (Section 4: with exact predictions A_min reduces to the hindsight rule)."""
    rng = np.random.default_rng(11)
    for _ in range(200):
        M, a, s, l, u, o = _rand_case(rng, n_max=12, o_max=10)
        res = [plain.run(p, M, a, s, o, o, o, completions=True) for p in (0, 1, 2)]
        assert _same(res[0], res[1]) and _same(res[1], res[2])
        assert res[1]["evictions"] == 0


def test_exact_intervals_c2_alpha1_instances():
    """The alpha = 1 quarter of the 1024-instance workload has exact intervals."""
    w = W.make_workload("c2", [768, 769, 1023])
    outs = [plain.run_workload(p, w) for p in (0, 1, 2)]
    for f in pins.FIELDS:
        assert np.array_equal(outs[0][f], outs[1][f]) and np.array_equal(outs[1][f], outs[2][f])


def test_amin_bounds_never_decrease():
    """Trace check: an evicted job's lower bound never drops and stays <= o (Section 4)."""
    rng = np.random.default_rng(13)
    for _ in range(100):
        M, a, s, l, u, o = _rand_case(rng, n_max=10, o_max=10, arrivals=False)
        tr = []
        literal.simulate(literal.AMIN, M, a, s, l, u, o, trace=tr)  # asserts bound <= o inside
        # every request completes exactly once
        fin = [i for rec in tr for i in rec["finished"]]
        assert sorted(fin) == list(range(len(o)))


def test_plain_batch_matches_single():
    w = W.make_workload("c2", [0, 300, 600, 900])
    for p in (0, 1, 2):
        rb = plain.run_workload(p, w, n_threads=4)
        seeds = w.tie_seeds()
        for i in range(w.n_instances):
            inst = w.instance(i)
            r = plain.run(p, inst["M"], inst["a"], inst["s"], inst["l"], inst["u"], inst["o"],
                          tie_seed=int(seeds[i]))
            for f in pins.FIELDS + ("status",):
                assert int(rb[i][f]) == r[f]
