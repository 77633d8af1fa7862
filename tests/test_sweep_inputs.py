"""Interval constructions and the dataset stand-in of the paper's experiments (Section 6); no GPU."""
from fractions import Fraction

import numpy as np

from paper_2508_14544_gb300 import workloads as W


def test_buckets_edges():
    o = np.array([1, 99, 100, 101, 200, 201, 883, 1000])
    l, u = W.intervals_buckets(o)
    assert l.tolist() == [1, 1, 1, 101, 101, 201, 801, 901]
    assert (u - l).tolist() == [99] * 8
    assert np.all((l <= o) & (o <= u))


def test_rough_contains_every_output():
    o = np.arange(1, 1001)
    l, u = W.intervals_rough(o)
    assert np.all(l == 1) and np.all(u == 1000)


def test_overlap_rounds_outwards_exactly():
    o = np.arange(1, 1001)
    for x in (Fraction(1, 10), Fraction(19, 20), Fraction(99, 100)):
        l, u = W.intervals_overlap(o, x)
        assert np.all((1 <= l) & (l <= o) & (o <= u))
        # exact rational bounds: l = max(1, floor((1-x) o)), u = ceil((1+x) o)
        for oi, li, ui in zip(o[::37], l[::37], u[::37]):
            lo = (1 - x) * int(oi)
            hi = (1 + x) * int(oi)
            assert li == max(1, lo.numerator // lo.denominator)
            assert ui == -((-hi.numerator) // hi.denominator)


def test_lookalike_matches_printed_statistics():
    """Section 6 prints prompt sizes 1..468 (mean 41, median 11, variance 4961) and outputs 1..883
    (mean 85, median 43, variance 9702) for its 2,000 samples; pools of the stand-in agree to the
    sampling noise of 2,000 draws and of the fit (means within 20 %, medians within 25 %,
    variances within 35 %, ranges inside the printed ones)."""
    for seed in range(3):
        s, o = W.lookalike_pool(seed)
        for v, (lo, hi, mean, med, var) in ((s, (1, 468, 41, 11, 4961)), (o, (1, 883, 85, 43, 9702))):
            assert v.min() >= lo and v.max() <= hi
            assert abs(v.mean() - mean) / mean < 0.2
            assert abs(np.median(v) - med) / med < 0.25
            assert abs(v.var() - var) / var < 0.35


def test_sweep_layout_and_reproducibility():
    w1 = W.make_sweep("overlap:1/10", seeds=2)
    w2 = W.make_sweep("overlap:1/10", seeds=2)
    assert w1.n_instances == 20
    assert np.diff(w1.offsets).tolist() == list(range(200, 2001, 200)) * 2
    for a in ("arrival", "prompt", "lower", "upper", "true_o"):
        assert np.array_equal(getattr(w1, a), getattr(w2, a))
    assert np.all(w1.arrival == 0)
    # the subsets of one seed come from one pool: every (s, o) pair of a load-200 instance occurs in
    # the pool of that seed
    s_pool, o_pool = W.lookalike_pool(0)
    pool = set(zip(s_pool.tolist(), o_pool.tolist()))
    lo, hi = int(w1.offsets[0]), int(w1.offsets[1])
    assert set(zip(w1.prompt[lo:hi].tolist(), w1.true_o[lo:hi].tolist())) <= pool
