"""A_min's random eviction ties (Algorithm milb / milbrevise: "break ties uniformly at random"),
pinned on the CPU oracles (no GPU).

* The counter-based generator (SplitMix64) of both oracles reproduces the published outputs of
  its reference implementation, and its counter layout (step in the high word) follows from the
  generator's additive state.
* Theorem thm:no (Section 5, two-point output lengths): CR(A_min) <= (3 - alpha)/2 + O(1/M).  The
  mean ratio TEL(A_min)/TEL(H-SF) over seeded two-point instances stays under the bound with the
  random tie rule, and the index tie rule breaks it (so the pin can tell the two apart).
* Literal and plain oracles agree on instances full of ties.
* Admission keeps ties by index; a per-step random admission order changes the mean ratio by
  less than 0.02 on the same instances (the sensitivity of that reading).
"""
from fractions import Fraction

import numpy as np
import pytest

from oracle import literal, plain
from paper_2508_14544_gb300 import workloads as W
from tests import pins

GAMMA = 0x9E3779B97F4A7C15
MASK = (1 << 64) - 1


def two_point(n, M, l, u, frac_long, seeds, seed0=900):
    """n requests at t=0 with s = 1 and o in {l, u} (long with probability frac_long), interval
    [l, u] for every request: the family D_2 of Section 5."""
    parts = []
    for sd in seeds:
        rng = np.random.default_rng([777, sd])
        o = np.where(rng.random(n) < frac_long, u, l)
        parts.append(dict(a=np.zeros(n, int), s=np.ones(n, int), l=np.full(n, l), u=np.full(n, u), o=o))
    w = W.concat_instances("two-point", M, parts)
    w.seed0 = seed0
    return w


def test_splitmix64_published_vectors():
    for v in pins.load("splitmix64.json")["vectors"]:
        outs = [int(x, 16) for x in v["outputs_hex"]] if "outputs_hex" in v else [int(x) for x in v["outputs"]]
        for k, z in enumerate(outs, start=1):
            assert literal.splitmix64(v["seed"], k) == z
            assert literal.tie_key(v["seed"], 0, k - 1) == z >> 32
            assert plain.tie_key(v["seed"], 0, k - 1) == z >> 32


@pytest.mark.parametrize("seed,t,i", [(0, 1, 0), (5, 17, 3), (MASK, 123456, 99999), (1234567, 2**31 - 5, 7)])
def test_tie_key_counter_layout(seed, t, i):
    """SplitMix64's state after k steps is seed + k * gamma, so output t*2^32 + i + 1 of a seed is
    output i + 1 of the seed advanced by t*2^32 steps."""
    moved = (seed + (t << 32) * GAMMA) & MASK
    for key in (literal.tie_key, plain.tie_key):
        assert key(seed, t, i) == key(moved, 0, i)


# Two-point instances: (n, M, l, u); half of the requests long, 8 seeds each.
TWO_POINT = [(4000, 4000, 5, 10), (2000, 2000, 10, 20)]


def _mean_ratio(n, M, l, u, evict_ties):
    w = two_point(n, M, l, u, 0.5, range(8))
    h = plain.run_workload(2, w, n_threads=8)["total_latency"].astype(np.float64)
    r = plain.run_workload(1, w, n_threads=8, evict_ties=evict_ties)
    assert np.all(r["status"] == 0)
    return float(np.mean(r["total_latency"].astype(np.float64) / h))


@pytest.mark.parametrize("n,M,l,u", TWO_POINT)
def test_two_point_ratio_under_theorem_bound(n, M, l, u):
    """Theorem thm:no: the mean of TEL(A_min)/TEL(H-SF) over seeds stays below (3 - alpha)/2."""
    bound = float((3 - Fraction(l, u)) / 2)
    assert _mean_ratio(n, M, l, u, "hash") < bound - 0.03


@pytest.mark.parametrize("n,M,l,u", TWO_POINT)
def test_index_tie_rule_breaks_theorem_bound(n, M, l, u):
    """The rule of breaking eviction ties by request index cancels the most advanced of the tied
    jobs every time (admission starts tied jobs in index order); it fails the same pin."""
    bound = float((3 - Fraction(l, u)) / 2)
    assert _mean_ratio(n, M, l, u, "index") > bound + 0.05


def test_literal_equals_plain_on_ties():
    w = two_point(300, 300, 5, 10, 0.5, range(6))
    seeds = w.tie_seeds()
    ref = plain.run_workload(1, w, completions=True)
    for r in range(w.n_instances):
        inst = w.instance(r)
        got = literal.simulate(1, w.M, inst["a"], inst["s"], inst["l"], inst["u"], inst["o"],
                               tie_seed=int(seeds[r]))
        for f in pins.FIELDS:
            assert got[f] == int(ref[0][r][f]), (r, f)
        lo, hi = int(w.offsets[r]), int(w.offsets[r + 1])
        assert got["completion"] == ref[1][lo:hi].tolist()
        assert got["evictions"] > 0


@pytest.mark.parametrize("l,u", [(5, 10), (2, 10)])
def test_admission_tie_reading_sensitivity(l, u):
    """Admission ties by index (a fixed random order of the i.i.d. requests) against a fresh random
    order at every step: the mean ratio moves by less than 0.02."""
    w = two_point(300, 300, l, u, 0.5, range(16))
    seeds = w.tie_seeds()
    h = plain.run_workload(2, w)["total_latency"].astype(np.float64)
    diff = []
    for r in range(w.n_instances):
        inst = w.instance(r)
        args = (1, w.M, inst["a"], inst["s"], inst["l"], inst["u"], inst["o"])
        a = literal.simulate(*args, tie_seed=int(seeds[r]))["total_latency"]
        b = literal.simulate(*args, tie_seed=int(seeds[r]), admit_ties="hash")["total_latency"]
        diff.append((b - a) / h[r])
    assert abs(float(np.mean(diff))) < 0.02
