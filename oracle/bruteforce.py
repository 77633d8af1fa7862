"""Exact optima for tiny instances, used to pin the oracle's schedules from outside.

TEST INFRASTRUCTURE ONLY.  Only ``tests/`` may import this module.

* ``opt_exact``  - minimum TEL over *all* non-preemptive schedules that respect the memory limit
                   at every step (eq. constraintM under the W reading: a job started at p occupies
                   steps p..p+o-1 with memory s+1..s+o), found by exhaustive dynamic programming
                   over (step, running jobs with their starts, not-yet-started set).  Idling is
                   allowed, so with arrivals the optimum may wait for a short job.
* ``a_random``   - the auxiliary policy A_r (Algorithm random, Appendix B): fix a permutation,
                   and at every step add waiting jobs in permutation order, with the true output
                   lengths, while the future memory stays within M; stop at the first job that
                   does not fit.  It keeps an explicit per-step memory profile, so it shares no
                   feasibility code with ``literal.py``.
* ``opt_perm``   - minimum of A_r's TEL over all n! permutations.

Relations the tests assert (they pin the oracle without using it):
OPT_exact <= OPT_perm <= TEL(H-SF) = TEL(A_r with the shortest-first permutation), and
TEL(pi) >= OPT_exact for every policy pi (A_min too: the final runs of its jobs form a
feasible schedule, because they are a subset of what runs at every step).
"""
from __future__ import annotations

import itertools
from functools import lru_cache
from typing import Sequence

INF = float("inf")


def _running_fits(M: int, s, o, running: tuple, t: int) -> bool:
    """Exact future memory of jobs already started (true lengths), for every step >= t."""
    if not running:
        return True
    end = max(p + o[i] - 1 for i, p in running)
    for tp in range(t, end + 1):
        tot = 0
        for i, p in running:
            if p <= tp <= p + o[i] - 1:
                tot += s[i] + (tp - p) + 1
        if tot > M:
            return False
    return True


def opt_exact(M: int, a: Sequence[int], s: Sequence[int], o: Sequence[int]) -> int:
    """Minimum TEL = sum(C_i - a_i) over every feasible non-preemptive schedule."""
    n = len(o)
    a = tuple(int(x) for x in a)
    s = tuple(int(x) for x in s)
    o = tuple(int(x) for x in o)
    if any(s[i] + o[i] > M for i in range(n)):
        raise ValueError("infeasible instance")
    t_max = max(a) + sum(o) + 1  # a serial schedule finishes all starts before this

    @lru_cache(maxsize=None)
    def best(t: int, running: tuple, waiting: frozenset) -> float:
        if not waiting:
            return sum(p + o[i] - a[i] for i, p in running)
        if t > t_max:
            return INF
        arrived = sorted(i for i in waiting if a[i] <= t)
        if not running and not arrived:
            return best(min(a[i] for i in waiting), running, waiting)
        res = INF
        for r in range(len(arrived) + 1):
            for U in itertools.combinations(arrived, r):
                now = running + tuple((i, t) for i in U)
                if not _running_fits(M, s, o, now, t):
                    continue
                fin = sum(p + o[i] - a[i] for i, p in now if p + o[i] - 1 == t)
                still = tuple(sorted((i, p) for i, p in now if p + o[i] - 1 > t))
                res = min(res, fin + best(t + 1, still, waiting - frozenset(U)))
        return res

    v = best(min(a), (), frozenset(range(n)))
    best.cache_clear()
    return int(v)


def a_random(M: int, a: Sequence[int], s: Sequence[int], o: Sequence[int], perm: Sequence[int]) -> dict:
    """A_r with a fixed permutation (true lengths).  Returns TEL, completions and final starts."""
    n = len(o)
    rank = {j: r for r, j in enumerate(perm)}
    horizon = max(a) + sum(o) + 2
    load = [0] * (horizon + max(o) + 2)  # projected memory per absolute step of started jobs
    start = [None] * n
    done = 0
    t = min(a)
    while done < n:
        waiting = sorted((i for i in range(n) if start[i] is None and a[i] <= t), key=lambda i: rank[i])
        running = any(start[i] is not None and start[i] + o[i] - 1 >= t for i in range(n))
        if not waiting and not running:
            t = min(a[i] for i in range(n) if start[i] is None)
            continue
        for i in waiting:
            prof = [s[i] + k + 1 for k in range(o[i])]
            if all(load[t + k] + prof[k] <= M for k in range(o[i])):
                for k in range(o[i]):
                    load[t + k] += prof[k]
                start[i] = t
            else:
                break
        done = sum(1 for i in range(n) if start[i] is not None and start[i] + o[i] - 1 <= t)
        t += 1
    comp = [start[i] + o[i] for i in range(n)]
    return dict(total_latency=sum(comp[i] - a[i] for i in range(n)), completion=comp, start=start)


def opt_perm(M: int, a, s, o) -> int:
    """min over all permutations of A_r's TEL."""
    n = len(o)
    return min(a_random(M, a, s, o, p)["total_latency"] for p in itertools.permutations(range(n)))


def shortest_first_perm(o: Sequence[int]) -> list:
    return sorted(range(len(o)), key=lambda i: (o[i], i))
