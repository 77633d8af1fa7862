"""Seeded synthetic request workloads for the batched scheduler simulator.

This module only draws input arrays (arrival step, prompt size, predicted interval, true output
length).  It holds none of the scheduling arithmetic, so both the CPU oracle (``oracle/``) and the
CUDA path consume exactly the same arrays.

The paper evaluates on 2,000 sampled LMSYS-Chat-1M conversations (Section 6, "Dataset Overview").
That dataset is not available here; the five synthetic workloads below stand in for it.  Their
shapes follow the problem model of Section 2: every request has a prompt size s_i, a hidden output
length o_i and a predicted interval [l_i, u_i] containing o_i (Section 2, "Prediction Interval for
Output Length"; per-request intervals as in Section 4.2 and Experiments 2-3 of Section 6).

Interval rule (all workloads): alpha = a/b is a rational, l_i ~ U{ceil(alpha*o_i) .. o_i} and
u_i = ceil(l_i / alpha).  Both ceilings are computed in integers,
ceil(a*o/b) = (a*o + b - 1) // b and ceil(l*b/a) = (l*b + a - 1) // a, so l_i <= o_i <= u_i holds
exactly (no float rounding).

Per-instance seeding: instance i of a workload draws from ``numpy.random.default_rng(seed0 + i)``
in the fixed order s, o, l, arrivals, so any subset of instances is reproducible on its own.

The auxiliary policy A_r (Algorithm random) also needs a uniformly random permutation of each
instance's requests; ``Workload.ranks()`` draws it from a separate stream,
``numpy.random.default_rng([seed0 + i, 1])``, and returns rank[j] = position of request j.

A_min breaks eviction ties uniformly at random (Algorithm milb).  The simulator and the oracle
draw those ties themselves from a counter-based generator; the generator only supplies its seed,
one uint64 per instance: ``Workload.tie_seeds()`` = seed0 + i.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from fractions import Fraction
from typing import Callable, Sequence

import numpy as np

__all__ = [
    "Workload",
    "lookalike_pool",
    "intervals_rough",
    "intervals_buckets",
    "intervals_overlap",
    "make_sweep",
    "WORKLOADS",
    "make_workload",
    "make_instance",
    "rank_instances",
    "interval_for",
    "concat_instances",
]


@dataclass
class Workload:
    """A batch of independent scheduling instances in CSR layout (int32 SoA arrays)."""

    name: str
    M: int
    offsets: np.ndarray  # int64 [n_instances + 1]
    arrival: np.ndarray  # int32 [n_total]  a_i (step at which request i becomes eligible)
    prompt: np.ndarray  # int32 [n_total]  s_i
    lower: np.ndarray  # int32 [n_total]  l_i
    upper: np.ndarray  # int32 [n_total]  u_i
    true_o: np.ndarray  # int32 [n_total]  o_i
    alpha: list = field(default_factory=list)  # per-instance Fraction
    instance_ids: np.ndarray | None = None  # global instance id of each row
    seed0: int | None = None  # seed base of the named workload (for ranks())
    _ranks: np.ndarray | None = None

    @property
    def n_instances(self) -> int:
        return int(self.offsets.shape[0] - 1)

    @property
    def n_total(self) -> int:
        return int(self.offsets[-1])

    def instance(self, i: int) -> dict:
        lo, hi = int(self.offsets[i]), int(self.offsets[i + 1])
        return dict(
            M=self.M,
            a=self.arrival[lo:hi],
            s=self.prompt[lo:hi],
            l=self.lower[lo:hi],
            u=self.upper[lo:hi],
            o=self.true_o[lo:hi],
        )

    def ranks(self) -> np.ndarray:
        """A_r's random permutation of every instance, as int32 ranks in CSR layout: rank[j] is the
        position of request j in its instance's permutation.  Drawn per instance from
        default_rng([seed0 + id, 1]) (instance id = global id when known, else the row)."""
        if self._ranks is None:
            out = np.zeros(self.n_total, dtype=np.int32)
            base = 0 if self.seed0 is None else self.seed0
            for r in range(self.n_instances):
                lo, hi = int(self.offsets[r]), int(self.offsets[r + 1])
                iid = r if self.instance_ids is None else int(self.instance_ids[r])
                perm = np.random.default_rng([base + iid, 1]).permutation(hi - lo)
                rk = np.empty(hi - lo, dtype=np.int32)
                rk[perm] = np.arange(hi - lo, dtype=np.int32)
                out[lo:hi] = rk
            self._ranks = out
        return self._ranks

    def tie_seeds(self) -> np.ndarray:
        """Seed of A_min's random eviction ties for every instance (uint64): seed0 + id (instance
        id = global id when known, else the row)."""
        base = 0 if self.seed0 is None else int(self.seed0)
        ids = np.arange(self.n_instances, dtype=np.int64) if self.instance_ids is None else \
            np.asarray(self.instance_ids, dtype=np.int64)
        return (ids + base).astype(np.uint64)

    def uniform_n(self) -> int | None:
        d = np.diff(self.offsets)
        return int(d[0]) if d.size and np.all(d == d[0]) else None

    def subset(self, rows: Sequence[int]) -> "Workload":
        parts = [self.instance(int(i)) for i in rows]
        ids = None if self.instance_ids is None else self.instance_ids[np.asarray(rows, dtype=np.int64)]
        w = concat_instances(self.name, self.M, parts, [self.alpha[int(i)] for i in rows], ids)
        w.seed0 = self.seed0
        return w


def interval_for(o: np.ndarray, alpha: Fraction, rng: np.random.Generator) -> tuple[np.ndarray, np.ndarray]:
    """Draw l ~ U{ceil(alpha*o)..o} and set u = ceil(l/alpha), in exact integer arithmetic."""
    a, b = alpha.numerator, alpha.denominator
    o64 = o.astype(np.int64)
    lo = (a * o64 + b - 1) // b
    lo = np.maximum(lo, 1)
    l = rng.integers(lo, o64 + 1)  # inclusive upper bound via +1
    u = (l * b + a - 1) // a
    return l.astype(np.int32), u.astype(np.int32)


def _poisson_arrivals(n: int, rate: float, rng: np.random.Generator) -> np.ndarray:
    gaps = rng.exponential(scale=1.0 / rate, size=n)
    return np.floor(np.cumsum(gaps)).astype(np.int64).astype(np.int32)


# --- per-workload instance recipes -------------------------------------------------------------


def _c1(i: int, rng: np.random.Generator):
    n = 50
    s = rng.integers(1, 21, size=n)
    o = rng.integers(1, 101, size=n)
    alpha = Fraction(1, 2)
    l, u = interval_for(o, alpha, rng)
    return np.zeros(n, np.int32), s, o, l, u, alpha


_C2_ALPHAS = (Fraction(1, 5), Fraction(1, 2), Fraction(4, 5), Fraction(1, 1))


def _c2(i: int, rng: np.random.Generator):
    n = 1000
    s = rng.integers(1, 65, size=n)
    o = rng.integers(1, 513, size=n)
    alpha = _C2_ALPHAS[(i // 256) % 4]
    l, u = interval_for(o, alpha, rng)
    return np.zeros(n, np.int32), s, o, l, u, alpha


def _c3(i: int, rng: np.random.Generator):
    n = 10_000
    s = np.clip(np.rint(rng.lognormal(mean=5.0, sigma=0.8, size=n)), 1, 4096).astype(np.int64)
    o = np.clip(rng.geometric(p=1.0 / 300.0, size=n), 1, 4096).astype(np.int64)
    alpha = Fraction(3, 5)
    l, u = interval_for(o, alpha, rng)
    a = _poisson_arrivals(n, 0.5, rng)
    return a, s, o, l, u, alpha


def _c4(i: int, rng: np.random.Generator):
    n = 2000
    s = rng.integers(16, 257, size=n)
    short = rng.random(size=n) < 0.7
    o = np.where(short, rng.integers(1, 33, size=n), rng.integers(512, 2049, size=n))
    alpha = Fraction((i // 4096) % 10 + 1, 10)
    l, u = interval_for(o, alpha, rng)
    return np.zeros(n, np.int32), s, o, l, u, alpha


def _c5(i: int, rng: np.random.Generator):
    n = 100_000
    s = rng.integers(1, 2049, size=n)
    o = np.clip(rng.zipf(1.2, size=n), 1, 8192).astype(np.int64)
    alpha = Fraction(3, 10)
    l, u = interval_for(o, alpha, rng)
    a = _poisson_arrivals(n, 2.0, rng)
    return a, s, o, l, u, alpha


@dataclass(frozen=True)
class _Spec:
    name: str
    M: int
    n_instances: int
    seed0: int
    recipe: Callable
    description: str


WORKLOADS: dict[str, _Spec] = {
    "c1": _Spec("c1", 2000, 1, 0, _c1,
                "1 instance, n=50 at t=0, M=2000, s~U{1..20}, o~U{1..100}, alpha=1/2, seed 0"),
    "c2": _Spec("c2", 16384, 1024, 1_000_000, _c2,
                "1024 instances x n=1000 at t=0, M=16384, s~U{1..64}, o~U{1..512}, "
                "alpha in {1/5,1/2,4/5,1} (256 seeds each)"),
    "c3": _Spec("c3", 65536, 256, 2_000_000, _c3,
                "256 instances x n=10^4, Poisson arrivals rate 0.5/step, M=65536, "
                "s=round(lognormal(5,0.8)) in [1,4096], o~Geom(1/300) in [1,4096], alpha=3/5"),
    "c4": _Spec("c4", 32768, 40960, 3_000_000, _c4,
                "alpha in {0.1..1.0} x 4096 seeds, n=2000 at t=0, M=32768, s~U{16..256}, "
                "o: 70% U{1..32}, 30% U{512..2048}"),
    "c5": _Spec("c5", 500_000, 64, 4_000_000, _c5,
                "64 instances x n=10^5, Poisson arrivals rate 2/step, M=500000, s~U{1..2048}, "
                "o~Zipf(1.2) in [1,8192], alpha=3/10"),
}


def rank_instances(name: str, rank: int) -> range:
    """Instance ids simulated by one rank when every GPU runs its own copy of a workload's shape
    (weak scaling): rank r takes ids [r*N, (r+1)*N) of the workload's seed sequence."""
    n = WORKLOADS[name].n_instances
    return range(rank * n, (rank + 1) * n)


def make_instance(name: str, i: int) -> dict:
    """One instance of a named workload as a dict of int32 arrays plus M and alpha."""
    spec = WORKLOADS[name]
    rng = np.random.default_rng(spec.seed0 + i)
    a, s, o, l, u, alpha = spec.recipe(i, rng)
    return dict(
        M=spec.M,
        a=np.asarray(a, np.int32),
        s=np.asarray(s, np.int32),
        o=np.asarray(o, np.int32),
        l=np.asarray(l, np.int32),
        u=np.asarray(u, np.int32),
        alpha=alpha,
    )


def concat_instances(name: str, M: int, parts: list[dict], alphas: list | None = None,
                     ids: np.ndarray | None = None) -> Workload:
    sizes = np.array([len(p["o"]) for p in parts], dtype=np.int64)
    offsets = np.zeros(len(parts) + 1, dtype=np.int64)
    np.cumsum(sizes, out=offsets[1:])

    def cat(k):
        if not parts:
            return np.zeros(0, np.int32)
        return np.ascontiguousarray(np.concatenate([np.asarray(p[k], np.int32) for p in parts]))

    return Workload(
        name=name,
        M=int(M),
        offsets=offsets,
        arrival=cat("a"),
        prompt=cat("s"),
        lower=cat("l"),
        upper=cat("u"),
        true_o=cat("o"),
        alpha=list(alphas) if alphas is not None else [p.get("alpha") for p in parts],
        instance_ids=ids,
    )


def make_workload(name: str, instances: Sequence[int] | range | None = None) -> Workload:
    """Generate a named workload (all instances, or the listed instance ids)."""
    spec = WORKLOADS[name]
    ids = range(spec.n_instances) if instances is None else instances
    ids = np.asarray(list(ids), dtype=np.int64)
    parts = [make_instance(name, int(i)) for i in ids]
    w = concat_instances(name, spec.M, parts, [p["alpha"] for p in parts], ids)
    w.seed0 = spec.seed0
    return w


# --- the paper's experiment setups (Section 6) on a synthetic stand-in for its dataset ---------
#
# The paper samples 2,000 LMSYS-Chat-1M conversations and prints only summary statistics of them
# (Section 6, "Dataset Overview"): prompt sizes 1..468 (mean 41, median 11, variance 4961), output
# lengths 1..883 (mean 85, median 43, variance 9702).  The dataset is not available here and none
# of its items is reproduced: the pool below draws from lognormal distributions truncated to those
# ranges (rounded to integers, out-of-range draws rejected), with (mu, sigma) fitted to the printed
# mean, median and variance.  Fitted: prompts mu 2.3505, sigma 2.0308 (mean 39.8, median 11,
# variance 5033); outputs mu 3.8006, sigma 1.1094 (mean 78.3, median 44, variance 9903).

_LOOKALIKE_S = (2.3505, 2.0308, 1, 468)
_LOOKALIKE_O = (3.8006, 1.1094, 1, 883)
SWEEP_SEED0 = 5_000_000


def _trunc_lognormal(rng: np.random.Generator, n: int, mu: float, sigma: float, lo: int, hi: int) -> np.ndarray:
    out = np.empty(0, dtype=np.int64)
    while out.size < n:
        v = np.rint(np.exp(rng.normal(mu, sigma, size=2 * (n - out.size) + 16))).astype(np.int64)
        out = np.concatenate([out, v[(v >= lo) & (v <= hi)]])
    return out[:n]


def lookalike_pool(seed: int, n: int = 2000) -> tuple[np.ndarray, np.ndarray]:
    """(s, o) of a pool of n synthetic requests shaped like the paper's sample."""
    rng = np.random.default_rng([SWEEP_SEED0, seed])
    s = _trunc_lognormal(rng, n, *_LOOKALIKE_S)
    o = _trunc_lognormal(rng, n, *_LOOKALIKE_O)
    return s, o


def intervals_rough(o: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """Experiment 1 (rough prediction): [1, 1000] for every request."""
    return np.ones_like(o), np.full_like(o, 1000)


def intervals_buckets(o: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """Experiment 2 (non-overlapping classification): the bucket [100b + 1, 100b + 100] holding o."""
    l = 100 * ((o - 1) // 100) + 1
    return l, l + 99


def intervals_overlap(o: np.ndarray, x: Fraction) -> tuple[np.ndarray, np.ndarray]:
    """Experiment 3 (overlapping intervals): [(1 - x) o, (1 + x) o] with the ends rounded outwards
    (floor, ceil) in exact integer arithmetic and l >= 1, so l <= o <= u."""
    a, b = x.numerator, x.denominator
    o64 = o.astype(np.int64)
    l = np.maximum(((b - a) * o64) // b, 1)
    u = -((-(b + a) * o64) // b)
    return l, u


def make_sweep(experiment: str, loads: Sequence[int] = tuple(range(200, 2001, 200)), seeds: int = 4,
               M: int = 10000) -> Workload:
    """Instances of the paper's load sweep (Section 6, "Experiment Setup"): for each seed a pool
    of 2000 requests, and for each load n a random subset of n of them, all arriving at t = 0, with
    the intervals of ``experiment``: "rough", "buckets" or "overlap:a/b" (x = a/b).  Instance
    order: seed-major, then load.  ``instance_ids`` holds (seed, n) pairs encoded as
    seed * 100000 + n."""
    if experiment == "rough":
        fn = intervals_rough
    elif experiment == "buckets":
        fn = intervals_buckets
    elif experiment.startswith("overlap:"):
        x = Fraction(experiment.split(":", 1)[1])
        if not 0 < x < 1:
            raise ValueError("overlap x must lie in (0, 1)")
        fn = lambda o: intervals_overlap(o, x)  # noqa: E731
    else:
        raise ValueError(f"unknown experiment {experiment!r}")
    parts, ids = [], []
    for seed in range(seeds):
        s_pool, o_pool = lookalike_pool(seed)
        rng = np.random.default_rng([SWEEP_SEED0, seed, 1])
        for n in loads:
            pick = rng.choice(s_pool.size, size=int(n), replace=False)
            s, o = s_pool[pick], o_pool[pick]
            l, u = fn(o)
            parts.append(dict(a=np.zeros(int(n), np.int32), s=s, o=o, l=l, u=u))
            ids.append(seed * 100000 + int(n))
    return concat_instances(f"sweep-{experiment}", M, parts, None, np.asarray(ids, np.int64))
