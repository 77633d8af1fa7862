"""CUDA path (through the C ABI) vs the CPU oracle: bit-exact on every integer output."""
import numpy as np
import pytest

from tests import pins
from tests.gpu_helpers import FIELDS, assert_same, gpu_run, oracle_run

pytestmark = pytest.mark.gpu

POLS = (0, 1, 2, 3, 4)  # A_max, A_min, H-SF, A_r, A_ell


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()


def _gpu_sim(p, M, a, s, l, u, o, rank=None, tie_seed=0):
    from paper_2508_14544_gb300 import workloads as W
    w = W.concat_instances("pin", M, [dict(a=a, s=s, l=l, u=u, o=o)])
    w.seed0 = int(tie_seed)  # the one instance's tie seed is seed0 + 0
    res, comp = gpu_run(p, w, completions=True, rank=rank)
    out = {k: int(res[0][k]) for k in FIELDS}
    out["completion"] = comp.tolist()
    return out


def test_paper_pins_on_gpu():
    """Example 1, the Definition-1 example, the hand traces (A_min, A_ell, A_r) and the wave closed
    forms (all policies, and A_ell's two-pass waves)."""
    fails = pins.check_all(_gpu_sim)
    assert not fails, fails


def _random_tiny_workload(seed, n_inst=1500, arrivals=True):
    from paper_2508_14544_gb300 import workloads as W
    rng = np.random.default_rng(seed)
    parts = []
    M = 40
    for i in range(n_inst):
        n = int(rng.integers(0, 12))
        o = rng.integers(1, 10, n)
        l = np.array([rng.integers(1, x + 1) for x in o], dtype=np.int64)
        u = o + rng.integers(0, 8, n)
        s = rng.integers(1, 6, n)
        u = np.minimum(u, M - s)
        a = rng.integers(0, 12, n) if arrivals else np.zeros(n, int)
        parts.append(dict(a=a, s=s, l=l, u=u, o=o))
    return W.concat_instances("tiny", M, parts)


@pytest.mark.parametrize("arrivals", [False, True])
@pytest.mark.parametrize("pol", POLS)
def test_random_tiny_batch(pol, arrivals):
    w = _random_tiny_workload(100 + arrivals, arrivals=arrivals)
    got, comp = gpu_run(pol, w, completions=True)
    ref, rcomp = oracle_run(pol, w, completions=True)
    assert_same(got, ref, tag=f"tiny pol={pol}")
    assert np.array_equal(comp, rcomp)


def _random_mixed_workload(seed, M):
    """Instance sizes around the kernel's size thresholds (delta capacity 64 / 128 / 256 at 1024 /
    4096 requests, one-chunk active sets up to 128 jobs, windows of 32), random accuracy, memory
    limits from tight to loose, and arrivals at t=0, spread out, or in bursts."""
    from fractions import Fraction

    from paper_2508_14544_gb300 import workloads as W
    rng = np.random.default_rng(seed)
    parts = []
    sizes = [1, 7, 31, 33, 63, 65, 200, 1000, 1024, 1025, 2100, 4096, 4097]
    for i in range(2 * len(sizes)):
        n = sizes[i % len(sizes)]
        s = rng.integers(1, 17, n)
        o = rng.integers(1, 61, n)
        alpha = [Fraction(1, 10), Fraction(1, 4), Fraction(1, 2), Fraction(1)][i % 4]
        l, u = W.interval_for(o, alpha, rng)
        kind = (i // len(sizes) + i) % 3
        if kind == 0:
            a = np.zeros(n, np.int64)
        elif kind == 1:
            a = np.sort(rng.integers(0, 3 * n + 1, n))
        else:
            a = np.sort(rng.integers(0, 8, n)) * 250
        parts.append(dict(a=a, s=s, l=l, u=u, o=o))
    return W.concat_instances("mixed", M, parts)


def _staging_workload(seed):
    """Instances sized around the staging sort's boundaries (radix passes take 256 elements per
    round, shared memory holds up to 2048 requests, larger ones go to the global-memory sort), with
    arrival steps in random order over a wide range (several arrival-digit passes) and keys drawn
    from a few values (long runs of ties, which the sort must keep in index order)."""
    from fractions import Fraction

    from paper_2508_14544_gb300 import workloads as W
    rng = np.random.default_rng(seed)
    parts = []
    for i, n in enumerate([2, 3, 255, 256, 257, 511, 2047, 2048, 2049]):
        s = rng.integers(1, 9, n)
        o = rng.choice([1, 2, 3, 17, 40], n)
        l, u = W.interval_for(o, [Fraction(1, 3), Fraction(1)][i % 2], rng)
        if i % 3 == 0:
            a = np.zeros(n, np.int64)
        elif i % 3 == 1:
            a = rng.integers(0, 1 << 20, n)  # unsorted, up to 20 bits
        else:
            a = rng.choice([0, 5, 4096, 70000], n)  # few distinct arrival steps
        parts.append(dict(a=a, s=s, l=l, u=u, o=o))
    return W.concat_instances("staging", 400, parts)


@pytest.mark.parametrize("pol", POLS)
def test_staging_sort_boundaries(pol):
    w = _staging_workload(11)
    got, comp = gpu_run(pol, w, completions=True)
    ref, rcomp = oracle_run(pol, w, completions=True)
    assert_same(got, ref, tag=f"staging pol={pol}")
    assert np.array_equal(comp, rcomp)


@pytest.mark.parametrize("M", [700, 6000])
@pytest.mark.parametrize("pol", POLS)
def test_random_mixed_sizes(pol, M):
    w = _random_mixed_workload(7, M)
    got, comp = gpu_run(pol, w, completions=True)
    ref, rcomp = oracle_run(pol, w, completions=True)
    assert_same(got, ref, tag=f"mixed pol={pol}")
    assert np.array_equal(comp, rcomp)


@pytest.mark.parametrize("pol", POLS)
def test_c1(pol):
    from paper_2508_14544_gb300 import workloads as W
    w = W.make_workload("c1")
    got, comp = gpu_run(pol, w, completions=True)
    ref, rcomp = oracle_run(pol, w, completions=True)
    assert_same(got, ref, tag="c1")
    assert np.array_equal(comp, rcomp)


@pytest.fixture(scope="module")
def c2():
    from paper_2508_14544_gb300 import workloads as W
    return W.make_workload("c2")


@pytest.mark.parametrize("pol", POLS)
def test_c2_full(c2, pol):
    """All 1024 instances of the 1000-request workload, in the launch configuration the bench uses."""
    got, _ = gpu_run(pol, c2)
    ref = oracle_run(pol, c2)
    assert_same(got, ref, tag=f"c2 pol={pol}")


def test_c2_competitive_ratio(c2):
    from paper_2508_14544_gb300 import Simulator
    sims = {}
    for pol in POLS:
        s = Simulator(pol, c2.M, c2.n_instances)
        s.load_workload(c2)
        s.run()
        sims[pol] = s
    ref = {pol: oracle_run(pol, c2) for pol in POLS}
    for pol in (0, 1):
        cr = sims[pol].competitive_ratio(sims[2])
        want = ref[pol]["total_latency"].astype(np.float64) / ref[2]["total_latency"].astype(np.float64)
        assert np.array_equal(cr, want)  # same IEEE division of the same integers
        # alpha = 1 (the last 256 instances): exact intervals, every policy coincides with H-SF
        assert np.all(cr[768:] == 1.0)
    for s in sims.values():
        s.close()


@pytest.mark.parametrize("pol", POLS)
def test_c3_full(pol):
    from paper_2508_14544_gb300 import workloads as W
    w = W.make_workload("c3")
    got, _ = gpu_run(pol, w)
    ref = oracle_run(pol, w)
    assert_same(got, ref, tag=f"c3 pol={pol}")
