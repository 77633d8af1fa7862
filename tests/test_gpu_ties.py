"""A_min's random cancellation ties on the GPU (Algorithm milb / milbrevise: "break ties uniformly
at random"): bit-exact with the CPU oracle on instances full of ties, under both tie rules."""
import numpy as np
import pytest

from tests.gpu_helpers import assert_same, gpu_run, oracle_run
from tests.test_amin_ties import TWO_POINT, two_point

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()


@pytest.mark.parametrize("n,M,l,u", TWO_POINT)
@pytest.mark.parametrize("ties", ["hash", "index"])
def test_two_point_instances(n, M, l, u, ties):
    """The instances of the Theorem thm:no pin: every cancellation step is a tie."""
    w = two_point(n, M, l, u, 0.5, range(8))
    got, comp = gpu_run(1, w, completions=True, evict_ties=int(ties == "index"))
    ref, rcomp = oracle_run(1, w, completions=True, evict_ties=ties)
    assert_same(got, ref, tag=f"two-point {ties}")
    assert np.array_equal(comp, rcomp)
    assert np.all(got["evictions"] > 0)


def test_one_chunk_and_wide_active_sets():
    """Small s and short lengths make active sets above one chunk (128 entries) as well as below;
    ties everywhere (all lower bounds equal)."""
    from paper_2508_14544_gb300 import workloads as W
    parts = []
    for k, (n, M) in enumerate([(300, 200), (1500, 1200), (3000, 2500), (600, 900)]):
        rng = np.random.default_rng([31, k])
        o = rng.integers(1, 12, n)
        parts.append(dict(a=np.zeros(n, int), s=np.ones(n, int), l=np.ones(n, int), u=o + 3, o=o))
    for M in (200, 900, 2500):
        w = W.concat_instances("wide", M, parts[:3] if M >= 2500 else parts[:1])
        w.seed0 = 4242
        got, comp = gpu_run(1, w, completions=True)
        ref, rcomp = oracle_run(1, w, completions=True)
        assert_same(got, ref, tag=f"wide M={M}")
        assert np.array_equal(comp, rcomp)


def test_seeds_change_results_and_reset():
    """Different seeds give different (oracle-equal) schedules; sim_set_tie_seeds(None) goes back
    to seed 0 for every instance."""
    from oracle import plain
    from paper_2508_14544_gb300 import Simulator
    w = two_point(2000, 2000, 5, 10, 0.5, range(4))
    with Simulator(1, w.M, w.n_instances) as sim:
        sim.load(w.offsets, w.arrival, w.prompt, w.lower, w.upper, w.true_o)
        outs = []
        for seeds in (np.arange(4, dtype=np.uint64), np.arange(4, dtype=np.uint64) + 1000, None):
            sim.set_tie_seeds(seeds)
            got = sim.run()
            ts = np.zeros(4, np.uint64) if seeds is None else seeds
            ref = plain.run_batch(1, w.M, w.offsets, w.arrival, w.prompt, w.lower, w.upper, w.true_o,
                                  tie_seeds=ts, n_threads=4)
            assert_same(got, ref, tag=f"seeds {None if seeds is None else seeds.tolist()}")
            outs.append(got["total_latency"].copy())
        assert not np.array_equal(outs[0], outs[1])
