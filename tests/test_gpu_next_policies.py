"""A_r and A_ell through the C ABI: argument checks and properties beyond the oracle parity of
test_gpu_parity.py."""
import numpy as np
import pytest

from tests.gpu_helpers import FIELDS, assert_same, gpu_run, oracle_run

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()


def test_ar_needs_ranks():
    from paper_2508_14544_gb300 import SIM_AR, SimError, Simulator
    from paper_2508_14544_gb300 import workloads as W
    w = W.make_workload("c1")
    with Simulator(SIM_AR, w.M, w.n_instances) as sim:
        with pytest.raises(SimError) as ei:
            sim.load(w.offsets, w.arrival, w.prompt, w.lower, w.upper, w.true_o)
        assert ei.value.code == -1


def test_ar_negative_rank_is_instance_inval():
    from paper_2508_14544_gb300 import workloads as W
    parts = [dict(a=[0, 0], s=[1, 1], l=[1, 1], u=[2, 2], o=[1, 2]) for _ in range(3)]
    w = W.concat_instances("r", 20, parts)
    rank = np.array([0, 1, 1, -1, 1, 0], np.int32)
    got, _ = gpu_run(3, w, rank=rank)
    assert got["status"].tolist() == [0, -1, 0]


def test_ar_rank_ties_by_index_and_shortest_first_equals_hsf():
    """Equal ranks fall back to the request index; ranks sorted by (o, index) reproduce H-SF."""
    from paper_2508_14544_gb300 import workloads as W
    w = W.make_workload("c2", range(0, 1024, 16))
    r_zero, _ = gpu_run(3, w, rank=np.zeros(w.n_total, np.int32))
    r_idx, _ = gpu_run(3, w, rank=np.concatenate([np.arange(w.offsets[i + 1] - w.offsets[i], dtype=np.int32)
                                                  for i in range(w.n_instances)]))
    assert_same(r_zero, r_idx, tag="ties")
    sf = np.zeros(w.n_total, np.int32)
    for i in range(w.n_instances):
        lo, hi = int(w.offsets[i]), int(w.offsets[i + 1])
        order = np.lexsort((np.arange(hi - lo), w.true_o[lo:hi]))
        sf[lo + order] = np.arange(hi - lo, dtype=np.int32)
    r_sf, _ = gpu_run(3, w, rank=sf)
    r_hsf, _ = gpu_run(2, w)
    assert_same(r_sf, r_hsf, tag="shortest-first")


def test_aell_two_point_fluid_ratio():
    """Proof of the A_ell theorem: on a 4000-request two-point instance with M = 4000 the ratio
    TEL(A_ell)/TEL(H-SF) is within 0.02 of 1 + (a^2 x_l x_u + 2 a^2 x_u^2)/(a^2 x_l^2 + 2 a^2 x_l x_u
    + x_u^2); the GPU values equal the oracle's."""
    from paper_2508_14544_gb300 import workloads as W
    rng = np.random.default_rng(1)
    n_l, n_u, l, u = 3000, 1000, 50, 100
    o = np.array([l] * n_l + [u] * n_u)
    rng.shuffle(o)
    n = n_l + n_u
    w = W.concat_instances("d2", 4000, [dict(a=np.zeros(n, int), s=np.ones(n, int), l=np.full(n, l),
                                               u=np.full(n, u), o=o)])
    ga, _ = gpu_run(4, w)
    gh, _ = gpu_run(2, w)
    assert_same(ga, oracle_run(4, w), tag="d2 A_ell")
    al = l / u
    cr = 1 + (al ** 2 * n_l * n_u + 2 * al ** 2 * n_u ** 2) / (al ** 2 * n_l ** 2 + 2 * al ** 2 * n_l * n_u + n_u ** 2)
    assert abs(int(ga["total_latency"][0]) / int(gh["total_latency"][0]) - cr) < 0.02


def test_aell_capacity_fallback_identical():
    """Promotions re-enter the queue through the same delta as A_min's cancellations; a small
    shared-memory capacity forces the global-memory re-run, with identical results."""
    from paper_2508_14544_gb300 import workloads as W
    w = W.make_workload("c2", range(0, 1024, 32))
    a, _ = gpu_run(4, w)
    b, _ = gpu_run(4, w, smem_active_cap=128)
    for f in FIELDS:
        assert np.array_equal(a[f], b[f])


def test_noalloc_rejects_new_policies():
    import ctypes

    from paper_2508_14544_gb300._lib import RESULT_DTYPE, lib
    from paper_2508_14544_gb300 import workloads as W
    w = W.make_workload("c1")
    res = np.zeros(1, RESULT_DTYPE)
    for pol in (3, 4):
        rc = lib().sim_run_noalloc(pol, w.M, 1, w.offsets.ctypes.data, None, None, None, None, None,
                                   res.ctypes.data, None)
        assert rc == -1


@pytest.mark.parametrize("experiment", ["rough", "buckets", "overlap:1/10", "overlap:99/100"])
def test_sweep_instances_match_oracle(experiment):
    """The paper's experiment setups (Section 6) on the dataset stand-in: one seed, loads
    200..2000, every policy, bit-exact against the oracle."""
    from paper_2508_14544_gb300 import workloads as W
    w = W.make_sweep(experiment, seeds=1)
    for pol in (0, 1, 2, 4):
        got, _ = gpu_run(pol, w)
        assert_same(got, oracle_run(pol, w), tag=f"{experiment} pol={pol}")
