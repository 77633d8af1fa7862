"""C-ABI behaviour on the GPU: statuses, options, host vs device loads, reruns, edge cases."""
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


def _w(parts, M):
    from paper_2508_14544_gb300 import workloads as W
    return W.concat_instances("edge", M, parts)


def test_empty_and_ragged_instances():
    parts = [dict(a=[], s=[], l=[], u=[], o=[]),
             dict(a=[0], s=[3], l=[2], u=[5], o=[4]),
             dict(a=[], s=[], l=[], u=[], o=[]),
             dict(a=[5, 5, 9], s=[1, 2, 3], l=[1, 1, 1], u=[3, 3, 3], o=[2, 3, 1])]
    w = _w(parts, 12)
    for pol in (0, 1, 2):
        got, comp = gpu_run(pol, w, completions=True)
        ref, rcomp = oracle_run(pol, w, completions=True)
        assert_same(got, ref, tag="edge")
        assert np.array_equal(comp, rcomp)
        assert got["steps"][0] == 0 and got["status"][0] == 0


def test_per_instance_validation_statuses():
    parts = [dict(a=[0], s=[1], l=[2], u=[3], o=[1]),      # l > o   -> INVAL
             dict(a=[0], s=[1], l=[1], u=[1], o=[2]),      # o > u   -> INVAL
             dict(a=[-1], s=[1], l=[1], u=[1], o=[1]),     # a < 0   -> INVAL
             dict(a=[0], s=[0], l=[1], u=[1], o=[1]),      # s < 1   -> INVAL
             dict(a=[0], s=[5], l=[1], u=[9], o=[6]),      # s+o > M -> INFEASIBLE
             dict(a=[0], s=[5], l=[1], u=[9], o=[4]),      # s+u > M: A_max only
             dict(a=[0, 1], s=[1, 1], l=[1, 1], u=[2, 2], o=[1, 2])]
    w = _w(parts, 10)
    for pol in (0, 1, 2):
        got, _ = gpu_run(pol, w)
        ref = oracle_run(pol, w)
        assert_same(got, ref, tag=f"validation pol={pol}")
        assert list(got["status"][:5]) == [-1, -1, -1, -1, -2]
        assert got["status"][5] == (-2 if pol == 0 else 0)


def test_step_cap_matches_oracle():
    from paper_2508_14544_gb300 import workloads as W
    w = W.make_workload("c2", [0, 300, 600, 900])
    for cap in (1, 3, 500):
        for pol in (0, 1, 2):
            got, _ = gpu_run(pol, w, step_cap=cap)
            ref = oracle_run(pol, w, step_cap=cap)
            assert_same(got, ref, tag=f"cap={cap}")
            assert np.all(got["status"] == -3)
            assert np.all(got["steps"] == cap)


def test_capacity_fallback_identical():
    """A 128-slot shared-memory active set forces the larger instances onto the global-memory path."""
    from paper_2508_14544_gb300 import workloads as W
    w = W.make_workload("c2", range(0, 1024, 32))
    for pol in (0, 1, 2):
        a, ca = gpu_run(pol, w, completions=True)
        b, cb = gpu_run(pol, w, completions=True, smem_active_cap=128)
        for f in FIELDS:
            assert np.array_equal(a[f], b[f])
        assert np.array_equal(ca, cb)


def test_host_and_device_loads_and_reruns_agree():
    from paper_2508_14544_gb300 import Simulator
    from paper_2508_14544_gb300 import workloads as W
    w = W.make_workload("c2", range(0, 1024, 64))
    for pol in (0, 1, 2):
        a, _ = gpu_run(pol, w, device_load=True)
        b, _ = gpu_run(pol, w, device_load=False)
        for f in FIELDS:
            assert np.array_equal(a[f], b[f])
        with Simulator(pol, w.M, w.n_instances) as sim:
            sim.load_workload(w)
            r1 = sim.run()
            r2 = sim.run()
        for f in FIELDS:
            assert np.array_equal(r1[f], r2[f]) and np.array_equal(r1[f], a[f])


@pytest.mark.parametrize("wpb,wps", [(1, 0), (2, 0), (8, 0), (4, 4)])
def test_launch_shapes_agree(wpb, wps):
    """Warps per block and resident warps per SM change only the schedule of instances on the
    GPU, never a result."""
    from paper_2508_14544_gb300 import workloads as W
    w = W.make_workload("c2", range(5, 1024, 41))
    for pol in (0, 1, 2):
        a, _ = gpu_run(pol, w)
        b, _ = gpu_run(pol, w, warps_per_block=wpb, warps_per_sm=wps)
        for f in FIELDS:
            assert np.array_equal(a[f], b[f])


def test_residency_tuning():
    """SIM_OPT_TUNE_RESIDENCY: the first run of a load shape simulates with all three residencies
    (at least three simulation launches, plus any global-memory re-runs), later runs and reloads
    of the same shape launch as the chosen one does, a new shape is tuned again, and no result
    changes."""
    from paper_2508_14544_gb300 import POLICIES, Simulator
    from paper_2508_14544_gb300 import workloads as W
    w = W.make_workload("c2", range(3, 1024, 17))
    w2 = W.make_workload("c2", range(0, 1024, 29))
    for pol in ("A_min", "A_max"):
        ref, _ = gpu_run(POLICIES[pol], w)
        ref2, _ = gpu_run(POLICIES[pol], w2)
        with Simulator(POLICIES[pol], w.M, w.n_instances, tune_residency=1) as sim:
            sim.load_workload(w)
            k0 = sim.kernel_launches()
            r1 = sim.run()
            k1 = sim.kernel_launches()
            r2 = sim.run()
            k2 = sim.kernel_launches()
            sim.load_workload(w)
            k3 = sim.kernel_launches()
            r3 = sim.run()
            k4 = sim.kernel_launches()
            assert k1 - k0 >= 3 and k2 - k1 == k4 - k3 and 1 <= k2 - k1 <= 2
            for r in (r1, r2, r3):
                for f in FIELDS:
                    assert np.array_equal(r[f], ref[f])
        with Simulator(POLICIES[pol], w2.M, w2.n_instances, tune_residency=1) as sim:
            sim.load_workload(w2)
            k0 = sim.kernel_launches()
            r = sim.run()
            assert sim.kernel_launches() - k0 >= 3
            for f in FIELDS:
                assert np.array_equal(r[f], ref2[f])


@pytest.mark.parametrize("pol", [0, 1, 2, 3, 4])
def test_dense_residency(pol):
    """SIM_OPT_DENSE_RESIDENCY (12 warps per SM, 384 shared-memory slots) gives the oracle's results;
    an instance of 1000 one-token-prompt jobs holds more than 384 of them at once and is re-run in
    global memory (two launches)."""
    from paper_2508_14544_gb300 import workloads as W
    w = W.make_workload("c4", range(5, 40960, 40))
    rng = np.random.default_rng(44)
    n = 1000
    o = rng.integers(1, 6, n)
    big = dict(a=np.zeros(n, np.int64), s=np.ones(n, np.int64), l=np.ones(n, np.int64), u=o + 2, o=o)
    parts = [w.instance(i) for i in range(w.n_instances)] + [big]
    wb = W.concat_instances("dense", w.M, parts, None, None)
    wb.seed0 = 77
    ref = oracle_run(pol, wb)
    from paper_2508_14544_gb300 import Simulator
    with Simulator(pol, wb.M, wb.n_instances, dense_residency=1) as sim:
        sim.set_tie_seeds(wb.tie_seeds())
        if pol == 3:
            sim.load(wb.offsets, wb.arrival, wb.prompt, wb.lower, wb.upper, wb.true_o, rank=wb.ranks())
        else:
            sim.load(wb.offsets, wb.arrival, wb.prompt, wb.lower, wb.upper, wb.true_o)
        k0 = sim.kernel_launches()
        got = sim.run()
        assert sim.kernel_launches() - k0 == 2
    for f in FIELDS:
        assert np.array_equal(got[f], ref[f]), (pol, f)


def test_more_instances_than_warps():
    """One resident warp per SM (152 warps) for 342 instances: every warp simulates several
    instances in turn, reusing its workspace, and the results do not change."""
    from paper_2508_14544_gb300 import workloads as W
    w = W.make_workload("c2", range(0, 1024, 3))
    for pol in (0, 1, 2):
        a, _ = gpu_run(pol, w)
        b, _ = gpu_run(pol, w, warps_per_block=1, warps_per_sm=1)
        for f in FIELDS:
            assert np.array_equal(a[f], b[f])


def test_sparse_arrivals_and_bursts():
    """Idle gaps (time jumps), one large burst (bulk insert through the delta queue), and many
    evictions for A_min, at sizes that exercise delta merges."""
    from fractions import Fraction

    from paper_2508_14544_gb300 import workloads as W
    rng = np.random.default_rng(3)
    parts = []
    for i in range(24):
        n = 1500
        s = rng.integers(1, 40, n)
        o = rng.integers(1, 200, n)
        l, u = W.interval_for(o, Fraction(1, 4), rng)
        a = np.sort(rng.integers(0, 4000, n))
        if i % 3 == 0:
            a[300:900] = a[300]  # a burst of 600 arrivals in one step
        if i % 3 == 1:
            a = a * 7  # long idle gaps
        parts.append(dict(a=a, s=s, l=l, u=u, o=o))
    w = W.concat_instances("arrivals", 3000, parts)
    for pol in (0, 1, 2):
        got, comp = gpu_run(pol, w, completions=True)
        ref, rcomp = oracle_run(pol, w, completions=True)
        assert_same(got, ref, tag=f"arrivals pol={pol}")
        assert np.array_equal(comp, rcomp)


def test_unsorted_arrivals():
    """Arrival steps not in index order: staging sorts by (arrival, key, index)."""
    from fractions import Fraction

    from paper_2508_14544_gb300 import workloads as W
    rng = np.random.default_rng(4)
    parts = []
    for i in range(40):
        n = int(rng.integers(1, 300))
        s = rng.integers(1, 20, n)
        o = rng.integers(1, 60, n)
        l, u = W.interval_for(o, Fraction(1, 2), rng)
        a = rng.integers(0, 200, n)
        parts.append(dict(a=a, s=s, l=l, u=u, o=o))
    w = W.concat_instances("unsorted", 600, parts)
    for pol in (0, 1, 2):
        got, comp = gpu_run(pol, w, completions=True)
        ref, rcomp = oracle_run(pol, w, completions=True)
        assert_same(got, ref, tag="unsorted")
        assert np.array_equal(comp, rcomp)


def test_long_requests_narrow_and_wide_kernels_agree():
    """Lengths of ~3e5 steps: with the default 512-slot shared-memory capacity the 32-bit kernel is
    valid (512 x (2 lmax + 2) + 2^27 < 2^31); with a 4096-slot capacity it is not, so every
    instance is re-run by the 64-bit global-memory kernel.  Both equal the oracle."""
    from paper_2508_14544_gb300 import workloads as W
    rng = np.random.default_rng(21)
    parts = []
    M = 1_000_000
    for _ in range(6):
        n = 12
        o = rng.integers(1000, 300_000, n)
        l = np.maximum(o // 3, 1)
        u = np.minimum(o * 2, M - 100)
        s = rng.integers(1, 50, n)
        a = rng.integers(0, 200_000, n)
        parts.append(dict(a=a, s=s, l=l, u=u, o=o))
    w = W.concat_instances("long", M, parts)
    for pol in (0, 1, 2, 4):
        ref = oracle_run(pol, w)
        narrow, _ = gpu_run(pol, w)
        wide, _ = gpu_run(pol, w, smem_active_cap=4096)
        for f in FIELDS:
            assert np.array_equal(narrow[f], ref[f]), (pol, f)
            assert np.array_equal(wide[f], ref[f]), (pol, f)


def test_cancellation_order_with_long_bounds():
    """A_min's cancellation order (estimate, random tie key, index) with upper bounds of 1.2e6 on a
    4096-request instance, next to a 1000-request instance with short lengths: both kernels (the
    shared-memory one and the checking global-memory one) equal the oracle."""
    from paper_2508_14544_gb300 import workloads as W
    rng = np.random.default_rng(33)
    parts = []
    for n, big in ((4096, True), (1000, False)):
        o = rng.integers(1, 40, n)
        l = np.maximum(o // 4, 1)
        u = o * 4
        if big:
            u[rng.choice(n, 3, replace=False)] = 1_200_000
        s = rng.integers(1, 8, n)
        parts.append(dict(a=np.zeros(n, np.int64), s=s, l=l, u=u, o=o))
    w = W.concat_instances("unpacked", 600, parts)
    for pol in (1, 2):
        ref = oracle_run(pol, w)
        narrow, _ = gpu_run(pol, w)
        wide, _ = gpu_run(pol, w, debug_checks=1)
        for f in FIELDS:
            assert np.array_equal(narrow[f], ref[f]), (pol, f)
            assert np.array_equal(wide[f], ref[f]), (pol, f)
        if pol == 1:
            assert ref["evictions"][0] > 100 and ref["evictions"][1] > 100


def test_command_lines(capsys):
    """`python -m paper_2508_14544_gb300.run` and `.sweep` through the C ABI."""
    import json

    from paper_2508_14544_gb300 import run, sweep
    run.main(["--workload", "c1", "--policy", "A_ell", "--repeat", "2"])
    lines = [json.loads(l) for l in capsys.readouterr().out.splitlines() if l.startswith("{")]
    assert len(lines) == 2 and lines[0]["worst_status"] == 0 and lines[0]["request_steps"] == lines[1]["request_steps"]
    run.main(["--workload", "c1", "--policy", "A_r"])
    assert json.loads(capsys.readouterr().out.splitlines()[0])["worst_status"] == 0
    sweep.main(["--experiments", "buckets", "--policies", "A_min,H-SF", "--seeds", "1"])
    out = [json.loads(l) for l in capsys.readouterr().out.splitlines() if l.startswith("{")]
    assert [o["policy"] for o in out] == ["A_min", "H-SF"]
    assert all(len(o["avg_latency"]) == 10 for o in out)


@pytest.mark.parametrize("pol", [0, 1, 2, 3, 4])
def test_debug_checks_hold_and_change_nothing(pol):
    """SIM_OPT_DEBUG_CHECKS: the invariants hold at every event of the 1000-request instances
    (all alphas) and of an online workload with bursts, and the results are unchanged."""
    from paper_2508_14544_gb300 import workloads as W
    for w in (W.make_workload("c2", range(3, 1024, 64)), W.make_workload("c3", [5, 9])):
        a, _ = gpu_run(pol, w)
        b, _ = gpu_run(pol, w, debug_checks=1)
        assert np.all(b["status"] == 0)
        for f in FIELDS:
            assert np.array_equal(a[f], b[f]), (pol, f)


def test_largest_memory_limit():
    """M = 2^26 (the largest the ABI accepts) with requests of up to ~2^25 tokens: the 32-bit
    bound fails, so the 64-bit kernel runs every instance; results equal the oracle (which steps
    every one of the ~10^8 batches)."""
    from paper_2508_14544_gb300 import workloads as W
    M = 1 << 26
    parts = [dict(a=[0, 0, 5, 9], s=[1000, 7, 1, 1 << 20], l=[1, 5, 1 << 24, 3],
                  u=[1 << 25, 9, 1 << 25, (1 << 25) - (1 << 20)], o=[1 << 24, 9, (1 << 24) + 3, 1 << 22]),
             dict(a=[0], s=[(1 << 26) - 2], l=[1], u=[2], o=[2])]
    w = W.concat_instances("maxm", M, parts)
    for pol in (0, 1, 2, 4):
        got, _ = gpu_run(pol, w)
        ref = oracle_run(pol, w)
        for f in FIELDS:
            assert np.array_equal(got[f], ref[f]), (pol, f)


def test_step_counter_limit_is_a_step_cap():
    """Steps are 32-bit: an instance whose steps would pass 2^31 - 2^27 (2^30 under A_ell) stops
    with SIM_E_STEPCAP instead of wrapping; instances far from the limit are unaffected."""
    from paper_2508_14544_gb300 import workloads as W
    near = (1 << 31) - (1 << 27) - 50
    parts = [dict(a=[near, near], s=[1, 1], l=[10, 10], u=[100, 100], o=[100, 90]),
             dict(a=[0, 3], s=[1, 2], l=[1, 1], u=[5, 5], o=[4, 5])]
    w = W.concat_instances("late", 1000, parts)
    ref = oracle_run(0, w)
    for pol in (0, 1, 2):
        got, _ = gpu_run(pol, w)
        assert got["status"].tolist() == [-3, 0], pol
        r = oracle_run(pol, w)
        for f in FIELDS:
            assert got[f][1] == r[f][1]
    late = W.concat_instances("late_ell", 1000, [dict(a=[(1 << 30) - 5], s=[1], l=[10], u=[100], o=[100])])
    got, _ = gpu_run(4, late)
    assert got["status"].tolist() == [-3]
    del ref
