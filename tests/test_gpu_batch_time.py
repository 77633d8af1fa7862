"""Latency in time units under a linear batch-time model (Section 6) on the GPU: the integer sums
equal the CPU oracle's exactly and the two doubles per instance are bit-identical (the same
products and sums in the same order, without fused multiply-adds)."""
import numpy as np
import pytest

from tests.gpu_helpers import n_threads
from tests.test_gpu_parity import _random_mixed_workload, _random_tiny_workload

pytestmark = pytest.mark.gpu

COEFS = [(0.7, 0.013, 1.1e-4, 3.3e-3, 0.25), (1.0, 0.0, 0.0, 0.0, 1.0), (12.5, 0.31, 2.7e-5, 0.017, 3.0)]


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()


def _check(pol, w):
    import torch

    from oracle import plain
    from paper_2508_14544_gb300 import Simulator
    with Simulator(pol, w.M, w.n_instances, batch_time=1) as sim:
        sim.set_tie_seeds(w.tie_seeds())
        rank = torch.from_numpy(w.ranks()).cuda() if pol == 3 else None
        dev = [torch.from_numpy(np.ascontiguousarray(x)).cuda() for x in
               (w.arrival, w.prompt, w.lower, w.upper, w.true_o)]
        sim.load(w.offsets, *dev, rank=rank)
        got = sim.run()
        sums = sim.batch_time_sums()
        times = [sim.batch_time(c) for c in COEFS]
    ref, rsums = plain.run_workload(pol, w, n_threads=n_threads(), time_sums=True)
    assert np.array_equal(got["total_latency"], ref["total_latency"])
    assert np.array_equal(sums, rsums), np.nonzero(np.any(sums != rsums, axis=1))[0][:10]
    ok = ref["status"] == 0
    assert np.array_equal(sums[ok][:, 0], ref["total_latency"][ok])  # X0 = TEL
    for c, t in zip(COEFS, times):
        want = plain.batch_time(ref, rsums, c)
        assert np.array_equal(np.isnan(t), np.isnan(want))
        assert np.array_equal(t[~np.isnan(t)], want[~np.isnan(want)])  # bit-identical


@pytest.mark.parametrize("pol", [0, 1, 2, 3, 4])
def test_tiny_random_with_arrivals(pol):
    _check(pol, _random_tiny_workload(300, n_inst=600, arrivals=True))


@pytest.mark.parametrize("pol", [0, 1, 2, 4])
@pytest.mark.parametrize("M", [700, 6000])
def test_mixed_sizes(pol, M):
    _check(pol, _random_mixed_workload(11, M))


@pytest.mark.parametrize("name", ["c1", "c2", "c3"])
@pytest.mark.parametrize("pol", [0, 1, 2])
def test_named_workloads(name, pol):
    from paper_2508_14544_gb300 import workloads as W
    _check(pol, W.make_workload(name))


@pytest.mark.parametrize("pol", [0, 1, 2])
def test_online_1e5_requests_sampled(pol):
    from paper_2508_14544_gb300 import workloads as W
    _check(pol, W.make_workload("c5", [3, 40]))
