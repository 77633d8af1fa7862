"""Every instance of the two largest workloads, every policy, bit-exact against the C oracle
(the oracle runs on all host cores: a few minutes in all).

* alpha sweep: 40960 instances x n=2000 at t=0, M=32768 (the bench workload);
* online: 64 instances x n=10^5 Poisson arrivals, M=500000, queues of up to ~10^5 requests in
  global memory.
Besides the equality, the invariants that the model fixes are checked on every instance."""
import numpy as np
import pytest

from tests.gpu_helpers import assert_same, gpu_run, oracle_run

pytestmark = pytest.mark.gpu

POLS = (0, 1, 2, 3, 4)


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()


@pytest.fixture(scope="module")
def c4():
    from paper_2508_14544_gb300 import workloads as W
    return W.make_workload("c4")


@pytest.fixture(scope="module")
def c5():
    from paper_2508_14544_gb300 import workloads as W
    return W.make_workload("c5")


def _invariants(pol, w, got):
    assert np.all(got["status"] == 0)
    assert np.all(got["peak_memory"] <= w.M)
    so = np.add.reduceat(w.true_o.astype(np.int64), w.offsets[:-1])
    if pol in (0, 2, 3):
        assert np.all(got["evictions"] == 0)
        assert np.array_equal(got["request_steps"], so)
    elif pol == 4:
        # promote-l: every request with o > l is promoted exactly once, wasting l tokens
        longer = w.true_o > w.lower
        assert np.array_equal(got["evictions"], np.add.reduceat(longer.astype(np.int64), w.offsets[:-1]))
        wasted = np.add.reduceat(np.where(longer, w.lower, 0).astype(np.int64), w.offsets[:-1])
        assert np.array_equal(got["request_steps"], so + wasted)
    else:
        assert np.all(got["request_steps"] >= so)


@pytest.mark.parametrize("pol", POLS)
def test_alpha_sweep_all_instances(c4, pol):
    got, _ = gpu_run(pol, c4)
    ref = oracle_run(pol, c4)
    assert_same(got, ref, tag=f"c4 pol={pol}")
    _invariants(pol, c4, got)


@pytest.mark.parametrize("pol", POLS)
def test_online_1e5_all_instances(c5, pol):
    got, _ = gpu_run(pol, c5)
    ref = oracle_run(pol, c5)
    assert_same(got, ref, tag=f"c5 pol={pol}")
    _invariants(pol, c5, got)
