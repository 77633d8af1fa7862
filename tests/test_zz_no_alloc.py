"""sim_run_noalloc (the entry point for callers that cannot allocate device memory) against the
regular sim_load_csr + sim_run path.

Callers such as a serving process whose GPU memory is entirely reserved by its own pool, or a
latency-sensitive loop that must not make synchronising allocation calls, use sim_run_noalloc:
it keeps all of its scratch in a fixed device array inside the library.  This file is collected
last so that a run stopping at the first failure has already run every other test.
"""
import numpy as np
import pytest

from tests.gpu_helpers import FIELDS

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()


def _regular(pol, w):
    from paper_2508_14544_gb300 import Simulator
    with Simulator(pol, w.M, w.n_instances) as sim:
        sim.load_workload(w)
        return sim.run()


def _noalloc(pol, w, dev, out):
    import torch

    from paper_2508_14544_gb300 import _lib as L
    rc = L.sim_run_noalloc(pol, w.M, np.ascontiguousarray(w.offsets, dtype=np.int64), *dev, out)
    assert rc == L.SIM_OK, L.sim_last_error(None)
    torch.cuda.synchronize()
    host = out.cpu().numpy().view(L.RESULT_DTYPE).reshape(-1)
    return host


def test_noalloc_matches_sim_run_two_calls_in_a_row():
    import torch

    from paper_2508_14544_gb300 import workloads as W
    from paper_2508_14544_gb300 import _lib as L
    w = W.make_workload("c2", list(range(0, 1024, 11)))  # 94 instances, all four alphas
    dev = [torch.from_numpy(np.ascontiguousarray(x)).cuda() for x in (w.arrival, w.prompt, w.lower, w.upper, w.true_o)]
    out = torch.zeros(w.n_instances * L.RESULT_DTYPE.itemsize, dtype=torch.uint8, device="cuda")
    for pol in (L.SIM_AMIN, L.SIM_AMAX):  # two calls in a row, sharing the library's fixed scratch
        ref = _regular(pol, w)
        got = _noalloc(pol, w, dev, out)
        for f in FIELDS:
            assert np.array_equal(got[f], ref[f]), (pol, f)
        assert np.all(got["status"] == 0)


def test_noalloc_rejects_oversize_inputs():
    import torch

    from paper_2508_14544_gb300 import _lib as L
    n = 2049  # one instance above the 2048-request limit
    dev = [torch.ones(n, dtype=torch.int32, device="cuda") for _ in range(5)]
    out = torch.zeros(L.RESULT_DTYPE.itemsize, dtype=torch.uint8, device="cuda")
    rc = L.sim_run_noalloc(L.SIM_HSF, 10_000, np.array([0, n], dtype=np.int64), *dev, out)
    assert rc == L.SIM_E_INVAL
    assert "2048" in L.sim_last_error(None)
