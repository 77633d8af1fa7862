"""sim_run_noalloc (the entry point for callers that cannot allocate device memory) against the
regular sim_load_csr + sim_run path and the CPU oracle.

Callers such as a serving process whose GPU memory is entirely reserved by its own pool, or a
latency-sensitive loop that must not make synchronising allocation calls, use sim_run_noalloc:
it keeps all of its scratch in a fixed device array inside the library.  This file is collected
last so that a run stopping at the first failure has already run every other test.
"""
import numpy as np
import pytest

from tests.gpu_helpers import FIELDS, n_threads

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()


def _regular(pol, w):
    """sim_load_csr + sim_run with default options (tie seed 0 for every instance, as the
    allocation-free entry point uses)."""
    from paper_2508_14544_gb300 import Simulator
    with Simulator(pol, w.M, w.n_instances) as sim:
        sim.load(w.offsets, w.arrival, w.prompt, w.lower, w.upper, w.true_o)
        return sim.run()


def _oracle(pol, w):
    from oracle import plain
    return plain.run_batch(pol, w.M, w.offsets, w.arrival, w.prompt, w.lower, w.upper, w.true_o,
                           n_threads=n_threads(), tie_seeds=np.zeros(w.n_instances, np.uint64))


def _dev(w):
    import torch
    return [torch.from_numpy(np.ascontiguousarray(x)).cuda() for x in (w.arrival, w.prompt, w.lower, w.upper, w.true_o)]


def _noalloc(pol, w, dev, out):
    import torch

    from paper_2508_14544_gb300 import _lib as L
    rc = L.sim_run_noalloc(pol, w.M, np.ascontiguousarray(w.offsets, dtype=np.int64), *dev, out)
    assert rc == L.SIM_OK, L.sim_last_error(None)
    torch.cuda.synchronize()
    return out.cpu().numpy().view(L.RESULT_DTYPE).reshape(-1)[: w.n_instances].copy()


def _check(got, ref, tag):
    for f in FIELDS:
        assert np.array_equal(got[f], ref[f]), (tag, f)


def test_noalloc_matches_sim_run_and_oracle_calls_in_a_row():
    import torch

    from paper_2508_14544_gb300 import workloads as W
    from paper_2508_14544_gb300 import _lib as L
    w = W.make_workload("c2", list(range(0, 1024, 11)))  # 94 instances, all four alphas
    dev = _dev(w)
    out = torch.zeros(w.n_instances * L.RESULT_DTYPE.itemsize, dtype=torch.uint8, device="cuda")
    for pol in (L.SIM_AMIN, L.SIM_AMAX, L.SIM_HSF, L.SIM_AMIN):  # calls in a row share the fixed scratch
        got = _noalloc(pol, w, dev, out)
        _check(got, _regular(pol, w), f"sim_run pol={pol}")
        _check(got, _oracle(pol, w), f"oracle pol={pol}")
        assert np.all(got["status"] == 0)


def test_noalloc_empty_instances():
    import torch

    from paper_2508_14544_gb300 import workloads as W
    from paper_2508_14544_gb300 import _lib as L
    rng = np.random.default_rng(3)
    parts = []
    for i in range(40):
        n = 0 if i % 3 == 0 else int(rng.integers(1, 300))
        o = rng.integers(1, 60, n)
        l = np.array([rng.integers(1, x + 1) for x in o], dtype=np.int64)
        parts.append(dict(a=np.sort(rng.integers(0, 50, n)), s=rng.integers(1, 20, n), l=l, u=o + 5, o=o))
    w = W.concat_instances("with-empty", 900, parts)
    dev = _dev(w)
    out = torch.zeros(w.n_instances * L.RESULT_DTYPE.itemsize, dtype=torch.uint8, device="cuda")
    for pol in (L.SIM_AMIN, L.SIM_AMAX, L.SIM_HSF):
        got = _noalloc(pol, w, dev, out)
        _check(got, _regular(pol, w), f"sim_run pol={pol}")
        _check(got, _oracle(pol, w), f"oracle pol={pol}")
        assert np.all(got["total_latency"][::3] == 0)


def test_noalloc_rejects_oversize_inputs():
    import torch

    from paper_2508_14544_gb300 import _lib as L
    n = 2049  # one instance above the 2048-request limit
    dev = [torch.ones(n, dtype=torch.int32, device="cuda") for _ in range(5)]
    out = torch.zeros(L.RESULT_DTYPE.itemsize, dtype=torch.uint8, device="cuda")
    rc = L.sim_run_noalloc(L.SIM_HSF, 10_000, np.array([0, n], dtype=np.int64), *dev, out)
    assert rc == L.SIM_E_INVAL
    assert "2048" in L.sim_last_error(None)
    # 300 instances of 1000 requests: each within the per-instance limit, 300,000 in total
    off = np.arange(301, dtype=np.int64) * 1000
    dev = [torch.ones(300_000, dtype=torch.int32, device="cuda") for _ in range(5)]
    out = torch.zeros(300 * L.RESULT_DTYPE.itemsize, dtype=torch.uint8, device="cuda")
    rc = L.sim_run_noalloc(L.SIM_AMIN, 10_000, off, *dev, out)
    assert rc == L.SIM_E_INVAL
    assert "262144" in L.sim_last_error(None)
