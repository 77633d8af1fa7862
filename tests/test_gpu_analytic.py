"""CUDA analytic evaluators (sim_cr_amin_lemma, sim_cr_amin_rho) against the CPU analytic oracle
and the paper's closed forms."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()


def test_lemma_matches_oracle_random_histograms():
    """Random histograms of several lengths (one chunk, many chunks, a ragged tail), s = 0 and
    s > 0: relative difference below 1e-12 (double, different summation order)."""
    from oracle import analytic as an
    from paper_2508_14544_gb300 import cr_amin_lemma
    rng = np.random.default_rng(8)
    for length, l, s in ((1, 1, 0.0), (7, 1, 0.0), (32, 3, 2.0), (33, 2, 1.5), (100, 5, 7.0), (257, 1, 0.0)):
        x = rng.random((40, length))
        x[::7, 1::3] = 0.0  # some zero bins (the first bin stays positive)
        got = cr_amin_lemma(x, l, s)
        ref = np.array([an.lemma_amin_cr(row, l, s) for row in x])
        assert np.all(np.abs(got - ref) <= 1e-12 * np.abs(ref)), (length, np.max(np.abs(got - ref) / ref))


def test_lemma_closed_forms_on_gpu():
    """LG theorem (q in (0, 0.85], truncated at u = 600), two-point form of the Theorem thm:no proof
    and its maximum 1 + (1 - a)/2 at t = 1/a."""
    from oracle import analytic as an
    from paper_2508_14544_gb300 import cr_amin_lemma
    qs = np.array([0.05, 0.2, 0.5, 0.7, 0.85])
    k = np.arange(1, 601, dtype=np.float64)
    x = np.stack([k * q ** (k - 1) for q in qs])
    got = cr_amin_lemma(x, 1, 0.0)
    want = np.array([an.lg_cr(q) for q in qs])
    assert np.all(np.abs(got - want) < 1e-12)
    l, u = 2, 10
    a = l / u
    ts = np.array([0.3, 1.0, 1 / a, 9.0])
    x = np.zeros((len(ts), u - l + 1))
    x[:, 0] = ts
    x[:, -1] = 1.0
    got = cr_amin_lemma(x, l, 0.0)
    assert np.all(np.abs(got - np.array([an.two_point_cr(a, t) for t in ts])) < 1e-12)
    assert abs(got[2] - (1 + (1 - a) / 2)) < 1e-12


def test_lemma_device_pointers():
    import torch

    from paper_2508_14544_gb300 import cr_amin_lemma
    rng = np.random.default_rng(9)
    x = rng.random((1000, 64))
    host = cr_amin_lemma(x, 1, 0.0)
    dev = cr_amin_lemma(torch.from_numpy(x).cuda(), 1, 0.0)
    torch.cuda.synchronize()
    assert np.array_equal(dev.cpu().numpy(), host)


def test_rho_matches_oracle_and_bounds():
    """Power iteration with O(u) products against scipy's dense generalized eigensolver: relative
    difference below 1e-10; 1 <= rho <= H_u; random positive histograms stay below rho."""
    from oracle import analytic as an
    from paper_2508_14544_gb300 import cr_amin_lemma, cr_amin_rho
    us = [1, 2, 3, 10, 31, 32, 33, 100, 500, 1000]
    got = cr_amin_rho(us)
    for u, r in zip(us, got):
        ref = an.rho(u)
        assert abs(r - ref) <= 1e-10 * ref, (u, r, ref)
        assert 1.0 - 1e-12 <= r <= sum(1 / i for i in range(1, u + 1)) + 1e-9
    rng = np.random.default_rng(10)
    x = rng.random((50, 100))
    assert np.all(cr_amin_lemma(x, 1, 0.0) <= got[us.index(100)] + 1e-9)


def test_rho_large_u_follows_the_fit():
    """The figure's fit 0.2555 log(u + 0.2793) + 1.1587 within 2 % up to u = 100000."""
    from paper_2508_14544_gb300 import cr_amin_rho
    us = [10, 100, 1000, 10000, 100000]
    got = cr_amin_rho(us)
    fit = 0.2555 * np.log(np.array(us) + 0.2793) + 1.1587
    assert np.all(np.abs(got - fit) / fit < 0.02), (got, fit)
    assert np.all(np.diff(got) > 0)


def test_invalid_arguments():
    from paper_2508_14544_gb300 import SimError, cr_amin_lemma, cr_amin_rho
    with pytest.raises(SimError):
        cr_amin_rho([0])
    with pytest.raises(SimError):
        cr_amin_lemma(np.ones((2, 3)), 0, 0.0)
    with pytest.raises(SimError):
        cr_amin_lemma(np.ones((2, 3)), 1, -1.0)
