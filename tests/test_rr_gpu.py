"""GPU parity of the App. A round-robin KV-pressure simulation
(maps_rr_pressure) against the plain oracle: every admission and completion
time, every decoder's high-pressure metrics and waiting statistics, and each
realisation's span -- bit for bit."""
import numpy as np
import pytest
import torch

from paper_2609_15359_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def M():
    if not torch.cuda.is_available():
        pytest.fail("CUDA device required for -m gpu tests")
    from paper_2609_15359_gb300 import maps
    return maps


def gpu_rr(M, N, C, tok, theta, arr, prompt, out):
    arr, prompt, out = np.atleast_2d(arr), np.atleast_2d(prompt), np.atleast_2d(out)
    n_real, n = arr.shape
    t = lambda x, dt: torch.from_numpy(np.ascontiguousarray(x, dtype=dt)).cuda()  # noqa: E731
    adm = torch.full((n_real, n), -1, dtype=torch.int64, device="cuda")
    done = torch.full((n_real, n), -1, dtype=torch.int64, device="cuda")
    stats = torch.full((n_real, N, 6), -1, dtype=torch.int64, device="cuda")
    tsim = torch.full((n_real,), -1, dtype=torch.int64, device="cuda")
    ws = M.Workspace()
    st = M.maps_rr_pressure(N, C, tok, theta, t(arr, np.int64), t(prompt, np.int32),
                            t(out, np.int32), adm, done, stats, tsim, ws=ws)
    assert st == 0
    return M.maps_check(ws), adm.cpu().numpy(), done.cpu().numpy(), stats.cpu().numpy(), \
        tsim.cpu().numpy()


def check(M, oracle, N, C, tok, theta, arr, prompt, out):
    st, adm, done, stats, tsim = gpu_rr(M, N, C, tok, theta, arr, prompt, out)
    assert st == 0
    for r in range(np.atleast_2d(arr).shape[0]):
        sto, a, d, s, ts = oracle.rr_pressure(N, C, tok, theta, np.atleast_2d(arr)[r],
                                              np.atleast_2d(prompt)[r], np.atleast_2d(out)[r])
        assert sto == 0
        assert np.array_equal(adm[r], a), r
        assert np.array_equal(done[r], d), r
        assert np.array_equal(stats[r], s), r
        assert tsim[r] == ts, r


def test_rr_app_a_setup_full_size(M, oracle):
    """N = 4, C = 50,000, t_tok = 1 ms, theta = 0.85, 10,000 requests, six
    utilisations from light load to overload, two workload draws."""
    w = W.make_rr(2)
    check(M, oracle, w["N"], w["C"], w["t_tok_us"], w["theta_ppm"], w["arrival_us"],
          w["prompt"], w["out_len"])


@pytest.mark.parametrize("N,C,n,theta,tie", [(1, 3000, 1, 500000, False), (1, 3000, 33, 850000, True),
                                             (3, 5000, 200, 850000, True), (7, 20000, 1000, 900000, False),
                                             (4, 50000, 3, 1000000, True), (16, 8000, 5000, 300000, False),
                                             (5, 2100, 700, 1, True)])
def test_rr_random(M, oracle, N, C, n, theta, tie):
    """Tight capacities (queues and head-of-line blocking), equal arrival
    times, more decoders than requests, thresholds at both ends."""
    rng = np.random.default_rng(N * 1000 + n)
    n_real = 3
    out = rng.integers(1, 300, (n_real, n))
    prompt = np.minimum(rng.integers(0, 2000, (n_real, n)), C - out)
    gaps = rng.integers(0, 3 if tie else 400_000, (n_real, n))
    arr = np.cumsum(gaps, axis=1) + rng.integers(0, 10**6, (n_real, 1))
    check(M, oracle, N, C, 1000, theta, arr, prompt, out)


def test_rr_errors(M, oracle):
    # a footprint above C could never be admitted
    st, *_ = gpu_rr(M, 2, 100, 1000, 850000, [[0, 1, 2]], [[10, 95, 10]], [[5, 10, 5]])
    assert st == M.MAPS_E_RANGE == oracle.rr_pressure(2, 100, 1000, 850000, [0, 1, 2],
                                                      [10, 95, 10], [5, 10, 5])[0]
    st, *_ = gpu_rr(M, 2, 100, 1000, 850000, [[0, 1]], [[10, 10]], [[5, 0]])
    assert st == M.MAPS_E_RANGE
    st, *_ = gpu_rr(M, 1, 100, 1000, 850000, [[5, 4]], [[1, 1]], [[1, 1]])
    assert st == M.MAPS_E_RANGE
    # more requests admitted at once on one decoder than its running set holds
    n = 2000
    st, *_ = gpu_rr(M, 1, 10**9, 1000, 850000, [np.zeros(n)], [np.zeros(n)], [np.full(n, 5)])
    assert st == M.MAPS_E_RANGE
    cfg = M.RRCfg(0, 1, 1, 1, 1)
    assert M.lib.maps_rr_pressure(cfg, 1, None, None, None, None, None, None, None, None, 0,
                                  None) == M.MAPS_E_INVALID
