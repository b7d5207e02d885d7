"""GPU parity of the App. A round-robin KV-pressure simulation
(maps_rr_pressure) against the plain oracle: every admission and completion
time, every decoder's high-pressure metrics and waiting statistics, and each
realisation's span -- bit for bit."""
import os

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


def test_rr_random_sweep(M, oracle):
    """Random configurations: 1 to 16 decoders, capacities from barely above
    the largest footprint to ample, 1 to 3,000 requests in 1 to 6
    realisations per call, thresholds from 1 ppm to 1, token times of 1 us
    to 2 ms, and arrivals from simultaneous to sparse.  MAPS_FUZZ_ITERATIONS
    runs a longer sweep."""
    rng = np.random.default_rng(59)
    for it in range(int(os.environ.get("MAPS_FUZZ_ITERATIONS", "40"))):
        N = int(rng.integers(1, 17))
        n = int(rng.integers(1, 3000))
        n_real = int(rng.integers(1, 7))
        out = rng.integers(1, int(rng.choice([5, 300, 3000])), (n_real, n))
        C = int(out.max()) + int(rng.choice([1, 500, 5000, 100_000]))
        prompt = np.minimum(rng.integers(0, 4000, (n_real, n)), C - out)
        gaps = rng.integers(0, int(rng.choice([1, 3, 50_000, 2_000_000])), (n_real, n))
        arr = np.cumsum(gaps, axis=1) + rng.integers(0, 10**6, (n_real, 1))
        theta = int(rng.choice([1, 300_000, 850_000, 1_000_000]))
        tok = int(rng.choice([1, 1000, 2000]))
        st, adm, done, stats, tsim = gpu_rr(M, N, C, tok, theta, arr, prompt, out)
        ref = [oracle.rr_pressure(N, C, tok, theta, arr[r], prompt[r], out[r]) for r in range(n_real)]
        # one call covers every realisation: it succeeds when each of them does
        assert (st == 0) == all(x[0] == 0 for x in ref), (it, N, C, n, st)
        if st == 0:
            for r, (_, a, d, s_, ts) in enumerate(ref):
                assert np.array_equal(adm[r], a), (it, r)
                assert np.array_equal(done[r], d), (it, r)
                assert np.array_equal(stats[r], s_), (it, r)
                assert tsim[r] == ts, (it, r)
