"""GPU parity of the streaming loop's policy variants (maps_stream_run with
dispatch_policy / local_order / accounting) against the plain oracle: every
choice, quantile, per-batch and per-decoder statistic, bit for bit."""
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


@pytest.fixture(scope="module")
def ws(M):
    return M.Workspace()


def dev(x, dt):
    return torch.from_numpy(np.ascontiguousarray(x, dtype=dt)).cuda()


def run_both(M, ws, oracle, w, N, D, H, cap, B, Wn, a, mw, pol, loc, acc):
    sto, cho, qo, so, dso = oracle.stream(N, D, H, cap, B, Wn, a, mw, w["arrival_ms"], w["prompt"],
                                          w["true"], w["pred"], dispatch=pol, local=loc,
                                          accounting=acc, with_dec_stats=True)
    nb = (N + B - 1) // B
    ch = torch.full((N,), -9, dtype=torch.int32, device="cuda")
    q = torch.full((nb,), -9, dtype=torch.int32, device="cuda")
    stats = torch.full((nb, 4), -9, dtype=torch.int64, device="cuda")
    ds = torch.full((D, 4), -9, dtype=torch.int64, device="cuda")
    cfg = M.stream_cfg(N, D, H, cap, B, Wn, a, mw, pol, loc, acc)
    st = M.maps_stream_run(cfg, dev(w["arrival_ms"][:N], np.int64), dev(w["prompt"][:N], np.int32),
                           dev(w["true"][:N], np.int32), dev(w["pred"][:N], np.int32), ch, q, stats,
                           ds, ws=ws)
    assert st == sto
    if st == 0:
        assert np.array_equal(q.cpu().numpy(), qo)
        assert np.array_equal(ch.cpu().numpy(), cho)
        assert np.array_equal(stats.cpu().numpy(), so)
        assert np.array_equal(ds.cpu().numpy(), dso)
    return so, dso


VARIANTS = [(p, l, a) for p in range(4) for l in range(2) for a in range(3)]


@pytest.mark.parametrize("pol,loc,acc", VARIANTS)
def test_variants_tight_capacity(M, ws, oracle, pol, loc, acc):
    """24 combinations on a 20,000-request prefix of the streaming workload
    whose capacity makes queues form and block."""
    w = W.make_stream(n_requests=20000)
    so, dso = run_both(M, ws, oracle, w, 20000, 32, 16384, 10000, 256, 500, 100000, 1000,
                       pol, loc, acc)
    assert so[:, 2].sum() > 0  # something waited


@pytest.mark.parametrize("N,D,H,cap,B,Wn,a,mw", [
    (300, 32, 16384, 262144, 256, 500, 100000, 1000),     # ragged, round robin throughout
    (20000, 4, 4096, 12000, 256, 500, 100000, 1000),      # few decoders, long queues
    (20000, 3, 2048, 9000, 100, 37, 300000, 50),          # promotions, small window
    (5000, 40, 1000, 20000, 33, 7, 500000, 0),            # more decoders than a warp's lanes
    (3000, 8, 16384, 3000, 256, 500, 100000, 1000),       # deficits past 2^21
    (3000, 200, 2048, 60000, 256, 300, 100000, 1000),     # dense-projection dispatch
])
@pytest.mark.parametrize("pol,loc,acc", [(1, 0, 0), (3, 1, 1), (2, 0, 2), (1, 1, 2), (3, 0, 0)])
def test_variants_shapes(M, ws, oracle, N, D, H, cap, B, Wn, a, mw, pol, loc, acc):
    w = W.make_stream(n_requests=N)
    run_both(M, ws, oracle, w, N, D, H, cap, B, Wn, a, mw, pol, loc, acc)


def test_default_policies_match_the_plain_call(M, ws, oracle):
    """The default fields are the MAPS loop: same outputs as the call made
    without per-decoder statistics."""
    w = W.make_stream(n_requests=8000)
    so, dso = run_both(M, ws, oracle, w, 8000, 32, 16384, 10000, 256, 500, 100000, 1000, 0, 0, 0)
    nb = (8000 + 255) // 256
    ch = torch.empty(8000, dtype=torch.int32, device="cuda")
    q = torch.empty(nb, dtype=torch.int32, device="cuda")
    stats = torch.empty((nb, 4), dtype=torch.int64, device="cuda")
    cfg = M.stream_cfg(8000, 32, 16384, 10000, 256, 500, 100000, 1000)
    assert M.maps_stream_run(cfg, dev(w["arrival_ms"][:8000], np.int64),
                             dev(w["prompt"][:8000], np.int32), dev(w["true"][:8000], np.int32),
                             dev(w["pred"][:8000], np.int32), ch, q, stats, ws=ws) == 0
    assert np.array_equal(stats.cpu().numpy(), so)


def test_variants_full_workload(M, ws, oracle):
    """All 1,000,000 requests, max-headroom dispatch with FCFS and held
    accounting, and least requests with staged accounting."""
    w = W.make_stream()
    for pol, loc, acc in [(1, 1, 2), (3, 0, 1)]:
        run_both(M, ws, oracle, w, w["N"], w["D"], w["H"], w["cap"], w["batch"], w["window"],
                 w["alpha_ppm"], w["max_wait"], pol, loc, acc)


def test_bad_policy_fields(M, ws):
    w = W.make_stream(n_requests=10)
    for bad in [(4, 0, 0), (-1, 0, 0), (0, 2, 0), (0, 0, 3)]:
        cfg = M.stream_cfg(10, 4, 64, 1000, 4, 5, 100000, 10, *bad)
        t = torch.zeros(10, dtype=torch.int32, device="cuda")
        st = M.maps_stream_run(cfg, dev(w["arrival_ms"][:10], np.int64), t, t, t, t,
                               torch.zeros(3, dtype=torch.int32, device="cuda"),
                               torch.zeros((3, 4), dtype=torch.int64, device="cuda"), ws=ws)
        assert st == M.MAPS_E_INVALID
