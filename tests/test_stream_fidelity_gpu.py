"""GPU parity of the streaming loop's fidelity modes (maps_stream_run with
per_step = 1: admission on every step with preemption; beta >= 0 with
prediction delays: deferral with the round-robin timeout) against the plain
oracle: every choice, quantile, per-batch and per-decoder statistic, bit for
bit."""
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


def run_both(M, ws, oracle, arr, prompt, true, pred, N, D, H, cap, B, Wn, a, mw, pol=0, loc=0,
             acc=0, per_step=1, beta=-1, delay=None):
    sto, cho, qo, so, dso = oracle.stream(N, D, H, cap, B, Wn, a, mw, arr, prompt, true, pred,
                                          dispatch=pol, local=loc, accounting=acc,
                                          with_dec_stats=True, per_step=per_step, beta=beta,
                                          pred_delay=delay)
    nb = (N + B - 1) // B
    ch = torch.full((N,), -9, dtype=torch.int32, device="cuda")
    q = torch.full((nb,), -9, dtype=torch.int32, device="cuda")
    stats = torch.full((nb, 4), -9, dtype=torch.int64, device="cuda")
    ds = torch.full((D, 4), -9, dtype=torch.int64, device="cuda")
    cfg = M.stream_cfg(N, D, H, cap, B, Wn, a, mw, pol, loc, acc, per_step, beta)
    st = M.maps_stream_run(cfg, dev(arr[:N], np.int64), dev(prompt[:N], np.int32),
                           dev(true[:N], np.int32), dev(pred[:N], np.int32), ch, q, stats, ds,
                           ws=ws, pred_delay=None if delay is None else dev(delay[:N], np.int32))
    assert st == sto
    if st == 0:
        assert np.array_equal(q.cpu().numpy(), qo)
        assert np.array_equal(ch.cpu().numpy(), cho)
        assert np.array_equal(stats.cpu().numpy(), so)
        assert np.array_equal(ds.cpu().numpy(), dso)
    return so, dso


def on_stream(M, ws, oracle, w, N, D, H, cap, B, Wn, a, mw, **kw):
    return run_both(M, ws, oracle, w["arrival_ms"], w["prompt"], w["true"], w["pred"], N, D, H,
                    cap, B, Wn, a, mw, **kw)


def test_hand_traces(M, ws, oracle):
    """The oracle's hand-traced preemption and deferral cases."""
    a = lambda *x: np.array(x)  # noqa: E731
    so, dso = run_both(M, ws, oracle, a(0, 3, 100), a(10, 10, 1), a(50, 20, 1), a(5, 5, 1), 3, 1,
                       64, 40, 1, 4, 100000, 1000)
    assert dso.tolist() == [[33, 0, 5, 2]]
    so, dso = run_both(M, ws, oracle, a(0, 1, 20, 60), a(10, 10, 1, 1), a(5, 5, 1, 1),
                       a(5, 5, 1, 1), 4, 1, 64, 70, 1, 4, 100000, 1000, per_step=0, beta=5,
                       delay=a(0, 50, 0, 0))
    assert so.tolist() == [[0, 1, 0, 0], [0, 0, 0, 0], [1, 1, 1, 0], [1, 2, 0, 0]]


@pytest.mark.parametrize("cap", [6000, 10000, 16000])
@pytest.mark.parametrize("acc", [0, 1, 2])
def test_per_step_preemption(M, ws, oracle, cap, acc):
    """Per-step admission on a 20,000-request prefix at capacities where
    queues form and (with occupancy accounting) decoders preempt."""
    w = W.make_stream(n_requests=20000)
    so, dso = on_stream(M, ws, oracle, w, 20000, 32, 16384, cap, 256, 500, 100000, 1000, acc=acc)
    if acc == 0 and cap <= 10000:
        assert dso[:, 3].sum() > 0


@pytest.mark.parametrize("per_step,beta", [(0, 0), (0, 300), (1, 300), (1, 1000), (0, 10**6)])
@pytest.mark.parametrize("pol", [0, 1, 2, 3])
def test_deferral(M, ws, oracle, per_step, beta, pol):
    """Prediction delays of up to 1.5 s: some requests wait for their bound,
    some time out to round robin, under every dispatch policy."""
    w = W.make_stream(n_requests=20000)
    delay = np.random.default_rng(3).integers(0, 1500, 20000).astype(np.int32)
    on_stream(M, ws, oracle, w, 20000, 32, 16384, 10000, 256, 500, 100000, 1000, pol=pol,
              per_step=per_step, beta=beta, delay=delay)


@pytest.mark.parametrize("N,D,H,cap,B,Wn,a,mw", [
    (300, 32, 16384, 262144, 256, 500, 100000, 1000),     # ragged, round robin throughout
    (20000, 4, 4096, 12000, 256, 500, 100000, 1000),      # few decoders, long queues
    (20000, 3, 2048, 9000, 100, 37, 300000, 50),          # promotions, small window
    (5000, 40, 1000, 20000, 33, 7, 500000, 0),            # more decoders than a warp's lanes
    (3000, 8, 16384, 3000, 256, 500, 100000, 1000),       # capacity far below demand
    (3000, 200, 2048, 60000, 256, 300, 100000, 1000),     # dense-projection dispatch
])
def test_shapes(M, ws, oracle, N, D, H, cap, B, Wn, a, mw):
    w = W.make_stream(n_requests=N)
    delay = np.random.default_rng(N).integers(0, 2000, N).astype(np.int32)
    on_stream(M, ws, oracle, w, N, D, H, cap, B, Wn, a, mw, per_step=1)
    on_stream(M, ws, oracle, w, N, D, H, cap, B, Wn, a, mw, per_step=1, beta=500, delay=delay,
              acc=1, loc=1)


def test_full_workload(M, ws, oracle):
    """All 1,000,000 requests: per-step admission at the workload's capacity
    with prediction delays and beta = 1 s, and at a capacity of 16,000 where
    decoders preempt."""
    w = W.make_stream()
    delay = np.random.default_rng(11).integers(0, 1500, w["N"]).astype(np.int32)
    args = (w["N"], w["D"], w["H"])
    rest = (w["batch"], w["window"], w["alpha_ppm"], w["max_wait"])
    on_stream(M, ws, oracle, w, *args, w["cap"], *rest, per_step=1, beta=1000, delay=delay)
    so, dso = on_stream(M, ws, oracle, w, *args, 16000, *rest, per_step=1)
    assert dso[:, 3].sum() > 0


def test_bad_fidelity_fields(M, ws):
    w = W.make_stream(n_requests=10)
    t = torch.zeros(10, dtype=torch.int32, device="cuda")
    out = (torch.zeros(3, dtype=torch.int32, device="cuda"),
           torch.zeros((3, 4), dtype=torch.int64, device="cuda"))
    cfg = M.stream_cfg(10, 4, 64, 1000, 4, 5, 100000, 10, per_step=2)
    assert M.maps_stream_run(cfg, dev(w["arrival_ms"][:10], np.int64), t, t, t, t, *out,
                             ws=ws) == M.MAPS_E_INVALID
    cfg = M.stream_cfg(10, 4, 64, 1000, 4, 5, 100000, 10, beta=5)  # beta without delays
    assert M.maps_stream_run(cfg, dev(w["arrival_ms"][:10], np.int64), t, t, t, t, *out,
                             ws=ws) == M.MAPS_E_INVALID
    ones = torch.ones(10, dtype=torch.int32, device="cuda")
    neg = torch.full((10,), -1, dtype=torch.int32, device="cuda")
    assert M.maps_stream_run(cfg, dev(w["arrival_ms"][:10], np.int64), ones, ones, ones, t, *out,
                             ws=ws, pred_delay=neg) == M.MAPS_E_RANGE
