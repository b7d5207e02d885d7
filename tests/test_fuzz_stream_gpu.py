"""Random configurations of the streaming loop against the plain oracle:
decoder counts from 1 to 48, capacities from starved to ample, batches from
one request to 300, windows from 1 to 600, every dispatch policy, local order
and accounting, and both fidelity modes (per-step admission; deferral with a
modelled prediction delay).  Every choice, quantile, per-batch and
per-decoder statistic must agree bit for bit, and so must the status.  Each
configuration is seeded, and a failure reports it."""
import os

import numpy as np
import pytest
import torch

from paper_2609_15359_gb300 import workloads as W

pytestmark = pytest.mark.gpu

# configurations per test; MAPS_FUZZ_ITERATIONS runs a longer sweep
ITERATIONS = int(os.environ.get("MAPS_FUZZ_ITERATIONS", "200"))


@pytest.fixture(scope="module")
def M():
    if not torch.cuda.is_available():
        pytest.fail("CUDA device required for -m gpu tests")
    from paper_2609_15359_gb300 import maps
    return maps


def dev(x, dt):
    return torch.from_numpy(np.ascontiguousarray(x, dtype=dt)).cuda()


def test_random_stream_configurations(M, oracle):
    rng = np.random.default_rng(53)
    ws = M.Workspace()
    for it in range(ITERATIONS):
        N = int(rng.integers(1, 5000))
        D = int(rng.choice([1, 2, 3, 8, 17, 32, 33, 48]))
        H = int(rng.choice([64, 1000, 4096, 16384]))
        cap = int(rng.choice([2_000, 8_000, 20_000, 100_000, 400_000]))
        B = int(rng.integers(1, 300))
        Wn = int(rng.integers(1, 600))
        a = int(rng.choice([1_000, 50_000, 100_000, 300_000]))
        mw = int(rng.choice([0, 50, 1000]))
        pol, loc, acc = int(rng.integers(0, 4)), int(rng.integers(0, 2)), int(rng.integers(0, 3))
        per_step = int(rng.integers(0, 2))
        beta = int(rng.choice([-1, -1, 200, 1000]))
        w = W.make_stream(seed=int(rng.integers(0, 2**31)), n_requests=N)
        delay = w["pred_delay_ms"][:N] if beta >= 0 else None
        conf = (it, N, D, H, cap, B, Wn, a, mw, pol, loc, acc, per_step, beta)
        sto, cho, qo, so, dso = oracle.stream(N, D, H, cap, B, Wn, a, mw, w["arrival_ms"],
                                              w["prompt"], w["true"], w["pred"], dispatch=pol,
                                              local=loc, accounting=acc, with_dec_stats=True,
                                              per_step=per_step, beta=beta, pred_delay=delay)
        nb = (N + B - 1) // B
        ch = torch.full((N,), -9, dtype=torch.int32, device="cuda")
        q = torch.full((nb,), -9, dtype=torch.int32, device="cuda")
        stats = torch.full((nb, 4), -9, dtype=torch.int64, device="cuda")
        ds = torch.full((D, 4), -9, dtype=torch.int64, device="cuda")
        cfg = M.stream_cfg(N, D, H, cap, B, Wn, a, mw, pol, loc, acc, per_step, beta)
        st = M.maps_stream_run(cfg, dev(w["arrival_ms"][:N], np.int64), dev(w["prompt"][:N], np.int32),
                               dev(w["true"][:N], np.int32), dev(w["pred"][:N], np.int32), ch, q,
                               stats, ds, ws=ws,
                               pred_delay=None if delay is None else dev(delay, np.int32))
        assert st == sto, conf
        if st == 0:
            assert np.array_equal(q.cpu().numpy(), qo), conf
            assert np.array_equal(ch.cpu().numpy(), cho), conf
            assert np.array_equal(stats.cpu().numpy(), so), conf
            assert np.array_equal(ds.cpu().numpy(), dso), conf
