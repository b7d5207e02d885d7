"""Random medium instances, past the one-block limits of every call, so that
the multi-kernel forms run on shapes nobody chose: several tiles and blocks
with ragged tails, skewed decoders, empty decoders, arrival in and out of
index order, bounds of a few bits to the full 31.  Each output is compared
element by element with the plain oracle (tier P), which the CPU tests pin
to the by-definition one; the statuses must agree.  Each draw is seeded, and
a failure reports its iteration."""
import os

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

# draws per test; MAPS_FUZZ_ITERATIONS runs a longer sweep
ITERATIONS = int(os.environ.get("MAPS_FUZZ_ITERATIONS", "100"))


@pytest.fixture(scope="module")
def M():
    if not torch.cuda.is_available():
        pytest.fail("CUDA device required for -m gpu tests")
    from paper_2609_15359_gb300 import maps
    return maps


def dev(x, dtype):
    return torch.from_numpy(np.ascontiguousarray(np.asarray(x, dtype=dtype))).cuda()


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def test_random_medium_calibration(M, oracle):
    rng = np.random.default_rng(41)
    ws = M.Workspace()
    for it in range(ITERATIONS):
        n = int(rng.integers(8193, 1_400_000))
        hi = int(rng.choice([50, 5_000, 2**20, 2**31 - 1]))
        L = rng.integers(0, hi, n, dtype=np.int64).astype(np.int32)
        P = rng.integers(0, hi, n, dtype=np.int64).astype(np.int32)
        P[: n // 3] = L[: n // 3]
        a = int(rng.integers(1_000, 999_000))
        m = int(rng.integers(0, 1_500_000))
        pred = rng.integers(0, 60_000, m).astype(np.int32)
        sto, qo = oracle.p_calibrate(L, P, a)
        if sto == 0 and m:
            sto, Uo = oracle.p_bound(pred, qo)
        U = torch.full((m + 1,), -9, dtype=torch.int32, device="cuda")
        st, q = M.maps_calibrate(dev(L, np.int32), dev(P, np.int32), a,
                                 dev(pred, np.int32) if m else None, U[:m] if m else None,
                                 q_host=True, ws=ws)
        assert st == sto, (it, n, m)
        if st == 0:
            assert q == qo, (it, n)
            Uh = host(U)
            assert (not m or np.array_equal(Uh[:m], Uo)) and Uh[m] == -9, (it, n, m)


def test_random_medium_occupancy_and_dispatch(M, oracle):
    rng = np.random.default_rng(43)
    ws = M.Workspace()
    for it in range(ITERATIONS):
        D = int(rng.integers(1, 300))
        H = int(rng.integers(1, 70_000))
        per = rng.integers(0, int(rng.integers(1, 5_000)), D)
        per[rng.random(D) < 0.2] = 0  # decoders without residents
        off = np.concatenate([[0], np.cumsum(per)]).astype(np.int64)
        R = int(off[-1])
        p = rng.integers(0, 2_000, R).astype(np.int32)
        g = rng.integers(0, 3_000, R).astype(np.int32)
        U = (g + rng.integers(-50, H + 100, R)).clip(0).astype(np.int32)
        sto, Ko = oracle.p_occupancy(D, H, off, p, g, U)
        K = torch.full((D, H), -7, dtype=torch.int32, device="cuda")
        assert M.maps_project_occupancy(D, H, dev(off, np.int64), dev(p, np.int32),
                                        dev(g, np.int32), dev(U, np.int32), K, None, ws=ws) == 0
        st = M.maps_check(ws)
        assert st == sto, (it, D, H, R)
        if st != 0:
            continue
        assert np.array_equal(host(K), Ko), (it, D, H, R)
        J = int(rng.integers(1, 70_000))
        cp = rng.integers(0, 4_000, J).astype(np.int32)
        cb = rng.integers(1, H + 200, J).astype(np.int32)
        cap = (Ko.max(axis=1).astype(np.int64) + rng.integers(-5_000, 300_000, D)).clip(
            0, 2**31 - 1).astype(np.int32)
        Q = rng.integers(0, 50, D).astype(np.int32)
        sto, cho, hro = oracle.p_dispatch_snapshot(D, H, Ko, cap, Q, cp, cb)
        ch = torch.full((J + 1,), -9, dtype=torch.int32, device="cuda")
        hr = torch.full((J + 1,), -9, dtype=torch.int64, device="cuda")
        assert M.maps_dispatch(M.MODE_SNAPSHOT, D, H, 1, K, dev(cap, np.int32), dev(Q, np.int32),
                               dev(cp, np.int32), dev(cb, np.int32), ch[:J], hr[:J], ws=ws) == 0
        st = M.maps_check(ws)
        assert st == sto, (it, D, H, J)
        if st == 0:
            assert np.array_equal(host(ch)[:J], cho), (it, D, H, J)
            assert np.array_equal(host(hr)[:J], hro), (it, D, H, J)
            assert host(ch)[J] == -9 and host(hr)[J] == -9, it


def test_random_medium_order(M, oracle):
    rng = np.random.default_rng(47)
    ws = M.Workspace()
    for it in range(ITERATIONS):
        N = int(rng.integers(4_609, 1_300_000))
        D = int(rng.choice([1, 7, 64, 256, 1024, 1025, 3000]))
        dec = rng.integers(0, D, N).astype(np.int32)
        skew = rng.random()
        dec[rng.random(N) < skew * 0.5] = int(rng.integers(0, D))  # one long queue, or none
        ubits = int(rng.integers(1, 32))
        U = rng.integers(0, 2**ubits, N, dtype=np.int64).astype(np.int32)
        wait = rng.integers(-10, 3_000, N).astype(np.int32)
        if rng.random() < 0.6:
            arr = np.sort(rng.integers(0, max(N // 2, 1), N)).astype(np.int32)
        else:
            arr = rng.integers(0, 2**31 - 1, N, dtype=np.int64).astype(np.int32)
        sto, po, so = oracle.p_order_local(D, dec, U, wait, arr, 1000)
        perm = torch.full((N + 1,), -1, dtype=torch.int32, device="cuda")
        seg = torch.full((D + 1,), -1, dtype=torch.int64, device="cuda")
        assert M.maps_order_local(D, dev(dec, np.int32), dev(U, np.int32), dev(wait, np.int32),
                                  dev(arr, np.int32), 1000, perm[:N], seg, ws=ws) == 0
        st = M.maps_check(ws)
        assert st == sto == 0, (it, N, D)
        assert np.array_equal(host(perm)[:N], po), (it, N, D, ubits)
        assert host(perm)[N] == -1 and np.array_equal(host(seg), so), (it, N, D)
