"""Random tiny instances through every call of the C ABI, against the
by-definition oracle: the status always, the outputs whenever the call
succeeds.  Sizes start at zero; lengths fall in and out of the domain;
horizons go down to one step; decoders may have no residents; values are
drawn from small ranges so that ties are everywhere.  Each draw is seeded,
and a failure reports its iteration."""
import os

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

# draws per test; MAPS_FUZZ_ITERATIONS runs a longer sweep
ITERATIONS = int(os.environ.get("MAPS_FUZZ_ITERATIONS", "3000"))


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


def test_random_tiny_calibration(M, oracle):
    rng = np.random.default_rng(31)
    ws = M.Workspace()
    for it in range(ITERATIONS):
        n = int(rng.integers(0, 40))
        L = rng.integers(0, 60, n).astype(np.int32)
        P = rng.integers(0, 60, n).astype(np.int32)
        a = int(rng.integers(1, 10**6))
        m = int(rng.integers(0, 10))
        query = rng.integers(0, 100, m).astype(np.int32)
        sto, qo = oracle.calibrate(L, P, a)
        if sto == 0 and m:
            sto, Uo = oracle.bound(query, qo)
        U = torch.full((m + 1,), -9, dtype=torch.int32, device="cuda")
        st, q = M.maps_calibrate(dev(L, np.int32), dev(P, np.int32), a,
                                 dev(query, np.int32) if m else None, U[:m] if m else None,
                                 q_host=True, ws=ws)
        assert st == sto, it
        if st == 0:
            assert q == qo, it
            Uh = host(U)
            assert (not m or np.array_equal(Uh[:m], Uo)) and Uh[m] == -9, it


def test_random_tiny_occupancy_dispatch_order(M, oracle):
    rng = np.random.default_rng(37)
    ws = M.Workspace()
    seen = set()
    for it in range(ITERATIONS):
        # occupancy
        D, H = int(rng.integers(1, 6)), int(rng.integers(1, 40))
        per = rng.integers(0, 6, D)
        off = np.concatenate([[0], np.cumsum(per)]).astype(np.int64)
        R = int(off[-1])
        p = rng.integers(0, 30, R).astype(np.int32)
        g = rng.integers(0, 2 * H + 2, R).astype(np.int32)
        U = rng.integers(0, 3 * H + 2, R).astype(np.int32)
        if R and it % 10 == 0:
            [p, g, U][it % 3][int(rng.integers(0, R))] = -1  # a length outside the domain
        sto, Ko = oracle.occupancy(D, H, off, p, g, U)
        K = torch.full((D, H), -7, dtype=torch.int32, device="cuda")
        assert M.maps_project_occupancy(D, H, dev(off, np.int64), dev(p, np.int32),
                                        dev(g, np.int32), dev(U, np.int32), K, None, ws=ws) == 0
        st = M.maps_check(ws)
        assert st == sto, it
        seen.add(("occupancy", st))
        if st != 0:
            continue
        assert np.array_equal(host(K), Ko), it
        # dispatch, every mode (ALG1 with the same residents, S of 1 to 4)
        J = int(rng.integers(0, 12))
        cp = rng.integers(0, 50, J).astype(np.int32)
        cb = rng.integers(0, 2 * H + 3, J).astype(np.int32)
        if J and it % 7 == 0:
            cb[0] = -2
        cap = (Ko.max(axis=1) + rng.integers(-40, 80, D)).clip(0).astype(np.int32)
        Q = rng.integers(0, 3, D).astype(np.int32)
        mode = it % 4
        S = int(rng.integers(1, 5)) if mode >= 2 else 1
        res = (off, p, g, U) if mode >= 2 else (None, None, None, None)
        sto, cho, hro, Kao, Qao = oracle.dispatch(mode, D, H, S, Ko if mode < 2 else None, cap, Q,
                                                  cp, cb, *res)
        Kd = dev(Ko, np.int32)
        Qd = dev(Q, np.int32)
        ch = torch.full((J + 1,), -9, dtype=torch.int32, device="cuda")
        hr = torch.full((J + 1,), -9, dtype=torch.int64, device="cuda")
        kw = {} if mode < 2 else dict(res_off=dev(off, np.int64), prompt=dev(p, np.int32),
                                      gen=dev(g, np.int32), bound=dev(U, np.int32))
        assert M.maps_dispatch(mode, D, H, S, Kd if mode < 2 else None, dev(cap, np.int32), Qd,
                               dev(cp, np.int32), dev(cb, np.int32), ch[:J], hr[:J], ws=ws,
                               **kw) == 0
        st = M.maps_check(ws)
        assert st == sto, (it, mode)
        seen.add(("dispatch", mode, st))
        if st == 0:
            assert np.array_equal(host(ch)[:J], cho), (it, mode)
            assert np.array_equal(host(hr)[:J], hro), (it, mode)
            assert host(ch)[J] == -9 and host(hr)[J] == -9, (it, mode)
            if mode in (1, 3):
                assert np.array_equal(host(Qd), Qao), (it, mode)
            if mode == 1:
                assert np.array_equal(host(Kd), Kao), (it, mode)
        # local order
        N = int(rng.integers(0, 30))
        dec = rng.integers(0, D, N).astype(np.int32)
        bnd = rng.integers(0, 8, N).astype(np.int32)
        wait = rng.integers(0, 6, N).astype(np.int32)
        arr = rng.integers(0, 10, N).astype(np.int32)
        if N and it % 11 == 0:
            dec[0] = D  # a decoder outside the domain
        sto, po, so = oracle.order_local(D, dec, bnd, wait, arr, 2)
        perm = torch.full((N + 1,), -1, dtype=torch.int32, device="cuda")
        seg = torch.full((D + 1,), -1, dtype=torch.int64, device="cuda")
        assert M.maps_order_local(D, dev(dec, np.int32), dev(bnd, np.int32), dev(wait, np.int32),
                                  dev(arr, np.int32), 2, perm[:N], seg, ws=ws) == 0
        st = M.maps_check(ws)
        assert st == sto, it
        seen.add(("order", st))
        if st == 0:
            assert np.array_equal(host(perm)[:N], po) and host(perm)[N] == -1, it
            assert np.array_equal(host(seg), so), it
    # both outcomes of every call came up
    for key in (("occupancy", 0), ("occupancy", M.MAPS_E_RANGE), ("order", 0),
                ("order", M.MAPS_E_RANGE)):
        assert key in seen, key
    for mode in range(4):
        assert ("dispatch", mode, 0) in seen and ("dispatch", mode, M.MAPS_E_RANGE) in seen, mode
