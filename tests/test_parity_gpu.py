"""GPU parity: the CUDA path through the C ABI against the CPU oracle.

Integer work throughout, so every comparison is bit-exact (tolerance 0).
Sizes: the hand-derived goldens, seeded random instances with ragged shapes
that span several tiles, and the benchmark workloads at full size (whole
outputs where the oracle finishes in seconds, sampled candidates otherwise).
"""
import numpy as np
import pytest
import torch

from paper_2609_15359_gb300 import workloads as W

pytestmark = pytest.mark.gpu

I32_MAX = 2**31 - 1


@pytest.fixture(scope="module")
def M():
    if not torch.cuda.is_available():
        pytest.fail("CUDA device required for -m gpu tests")
    from paper_2609_15359_gb300 import maps
    return maps


@pytest.fixture(scope="module")
def ws(M):
    return M.Workspace()


def dev(x, dtype=None):
    a = np.ascontiguousarray(x if dtype is None else np.asarray(x, dtype=dtype))
    return torch.from_numpy(a).cuda()


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


# ---------------------------------------------------------------------------
# helpers running one op on the GPU and returning (status, outputs)
# ---------------------------------------------------------------------------

def gpu_calibrate(M, ws, L, P, a, query=None):
    m = 0 if query is None else len(query)
    U = torch.empty(max(m, 1), dtype=torch.int32, device="cuda")
    qd = torch.zeros(1, dtype=torch.int32, device="cuda")
    st, q = M.maps_calibrate(dev(L, np.int32), dev(P, np.int32), a,
                             None if query is None else dev(query, np.int32),
                             U[:m] if m else None, qd, q_host=True, ws=ws)
    return st, q, int(host(qd)[0]), host(U[:m])


def gpu_occupancy(M, ws, D, H, off, p, g, u, with_kmax=False):
    K = torch.full((D, H), -7, dtype=torch.int32, device="cuda")
    km = torch.full(M.kmax_shape(D, H), -7, dtype=torch.int32, device="cuda") if with_kmax else None
    st = M.maps_project_occupancy(D, H, dev(off, np.int64), dev(p, np.int32), dev(g, np.int32),
                                  dev(u, np.int32), K, km, ws=ws)
    assert st == 0
    if with_kmax:
        return M.maps_check(ws), host(K), host(km).view(np.uint32)
    return M.maps_check(ws), host(K)


def kmax_of(K):
    """16-step block maxima of K + t (the summary's definition, in numpy)."""
    D, H = K.shape
    x = K.astype(np.int64) + np.arange(H)
    nb = (H + 15) // 16
    pad = np.full((D, nb * 16), -1, np.int64)
    pad[:, :H] = x
    return pad.reshape(D, nb, 16).max(axis=2).astype(np.uint32)


def gpu_dispatch(M, ws, mode, D, H, S, K, cap, Q, cp, cb, res=None, kmax=None):
    J = len(cp)
    Kd = None if K is None else dev(K, np.int32)
    kmd = None if kmax is None else dev(np.ascontiguousarray(kmax).view(np.int32))
    Qd = dev(Q, np.int32)
    ch = torch.full((max(J, 1),), -9, dtype=torch.int32, device="cuda")
    hr = torch.full((max(J, 1),), -9, dtype=torch.int64, device="cuda")
    kw = {}
    if res is not None:
        kw = dict(res_off=dev(res[0], np.int64), prompt=dev(res[1], np.int32),
                  gen=dev(res[2], np.int32), bound=dev(res[3], np.int32))
    st = M.maps_dispatch(mode, D, H, S, Kd, dev(cap, np.int32), Qd, dev(cp, np.int32),
                         dev(cb, np.int32), ch[:J], hr[:J], kmax=kmd, ws=ws, **kw)
    assert st == 0, st
    st = M.maps_check(ws)
    return st, host(ch[:J]), host(hr[:J]), (None if Kd is None else host(Kd)), host(Qd)


def gpu_order(M, ws, D, dec, U, wait, arr, mw):
    N = len(dec)
    perm = torch.full((max(N, 1),), -1, dtype=torch.int32, device="cuda")
    seg = torch.full((D + 1,), -1, dtype=torch.int64, device="cuda")
    st = M.maps_order_local(D, dev(dec, np.int32), dev(U, np.int32), dev(wait, np.int32),
                            dev(arr, np.int32), mw, perm[:N], seg, ws=ws)
    assert st == 0
    return M.maps_check(ws), host(perm[:N]), host(seg)


# ---------------------------------------------------------------------------
# golden worked examples
# ---------------------------------------------------------------------------

def test_golden_worked_example(M, ws, golden):
    c = golden["calibration"]
    for case in c["cases"]:
        st, q, qd, _ = gpu_calibrate(M, ws, c["true_len"], c["pred_len"], case["alpha_ppm"])
        assert st == case["status"]
        if st == 0:
            assert q == qd == case["q"]
    m = c["misround_case"]
    assert gpu_calibrate(M, ws, m["true_len"], m["pred_len"], m["alpha_ppm"])[1] == m["q"]
    b = c["bound"]
    st, q, _, U = gpu_calibrate(M, ws, [9, 9, 9, 9, 9, 9, 9, 9, 13], [9] * 9, 100000, b["pred"])
    assert st == 0 and q == 4 and U.tolist() == b["U"]

    d, cd = golden["decoders"], golden["candidates"]
    st, K = gpu_occupancy(M, ws, 2, 8, d["res_off"], d["res_prompt"], d["res_gen"], d["res_bound"])
    assert st == 0 and K.tolist() == d["K"]
    res = (d["res_off"], d["res_prompt"], d["res_gen"], d["res_bound"])
    st, ch, hr, _, _ = gpu_dispatch(M, ws, 0, 2, 8, 1, d["K"], d["cap"], d["Q"], cd["prompt"], cd["bound"])
    assert st == 0 and ch.tolist() == golden["snapshot"]["choice"]
    assert hr.tolist() == golden["snapshot"]["headroom"]
    s = golden["sequential"]
    st, ch, hr, Ka, Qa = gpu_dispatch(M, ws, 1, 2, 8, 1, d["K"], d["cap"], d["Q"], cd["prompt"], cd["bound"])
    assert st == 0 and ch.tolist() == s["choice"] and hr.tolist() == s["headroom"]
    assert Ka.tolist() == s["K_after"] and Qa.tolist() == s["Q_after"]
    a = golden["alg1"]
    st, ch, hr, _, _ = gpu_dispatch(M, ws, 2, 2, 8, 1, None, d["cap"], d["Q"], cd["prompt"], cd["bound"], res)
    assert st == 0 and ch.tolist() == a["choice"] and hr.tolist() == a["headroom"]
    st, ch, hr, _, Qa = gpu_dispatch(M, ws, 3, 2, 8, 1, None, d["cap"], d["Q"], cd["prompt"], cd["bound"], res)
    assert st == 0 and ch.tolist() == a["sequential_choice"]
    assert hr.tolist() == a["sequential_headroom"] and Qa.tolist() == a["sequential_Q_after"]
    o = golden["order"]
    st, perm, seg = gpu_order(M, ws, 1, o["dec"], o["bound"], o["wait"], o["arrival"], o["max_wait"])
    assert st == 0 and perm.tolist() == o["perm"] and seg.tolist() == o["seg_off"]


# ---------------------------------------------------------------------------
# calibration
# ---------------------------------------------------------------------------

# one-block sizes: a bitonic sort up to 2,048 scores, a radix select up to
# 8,192; then the cooperative kernel
@pytest.mark.parametrize("n", [1, 2, 3, 9, 10, 1000, 1024, 1025, 2048, 2049, 4097, 65537, 1000003])
def test_calibrate_random(M, ws, oracle, n):
    rng = np.random.default_rng(n)
    L = rng.integers(-(2**31), 2**31, n, dtype=np.int64).astype(np.int32) if n % 2 else \
        rng.integers(0, 3000, n).astype(np.int32)
    P = rng.integers(-(2**31), 2**31, n, dtype=np.int64).astype(np.int32) if n % 3 == 0 else \
        rng.integers(0, 3000, n).astype(np.int32)
    if n > 10:
        P[: n // 4] = L[: n // 4]  # exact zeros
    query = rng.integers(0, 5000, 4099).astype(np.int32)
    for a in (1, 50000, 100000, 200000, 900000, 999999):
        sto, qo = oracle.calibrate(L, P, a)
        if sto == 0:  # the call also bounds the queries, which may overflow
            sto, Uo = oracle.bound(query, qo)
        st, q, qd, U = gpu_calibrate(M, ws, L, P, a, query)
        assert st == sto, (n, a)
        if st == 0:
            assert q == qd == qo
            assert np.array_equal(U, Uo)


def test_calibrate_unaligned_and_ranges(M, ws, oracle):
    rng = np.random.default_rng(3)
    L = rng.integers(0, 10**6, 10001).astype(np.int32)
    P = rng.integers(0, 10**6, 10001).astype(np.int32)
    Ld, Pd = dev(L), dev(P)
    qd = torch.zeros(1, dtype=torch.int32, device="cuda")
    st, q = M.maps_calibrate(Ld[1:], Pd[1:], 100000, q_dev_out=qd, q_host=True, ws=ws)
    assert st == 0 and q == oracle.calibrate(L[1:], P[1:], 100000)[1]
    # score above INT32_MAX -> range error
    st, _ = M.maps_calibrate(dev([I32_MAX] * 3, np.int32), dev([-5] * 3, np.int32), 500000,
                             q_host=True, ws=ws)
    assert st == M.MAPS_E_RANGE
    # bound above INT32_MAX -> range error
    U = torch.empty(1, dtype=torch.int32, device="cuda")
    st, _ = M.maps_calibrate(dev([10] * 3, np.int32), dev([0] * 3, np.int32), 500000,
                             dev([I32_MAX - 3], np.int32), U, q_host=True, ws=ws)
    assert st == M.MAPS_E_RANGE
    # rank above n: unbounded, returned at once
    assert gpu_calibrate(M, ws, [1] * 8, [0] * 8, 100000)[0] == M.MAPS_E_UNBOUNDED
    assert gpu_calibrate(M, ws, [], [], 100000)[0] == M.MAPS_E_UNBOUNDED
    assert M.maps_calibrate(Ld, Pd, 0, ws=ws)[0] == M.MAPS_E_INVALID


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_calibrate_grid_bucket_edges(M, ws, oracle, seed):
    """Grid form (n above the one-block limit): scores on the first pass's bin
    edges (the last exact bin, each leading-bit boundary, each 7-bit step) and
    up to 2^32 - 1, so that quantiles resolve after one, two or three passes and
    some lie above INT32_MAX (range error)."""
    rng = np.random.default_rng(seed)
    edges = {0, 1, 1022, 1023, 1024, 1025, 2**32 - 1}
    for e in range(10, 32):
        step = 1 << (e - 7)
        edges |= {(1 << e) - 1, 1 << e, (1 << e) + 1, (1 << e) + step - 1, (1 << e) + step}
    edges = np.array(sorted(edges), dtype=np.int64)
    n = 20011
    s = rng.choice(edges, n)
    s[: n // 3] = rng.integers(0, 2**32, n // 3, dtype=np.int64)  # full range
    P = np.full(n, -(2**31), dtype=np.int64)
    small = s < 2**31 - 5000
    P[small] = rng.integers(-2000, 2000, int(small.sum()))
    L, P = (P + s).astype(np.int32), P.astype(np.int32)
    assert np.array_equal(np.maximum(L.astype(np.int64) - P, 0), s)
    seen = set()
    for a in (1, 30, 1000, 100000, 333333, 500000, 700000, 900000, 999000, 999999):
        sto, qo = oracle.calibrate(L, P, a)
        st, q, qd, _ = gpu_calibrate(M, ws, L, P, a)
        assert st == sto, (seed, a)
        seen.add(st)
        if st == 0:
            assert q == qd == qo, (seed, a)
    assert {0, M.MAPS_E_RANGE} <= seen


@pytest.mark.parametrize("n,m,shift", [
    # more scores than the grid keeps in registers: every pass reads them again
    (1300007, 4099, 0),
    # more predictions than the grid keeps in registers, at an unaligned address
    (20011, 1300003, 1),
    # just past the one-block limit, no queries; then a ragged, unaligned few
    (8193, 0, 0), (10001, 777, 1)])
def test_calibrate_fused_register_limits(M, ws, oracle, n, m, shift):
    """Calibration sets above the one-block limit take one cooperative kernel;
    its scores and predictions live in registers up to eight per thread, else
    they are read from memory: q, the bounds and the status match the oracle
    either way."""
    rng = np.random.default_rng(n + m)
    L = rng.integers(0, 40000, n).astype(np.int32)
    P = rng.integers(0, 40000, n).astype(np.int32)
    P[: n // 5] = L[: n // 5]
    query = rng.integers(0, 70000, m + shift).astype(np.int32)
    Ld, Pd, Qd = dev(L), dev(P), dev(query)
    U = torch.full((m + shift + 1,), -9, dtype=torch.int32, device="cuda")
    qd = torch.zeros(1, dtype=torch.int32, device="cuda")
    for a in (1000, 100000, 999999):  # ranks within n at every size here
        sto, qo = oracle.calibrate(L, P, a)
        st, q = M.maps_calibrate(Ld, Pd, a, Qd[shift:] if m else None, U[shift:shift + m] if m else None,
                                 qd, q_host=True, ws=ws)
        assert st == sto == 0 and q == qo == int(host(qd)[0]), (n, m, a)
        if m:
            Uh = host(U)
            assert np.array_equal(Uh[shift:shift + m], oracle.bound(query[shift:], qo)[1])
            assert Uh[:shift].tolist() == [-9] * shift and Uh[shift + m] == -9
    # a bound above INT32_MAX: the range error, the others still bounded
    big = query[shift:].copy() if m else np.zeros(1, np.int32)
    big[-1] = I32_MAX - 3
    Ub = torch.empty(len(big), dtype=torch.int32, device="cuda")
    st, q = M.maps_calibrate(Ld, Pd, 100000, dev(big), Ub, q_host=True, ws=ws)
    assert st == M.MAPS_E_RANGE
    assert np.array_equal(host(Ub)[:-1], oracle.bound(big[:-1], oracle.calibrate(L, P, 100000)[1])[1])


@pytest.mark.parametrize("name", ["tiny", "d16", "d64", "large"])
def test_calibrate_workloads(M, ws, oracle, name):
    w = W.make(name)
    query = np.concatenate([w["res_pred"], w["cand_pred"]])
    for a in w["alphas_ppm"]:
        sto, qo = oracle.calibrate(w["cal_true"], w["cal_pred"], a)
        st, q, qd, U = gpu_calibrate(M, ws, w["cal_true"], w["cal_pred"], a, query)
        assert st == sto == 0 and q == qd == qo
        assert np.array_equal(U, oracle.bound(query, qo)[1])


# ---------------------------------------------------------------------------
# occupancy
# ---------------------------------------------------------------------------

def random_residents(rng, D, H, per_max, with_empty=True):
    R_per = rng.integers(0 if with_empty else 1, per_max + 1, D)
    off = np.concatenate([[0], np.cumsum(R_per)]).astype(np.int64)
    R = int(off[-1])
    p = rng.integers(0, 3000, R).astype(np.int32)
    g = rng.integers(0, 2 * H + 3, R).astype(np.int32)
    U = rng.integers(0, 3 * H + 5, R).astype(np.int32)
    return off, p, g, U


@pytest.mark.parametrize("D,H", [(1, 1), (3, 3), (2, 8), (5, 511), (4, 512), (3, 513), (7, 4095),
                                 (2, 4097), (9, 4100), (3, 12289), (2, 65536),
                                 # 64 horizon tiles (the most the bucketed form takes), then
                                 # more, which stream every resident per tile instead
                                 (2, 524288), (2, 524292), (1, 600001)])
def test_occupancy_random(M, ws, oracle, D, H):
    rng = np.random.default_rng(D * 100003 + H)
    off, p, g, U = random_residents(rng, D, H, 700)
    sto, Ko = oracle.occupancy(D, H, off, p, g, U)
    st, K, km = gpu_occupancy(M, ws, D, H, off, p, g, U, with_kmax=True)
    assert st == sto == 0
    assert np.array_equal(K, Ko)
    assert np.array_equal(km, kmax_of(Ko))


@pytest.mark.parametrize("name", ["tiny", "d16", "d64", "large"])
def test_occupancy_workloads(M, ws, oracle, name):
    w = W.make(name)
    q = oracle.calibrate(w["cal_true"], w["cal_pred"], w["alphas_ppm"][0])[1]
    U = oracle.bound(w["res_pred"], q)[1]
    sto, Ko = oracle.occupancy(w["D"], w["H"], w["res_off"], w["res_prompt"], w["res_gen"], U)
    st, K, km = gpu_occupancy(M, ws, w["D"], w["H"], w["res_off"], w["res_prompt"], w["res_gen"],
                              U, with_kmax=True)
    assert st == sto == 0
    assert np.array_equal(K, Ko)
    assert np.array_equal(km, kmax_of(Ko))


@pytest.mark.parametrize("D,H,per", [(2, 20000, 9000), (3, 3000, 4097)])
def test_occupancy_many_residents_per_decoder(M, ws, oracle, D, H, per):
    """More residents on one decoder than a block stages at once."""
    rng = np.random.default_rng(H + per)
    off = np.arange(D + 1, dtype=np.int64) * per
    R = D * per
    p = rng.integers(0, 300, R).astype(np.int32)
    g = rng.integers(0, H, R).astype(np.int32)
    U = rng.integers(0, 2 * H, R).astype(np.int32)
    sto, Ko = oracle.occupancy(D, H, off, p, g, U)
    st, K, km = gpu_occupancy(M, ws, D, H, off, p, g, U, with_kmax=True)
    assert st == sto == 0
    assert np.array_equal(K, Ko)
    assert np.array_equal(km, kmax_of(Ko))


def test_occupancy_errors(M, ws, oracle):
    # K above INT32_MAX
    big = I32_MAX // 2
    st, _ = gpu_occupancy(M, ws, 1, 4, [0, 2], [big, big], [0, 0], [4, 4])
    assert st == M.MAPS_E_RANGE == oracle.occupancy(1, 4, [0, 2], [big, big], [0, 0], [4, 4])[0]
    st, K = gpu_occupancy(M, ws, 1, 4, [0, 1], [I32_MAX - 4], [0], [4])
    assert st == 0 and K[0].tolist() == [I32_MAX - 3, I32_MAX - 2, I32_MAX - 1, I32_MAX]
    st, _ = gpu_occupancy(M, ws, 1, 8, [0, 1], [-1], [0], [3])
    assert st == M.MAPS_E_RANGE
    st, _ = gpu_occupancy(M, ws, 2, 8, [0, 2, 1], [1, 1], [0, 0], [3, 3])
    assert st == M.MAPS_E_RANGE
    st, _ = gpu_occupancy(M, ws, 1, 8, [0, 5], [1, 1], [0, 0], [3, 3])  # beyond R
    assert st == M.MAPS_E_RANGE
    K = torch.empty((1, 8), dtype=torch.int32, device="cuda")
    assert M.maps_project_occupancy(0, 8, dev([0], np.int64), dev([1], np.int32), dev([0], np.int32),
                                    dev([1], np.int32), K, ws=ws) == M.MAPS_E_INVALID


# ---------------------------------------------------------------------------
# dispatch
# ---------------------------------------------------------------------------

def diverse_caps(rng, K, spread):
    """Capacities straddling each decoder's occupancy so that the feasible set
    changes from candidate to candidate (test input built from the oracle)."""
    base = K[:, 0].astype(np.int64)
    off = rng.integers(-spread, spread // 2, K.shape[0])
    off[rng.integers(K.shape[0])] = spread // 2 - 1  # at least one roomy decoder
    return np.clip(base + off, 0, I32_MAX).astype(np.int32)


def check_dispatch(M, ws, oracle, mode, D, H, K, cap, Q, cp, cb, S=1, res=None):
    sto, co, ho, Ko, Qo = oracle.dispatch(mode, D, H, S, K, cap, Q, cp, cb,
                                          *(res if res is not None else ()))
    runs = [None, kmax_of(np.asarray(K))] if mode == 0 else [None]
    for km in runs:  # SNAPSHOT: summary derived inside, and passed in
        st, ch, hr, Ka, Qa = gpu_dispatch(M, ws, mode, D, H, S, K, cap, Q, cp, cb, res, km)
        assert st == sto
        if st == 0:
            assert np.array_equal(ch, co)
            assert np.array_equal(hr, ho)
            if mode == 1:
                assert np.array_equal(Ka, Ko)
            assert np.array_equal(Qa, Qo)
    return co, ho


@pytest.mark.parametrize("D,H,J", [(1, 1, 1), (1, 9, 33), (2, 8, 40), (3, 100, 700), (5, 511, 1000),
                                   (17, 4100, 3000), (64, 4096, 5000), (255, 1000, 3000),
                                   (256, 8192, 6000), (257, 2048, 2000), (300, 777, 1500),
                                   (1024, 1024, 2000),
                                   # 32-column tiles (129..256 decoders), copied by TMA and,
                                   # with H not a multiple of 4, by plain loads
                                   (129, 3000, 2000), (200, 1001, 2000)])
def test_dispatch_snapshot_random(M, ws, oracle, D, H, J):
    rng = np.random.default_rng(D * 7919 + H)
    off, p, g, U = random_residents(rng, D, H, 40)
    _, K = oracle.occupancy(D, H, off, p, g, U)
    cap = diverse_caps(rng, K, 4000)
    # tied queue lengths for even D, all distinct for odd D
    Q = (rng.integers(0, 4, D) if D % 2 == 0 else rng.permutation(D)).astype(np.int32)
    cp = rng.integers(0, 3000, J).astype(np.int32)
    cb = rng.integers(0, 2 * H + 2, J).astype(np.int32)
    co, ho = check_dispatch(M, ws, oracle, 0, D, H, K, cap, Q, cp, cb)
    if J >= 100:
        assert (ho >= 0).any() and (ho < 0).any()  # both branches exercised
        if D >= 8:
            assert len(set(co.tolist())) > 1


@pytest.mark.parametrize("name", ["tiny", "d16", "d64"])
@pytest.mark.parametrize("variant", ["given", "feasible", "diverse"])
def test_dispatch_snapshot_workloads(M, ws, oracle, name, variant):
    w = W.make(name, feasible=(variant == "feasible"))
    rng = np.random.default_rng(11)
    for a in w["alphas_ppm"]:
        q = oracle.calibrate(w["cal_true"], w["cal_pred"], a)[1]
        U = oracle.bound(w["res_pred"], q)[1]
        cb = oracle.bound(w["cand_pred"], q)[1]
        _, K = oracle.occupancy(w["D"], w["H"], w["res_off"], w["res_prompt"], w["res_gen"], U)
        cap, Q = w["cap"], w["Q"]
        if variant == "diverse":
            cap = diverse_caps(rng, K, 3000)
            Q = rng.integers(0, 3, w["D"]).astype(np.int32)
        check_dispatch(M, ws, oracle, 0, w["D"], w["H"], K, cap, Q, w["cand_prompt"], cb)


@pytest.mark.parametrize("variant", ["given", "feasible", "diverse"])
def test_dispatch_snapshot_large_full(M, ws, oracle, variant):
    """Full size, in the benchmark's launch configuration: every one of the
    65,536 candidates against the plain oracle (pinned to the by-definition
    one in test_oracle_tier_p.py), and a sample of them against the
    by-definition oracle itself."""
    w = W.make("large", feasible=(variant == "feasible"))
    D, H, J = w["D"], w["H"], w["J"]
    q = oracle.calibrate(w["cal_true"], w["cal_pred"], w["alphas_ppm"][0])[1]
    U = oracle.bound(w["res_pred"], q)[1]
    cb = oracle.bound(w["cand_pred"], q)[1]
    _, K = oracle.p_occupancy(D, H, w["res_off"], w["res_prompt"], w["res_gen"], U)
    cap, Q = w["cap"], w["Q"]
    rng = np.random.default_rng(5)
    if variant == "diverse":
        cap = diverse_caps(rng, K, 6000)
        Q = rng.integers(0, 3, D).astype(np.int32)
    st, ch, hr, _, _ = gpu_dispatch(M, ws, 0, D, H, 1, K, cap, Q, w["cand_prompt"], cb,
                                    kmax=kmax_of(K))
    stp, cp_, hp_ = oracle.p_dispatch_snapshot(D, H, K, cap, Q, w["cand_prompt"], cb)
    assert st == stp == 0
    assert np.array_equal(ch, cp_)
    assert np.array_equal(hr, hp_)
    st2, ch2, hr2, _, _ = gpu_dispatch(M, ws, 0, D, H, 1, K, cap, Q, w["cand_prompt"], cb)
    assert st2 == 0 and np.array_equal(ch, ch2) and np.array_equal(hr, hr2)
    idx = np.concatenate([np.argsort(cb)[-32:], rng.choice(J, 300, replace=False)])
    sto, co, ho, _, _ = oracle.dispatch(0, D, H, 1, K, cap, Q, w["cand_prompt"][idx], cb[idx])
    assert sto == 0
    assert np.array_equal(ch[idx], co)
    assert np.array_equal(hr[idx], ho)


@pytest.mark.parametrize("D,H,J", [(1, 5, 20), (2, 8, 50), (3, 100, 300), (7, 513, 400),
                                   (32, 2048, 256), (100, 1000, 300), (1024, 64, 100)])
def test_dispatch_sequential_random(M, ws, oracle, D, H, J):
    rng = np.random.default_rng(D * 31 + H)
    off, p, g, U = random_residents(rng, D, H, 30)
    _, K = oracle.occupancy(D, H, off, p, g, U)
    cap = diverse_caps(rng, K, 3000)
    Q = rng.integers(0, 3, D).astype(np.int32)
    cp = rng.integers(0, 500, J).astype(np.int32)
    cb = rng.integers(0, H + 5, J).astype(np.int32)
    check_dispatch(M, ws, oracle, 1, D, H, K, cap, Q, cp, cb)


@pytest.mark.parametrize("name", ["tiny", "d16", "d64"])
def test_dispatch_sequential_workloads(M, ws, oracle, name):
    w = W.make(name, feasible=True)
    q = oracle.calibrate(w["cal_true"], w["cal_pred"], w["alphas_ppm"][0])[1]
    U = oracle.bound(w["res_pred"], q)[1]
    cb = oracle.bound(w["cand_pred"], q)[1]
    _, K = oracle.occupancy(w["D"], w["H"], w["res_off"], w["res_prompt"], w["res_gen"], U)
    check_dispatch(M, ws, oracle, 1, w["D"], w["H"], K, w["cap"], w["Q"], w["cand_prompt"], cb)


@pytest.mark.parametrize("S", [1, 16])
@pytest.mark.parametrize("name", ["tiny", "d16", "d64", "large"])
def test_dispatch_alg1_workloads(M, ws, oracle, name, S):
    w = W.make(name, feasible=True)
    q = oracle.calibrate(w["cal_true"], w["cal_pred"], w["alphas_ppm"][0])[1]
    U = oracle.bound(w["res_pred"], q)[1]
    cb = oracle.bound(w["cand_pred"], q)[1]
    res = (w["res_off"], w["res_prompt"], w["res_gen"], U)
    rng = np.random.default_rng(S)
    cap = (w["cap"].astype(np.int64) // 2 + rng.integers(0, w["cap"].max() // 8, w["D"])).astype(np.int32)
    Q = rng.integers(0, 3, w["D"]).astype(np.int32)
    co, ho = check_dispatch(M, ws, oracle, 2, w["D"], w["H"], None, cap, Q, w["cand_prompt"], cb, S, res)
    # SEQUENTIAL over every candidate (65,536 reservations in order at Large)
    check_dispatch(M, ws, oracle, 3, w["D"], w["H"], None, cap, Q, w["cand_prompt"], cb, S, res)


def test_dispatch_errors(M, ws, oracle):
    K = np.zeros((2, 8), np.int32)
    st, ch, _, _, _ = gpu_dispatch(M, ws, 0, 2, 8, 1, K, [5, 5], [0, 0], [1, -1], [2, 2])
    assert st == M.MAPS_E_RANGE and ch[1] == -1
    K[1, 3] = -1
    assert gpu_dispatch(M, ws, 0, 2, 8, 1, K, [5, 5], [0, 0], [1], [2])[0] == M.MAPS_E_RANGE
    assert gpu_dispatch(M, ws, 1, 2, 8, 1, K, [5, 5], [0, 0], [1], [2])[0] == M.MAPS_E_RANGE
    assert gpu_dispatch(M, ws, 0, 2, 8, 1, np.zeros((2, 8), np.int32), [5, -5], [0, 0], [1], [2])[0] \
        == M.MAPS_E_RANGE
    ch = torch.empty(1, dtype=torch.int32, device="cuda")
    z = dev([0, 0], np.int32)
    Kd = dev(np.zeros((2, 8), np.int32))
    assert M.maps_dispatch(7, 2, 8, 1, Kd, z, z, dev([1], np.int32), dev([1], np.int32), ch,
                           ws=ws) == M.MAPS_E_INVALID
    assert M.maps_dispatch(0, 1025, 8, 1, Kd, z, z, dev([1], np.int32), dev([1], np.int32), ch,
                           ws=ws) == M.MAPS_E_INVALID
    small = M.Workspace(256)
    assert M.lib.maps_dispatch(0, 2, 8, 1, M._ptr(Kd), None, M._ptr(z), M._ptr(z), None, 0, None, None,
                               None, 1, M._ptr(dev([1], np.int32)), M._ptr(dev([1], np.int32)),
                               M._ptr(ch), None, small.ptr, 256, M._stream(None)) == M.MAPS_E_WORKSPACE


# ---------------------------------------------------------------------------
# local order
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("N,D,sorted_arrival", [(0, 3, True), (1, 1, True), (2, 2, False),
                                                (100, 3, False), (4096, 8, True), (4097, 8, False),
                                                (50000, 64, True), (50001, 300, False),
                                                (300000, 256, False), (1000, 70000, True),
                                                # one-block calls: bitonic up to 1,024
                                                # entries, then stable passes
                                                (700, 5, True), (1024, 16, False),
                                                (1025, 16, True), (3000, 40, False),
                                                # the one-block form at its decoder limit,
                                                # then past it
                                                (2000, 4096, True), (2000, 4097, True),
                                                # one decoder's queue at, and past, the most a
                                                # block sorts in shared memory
                                                (4608, 1, True), (4609, 1, True),
                                                (5632, 1, True), (5633, 1, True),
                                                (20000, 2, True), (300000, 256, True),
                                                # a queue of 22 chunks: five merge levels
                                                (100000, 1, True),
                                                # more decoders than the stable scatter takes
                                                (60000, 1500, True),
                                                # the bucketing pass at its decoder limit, and
                                                # with a count not a multiple of four
                                                (200000, 1024, True), (200000, 1023, False),
                                                # past 304 x 4,096 entries the bucketing blocks
                                                # take several rounds (loads issued twice);
                                                # arrival out of order: the global key pass
                                                (1500000, 256, True), (1500000, 1024, False)])
def test_order_random(M, ws, oracle, N, D, sorted_arrival):
    rng = np.random.default_rng(N + D)
    dec = rng.integers(0, D, N).astype(np.int32)
    U = rng.integers(0, 60 if N < 5000 else 2**31 - 1, N, dtype=np.int64).astype(np.int32)
    wait = rng.integers(-10, 3000, N).astype(np.int32)
    if sorted_arrival:
        arr = np.sort(rng.integers(0, max(N // 2, 1), N)).astype(np.int32)
    else:
        arr = rng.integers(0, 2**31 - 1, N, dtype=np.int64).astype(np.int32)
        arr[: N // 3] = rng.integers(0, 50, N // 3)  # ties on arrival too
    sto, po, so = oracle.order_local(D, dec, U, wait, arr, 1000)
    st, perm, seg = gpu_order(M, ws, D, dec, U, wait, arr, 1000)
    assert st == sto == 0
    assert np.array_equal(perm, po)
    assert np.array_equal(seg, so)


@pytest.mark.parametrize("N,D,ubits,abits", [
    # one-block calls with arrival out of index order: when (decoder, not
    # promoted, bound, arrival, index) fits 64 bits one sort on it gives the
    # order (bitonic, then stable passes), otherwise two sorts do
    (700, 5, 15, 20), (3000, 40, 15, 20), (1000, 1, 31, 31), (4000, 300, 31, 31),
    # exactly 64 bits, and one bit more
    (1024, 16, 18, 31), (1024, 16, 19, 31)])
def test_order_small_unsorted_key_widths(M, ws, oracle, N, D, ubits, abits):
    rng = np.random.default_rng(N + D + ubits)
    dec = rng.integers(0, D, N).astype(np.int32)
    U = rng.integers(0, 2**ubits, N, dtype=np.int64).astype(np.int32)
    wait = rng.integers(-10, 3000, N).astype(np.int32)
    i = rng.integers(0, N)
    U[i], wait[i] = 2**ubits - 1, 0  # the full width, on an entry that is not promoted
    arr = rng.integers(0, 2**abits, N, dtype=np.int64).astype(np.int32)
    arr[rng.integers(0, N)] = 2**abits - 1
    arr[: N // 4] = arr[N // 4]  # ties on arrival
    sto, po, so = oracle.order_local(D, dec, U, wait, arr, 1000)
    st, perm, seg = gpu_order(M, ws, D, dec, U, wait, arr, 1000)
    assert st == sto == 0
    assert np.array_equal(perm, po)
    assert np.array_equal(seg, so)


def test_order_bucketing_rounds_range_error(M, ws, oracle):
    """An entry outside the decoder domain in a call whose bucketing blocks
    take several rounds: counted and placed at decoder 0 in both of its
    passes, reported as MAPS_E_RANGE, every write inside the outputs."""
    rng = np.random.default_rng(5)
    N, D = 1300000, 64
    dec = rng.integers(0, D, N).astype(np.int32)
    dec[777777] = -3
    dec[1299999] = D + 5
    U = rng.integers(0, 5000, N).astype(np.int32)
    wait = rng.integers(0, 3000, N).astype(np.int32)
    arr = np.arange(N, dtype=np.int32)
    assert oracle.order_local(D, dec, U, wait, arr, 1000)[0] == -2
    st, perm, seg = gpu_order(M, ws, D, dec, U, wait, arr, 1000)
    assert st == M.MAPS_E_RANGE
    assert perm.min() >= -1 and perm.max() < N


@pytest.mark.parametrize("N,D,blo,bhi,skew", [
    # one queue far past a block (16 chunks), bounds of 17 bits
    (70000, 256, 0, 70000, 0.95),
    # several long queues with ragged last chunks, 31-bit bounds
    (60001, 8, 0, 2**31 - 1, 0.0),
    # bounds in [2^20, 2^20 + 200): keys share their high bits
    (30000, 3, 2**20, 2**20 + 200, 0.5),
    # more decoders than the stable scatter takes, one long queue
    (40000, 1100, 0, 2**31 - 1, 0.9),
    # every entry in one queue of 15 runs (ranked pairwise: 210 pairs)
    (65536, 256, 0, 70000, 1.0),
    # sixteen queues of about 16 runs each: the first to reserve their pairs within
    # the budget are ranked pairwise, the others merged level by level
    (1120000, 16, 0, 2**31 - 1, 0.0)])
def test_order_long_queues(M, ws, oracle, N, D, blo, bhi, skew):
    rng = np.random.default_rng(N + D)
    dec = rng.integers(0, D, N).astype(np.int32)
    dec[rng.random(N) < skew] = D // 2
    U = rng.integers(blo, bhi, N, dtype=np.int64).astype(np.int32)
    wait = rng.integers(-10, 3000, N).astype(np.int32)
    arr = np.sort(rng.integers(0, N, N)).astype(np.int32)
    sto, po, so = oracle.order_local(D, dec, U, wait, arr, 1000)
    st, perm, seg = gpu_order(M, ws, D, dec, U, wait, arr, 1000)
    assert st == sto == 0
    assert np.array_equal(perm, po)
    assert np.array_equal(seg, so)


def test_order_degenerate_keys(M, ws, oracle):
    # every key identical: all digit passes trivial -> identity order
    N = 9000
    z = np.zeros(N, np.int32)
    st, perm, seg = gpu_order(M, ws, 1, z, z, z, z, 5)
    assert st == 0 and np.array_equal(perm, np.arange(N)) and seg.tolist() == [0, N]
    st, perm, _ = gpu_order(M, ws, 2, [3], [1], [0], [0], 5)
    assert st == M.MAPS_E_RANGE


@pytest.mark.parametrize("name,one_queue", [("d64", False), ("large", False), ("large", True)])
def test_order_workload_pipeline(M, ws, oracle, name, one_queue):
    """The benchmark's order step: residents plus dispatched candidates (spread over the
    decoders, or all on one decoder as when every candidate falls back to the same one)."""
    w = W.make(name)
    R, J, D = w["R"], w["J"], w["D"]
    rng = np.random.default_rng(1)
    q = oracle.calibrate(w["cal_true"], w["cal_pred"], w["alphas_ppm"][0])[1]
    U = oracle.bound(np.concatenate([w["res_pred"], w["cand_pred"]]), q)[1]
    cand_dec = np.full(J, 37, np.int32) if one_queue else rng.integers(0, D, J).astype(np.int32)
    dec = np.concatenate([w["res_dec"], cand_dec])
    wait = np.concatenate([w["res_wait"], np.zeros(J, np.int32)])
    arr = np.arange(R + J, dtype=np.int32)
    sto, po, so = oracle.order_local(D, dec, U, wait, arr, w["max_wait"])
    st, perm, seg = gpu_order(M, ws, D, dec, U, wait, arr, w["max_wait"])
    assert st == sto == 0
    assert np.array_equal(perm, po) and np.array_equal(seg, so)


def test_dispatch_snapshot_invalid_candidates(M, ws, oracle):
    """Candidates with a negative prompt or bound get choice -1 and headroom 0
    and record MAPS_E_RANGE; the others are still decided."""
    w = W.make("tiny", feasible=True)
    D, H = w["D"], w["H"]
    q = oracle.calibrate(w["cal_true"], w["cal_pred"], w["alphas_ppm"][0])[1]
    U = oracle.bound(w["res_pred"], q)[1]
    cb = oracle.bound(w["cand_pred"], q)[1].copy()
    cp = w["cand_prompt"].copy()
    cp[3], cb[7] = -1, -5
    _, K = oracle.occupancy(D, H, w["res_off"], w["res_prompt"], w["res_gen"], U)
    st, ch, hr, _, _ = gpu_dispatch(M, ws, M.MODE_SNAPSHOT, D, H, 1, K, w["cap"], w["Q"], cp, cb)
    sto, cho, hro, _, _ = oracle.dispatch(0, D, H, 1, K, w["cap"], w["Q"], cp, cb)
    assert st == sto == M.MAPS_E_RANGE
    assert np.array_equal(ch, cho) and np.array_equal(hr, hro)


def test_dispatch_kmax_checked_against_K(M, ws, oracle):
    """A caller's 16-step summary is compared with K at four blocks of every
    row: the summary of K itself passes, one that disagrees with K in the first
    block of a row is MAPS_E_INVALID."""
    w = W.make("d16", feasible=True)
    D, H = w["D"], w["H"]
    q = oracle.calibrate(w["cal_true"], w["cal_pred"], w["alphas_ppm"][0])[1]
    U = oracle.bound(w["res_pred"], q)[1]
    cb = oracle.bound(w["cand_pred"], q)[1]
    _, K = oracle.occupancy(D, H, w["res_off"], w["res_prompt"], w["res_gen"], U)
    km = kmax_of(K)
    st, ch, hr, _, _ = gpu_dispatch(M, ws, M.MODE_SNAPSHOT, D, H, 1, K, w["cap"], w["Q"],
                                    w["cand_prompt"], cb, kmax=km)
    _, cho, hro, _, _ = oracle.dispatch(0, D, H, 1, K, w["cap"], w["Q"], w["cand_prompt"], cb)
    assert st == 0 and np.array_equal(ch, cho) and np.array_equal(hr, hro)
    bad = km.copy()
    bad[5, 0] += 1
    st, _, _, _, _ = gpu_dispatch(M, ws, M.MODE_SNAPSHOT, D, H, 1, K, w["cap"], w["Q"],
                                  w["cand_prompt"], cb, kmax=bad)
    assert st == M.MAPS_E_INVALID


def test_dispatch_scoring_events(M, ws, oracle):
    """The benchmarking hook records its events around the scoring kernel and
    leaves the decisions unchanged."""
    w = W.make("tiny", feasible=True)
    q = oracle.calibrate(w["cal_true"], w["cal_pred"], w["alphas_ppm"][0])[1]
    U = oracle.bound(w["res_pred"], q)[1]
    cb = oracle.bound(w["cand_pred"], q)[1]
    _, K = oracle.occupancy(w["D"], w["H"], w["res_off"], w["res_prompt"], w["res_gen"], U)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    e1.record()
    assert M.maps_set_dispatch_events(e0, e1) == 0
    try:
        st, ch, hr, _, _ = gpu_dispatch(M, ws, 0, w["D"], w["H"], 1, K, w["cap"], w["Q"],
                                        w["cand_prompt"], cb)
    finally:
        M.maps_set_dispatch_events(None, None)
    torch.cuda.synchronize()
    _, cho, hro, _, _ = oracle.dispatch(0, w["D"], w["H"], 1, K, w["cap"], w["Q"],
                                        w["cand_prompt"], cb)
    assert st == 0 and np.array_equal(ch, cho) and np.array_equal(hr, hro)
    assert e0.elapsed_time(e1) > 0.0


# ---------------------------------------------------------------------------
# CUDA graph capture of the whole pass
# ---------------------------------------------------------------------------

def test_graph_capture_replay(M, oracle):
    """The four calls (calibrate + bound, occupancy, SNAPSHOT dispatch, local
    order) captured once in a CUDA graph: every replay reads the inputs as they
    are then and matches the oracle, including after the inputs change."""
    w0, w1 = W.make("tiny", feasible=True), W.make("tiny", seed=11)
    D, H, R, J = w0["D"], w0["H"], w0["R"], w0["J"]
    assert (D, H, R, J) == (w1["D"], w1["H"], w1["R"], w1["J"])
    a = w0["alphas_ppm"][0]
    n = len(w0["cal_true"])
    z = lambda k, dt=torch.int32: torch.zeros(k, dtype=dt, device="cuda")  # noqa: E731
    x = dict(cal_true=z(n), cal_pred=z(n), pred=z(R + J), off=z(D + 1, torch.int64), prompt=z(R),
             gen=z(R), cap=z(D), Q=z(D), cprompt=z(J), dec=z(R + J), wait=z(R + J),
             arr=torch.arange(R + J, dtype=torch.int32, device="cuda"))
    U, q = z(R + J), z(1)
    K = z(D * H).view(D, H)
    km = torch.zeros(M.kmax_shape(D, H), dtype=torch.int32, device="cuda")
    hr, perm, seg = z(J, torch.int64), z(R + J), z(D + 1, torch.int64)
    need = max(M.lib.maps_calibrate_workspace_size(n, R + J),
               M.lib.maps_project_occupancy_workspace_size(D, H, R),
               M.lib.maps_dispatch_workspace_size(M.MODE_SNAPSHOT, D, H, J),
               M.lib.maps_order_local_workspace_size(R + J, D))
    gws = M.Workspace(need, torch.device("cuda"))

    def load(w):
        for k, v in dict(cal_true=w["cal_true"], cal_pred=w["cal_pred"],
                         pred=np.concatenate([w["res_pred"], w["cand_pred"]]), off=w["res_off"],
                         prompt=w["res_prompt"], gen=w["res_gen"], cap=w["cap"], Q=w["Q"],
                         cprompt=w["cand_prompt"], wait=np.concatenate([w["res_wait"], np.zeros(J)]),
                         dec=np.concatenate([w["res_dec"], np.zeros(J)])).items():
            x[k].copy_(torch.from_numpy(np.ascontiguousarray(v).astype(x[k].cpu().numpy().dtype)))

    def run():
        assert M.maps_calibrate(x["cal_true"], x["cal_pred"], a, x["pred"], U, q, ws=gws)[0] == 0
        assert M.maps_project_occupancy(D, H, x["off"], x["prompt"], x["gen"], U[:R], K, km,
                                        ws=gws) == 0
        assert M.maps_dispatch(M.MODE_SNAPSHOT, D, H, 1, K, x["cap"], x["Q"], x["cprompt"],
                               U[R:], x["dec"][R:], hr, kmax=km, ws=gws) == 0
        assert M.maps_order_local(D, x["dec"], U, x["wait"], x["arr"], w0["max_wait"], perm, seg,
                                  ws=gws) == 0

    load(w0)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        run()  # warm-up outside the capture
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side, capture_error_mode="relaxed"):
        run()
    for w in (w0, w1, w0):
        load(w)
        g.replay()
        torch.cuda.synchronize()
        assert M.maps_check(gws) == 0
        sto, qo = oracle.calibrate(w["cal_true"], w["cal_pred"], a)
        Uo = oracle.bound(np.concatenate([w["res_pred"], w["cand_pred"]]), qo)[1]
        _, Ko = oracle.occupancy(D, H, w["res_off"], w["res_prompt"], w["res_gen"], Uo[:R])
        _, cho, hro, _, _ = oracle.dispatch(0, D, H, 1, Ko, w["cap"], w["Q"], w["cand_prompt"],
                                            Uo[R:])
        deco = np.concatenate([w["res_dec"], cho]).astype(np.int32)
        _, po, so = oracle.order_local(D, deco, Uo, np.concatenate([w["res_wait"], np.zeros(J, np.int32)]),
                                       np.arange(R + J, dtype=np.int32), w0["max_wait"])
        assert int(host(q)[0]) == qo and np.array_equal(host(U), Uo)
        assert np.array_equal(host(K), Ko)
        assert np.array_equal(host(x["dec"])[R:], cho) and np.array_equal(host(hr), hro)
        assert np.array_equal(host(perm), po) and np.array_equal(host(seg), so)


# ---------------------------------------------------------------------------
# determinism
# ---------------------------------------------------------------------------

def test_repeat_runs_identical(M, ws, oracle):
    w = W.make("d64")
    q = oracle.calibrate(w["cal_true"], w["cal_pred"], 100000)[1]
    U = oracle.bound(w["res_pred"], q)[1]
    cb = oracle.bound(w["cand_pred"], q)[1]
    outs = []
    for _ in range(3):
        _, K = gpu_occupancy(M, ws, w["D"], w["H"], w["res_off"], w["res_prompt"], w["res_gen"], U)
        _, ch, hr, _, _ = gpu_dispatch(M, ws, 0, w["D"], w["H"], 1, K, w["cap"], w["Q"],
                                       w["cand_prompt"], cb)
        outs.append((K, ch, hr))
    for o in outs[1:]:
        assert all(np.array_equal(x, y) for x, y in zip(o, outs[0]))


# ---------------------------------------------------------------------------
# streaming loop
# ---------------------------------------------------------------------------

def gpu_stream(M, ws, N, D, H, cap, B, Wn, a, mw, arrival, prompt, true, pred):
    nb = (N + B - 1) // B
    ch = torch.full((N,), -9, dtype=torch.int32, device="cuda")
    q = torch.full((nb,), -9, dtype=torch.int32, device="cuda")
    stats = torch.full((nb, 4), -9, dtype=torch.int64, device="cuda")
    cfg = M.stream_cfg(N, D, H, cap, B, Wn, a, mw)
    st = M.maps_stream_run(cfg, dev(arrival[:N], np.int64), dev(prompt[:N], np.int32),
                           dev(true[:N], np.int32), dev(pred[:N], np.int32), ch, q, stats, ws=ws)
    return st, host(ch), host(q), host(stats)


def check_stream(M, ws, oracle, N, D, H, cap, B, Wn, a, mw, w):
    args = (N, D, H, cap, B, Wn, a, mw, w["arrival_ms"], w["prompt"], w["true"], w["pred"])
    sto, cho, qo, so = oracle.stream(*args)
    st, ch, q, s = gpu_stream(M, ws, *args)
    assert st == sto
    if st == 0:
        assert np.array_equal(q, qo)
        assert np.array_equal(s, so)
        assert np.array_equal(ch, cho)
    return qo, so


def test_stream_golden(M, ws, stream_golden):
    c, r = stream_golden["config"], stream_golden["requests"]
    st, ch, q, s = gpu_stream(M, ws, c["N"], c["D"], c["H"], c["cap"], c["batch"], c["window"],
                              c["alpha_ppm"], c["max_wait"], np.array(r["arrival_ms"]),
                              np.array(r["prompt"]), np.array(r["true_len"]), np.array(r["pred"]))
    assert st == 0
    assert ch.tolist() == stream_golden["choice"]
    assert q.tolist() == stream_golden["q"]
    assert s.tolist() == stream_golden["stats"]


@pytest.mark.parametrize("N,D,H,cap,B,Wn,a,mw", [
    (1, 32, 16384, 262144, 256, 500, 100000, 1000),       # one request, round robin
    (300, 32, 16384, 262144, 256, 500, 100000, 1000),     # ragged last batch
    (20000, 32, 16384, 262144, 256, 500, 100000, 1000),   # the streaming workload's prefix
    (20000, 4, 4096, 12000, 256, 500, 100000, 1000),      # queues back up and block
    (20000, 3, 2048, 9000, 100, 37, 300000, 50),          # promotions, small window
    (5000, 5, 1000, 20000, 33, 7, 500000, 0),             # horizon below many bounds
    # capacity far below demand: waiting queues push M, and the deficits,
    # past 2^21 (the dispatch's 64-bit key comparison)
    (3000, 8, 16384, 3000, 256, 500, 100000, 1000),
    # 200 decoders x batches of 256: the end-step tables would need about 800 KB of
    # shared memory, so the loop dispatches through the dense projection instead
    (3000, 200, 2048, 60000, 256, 300, 100000, 1000),
    # 48 decoders: the shared-memory walk past one warp's decoders, with queues
    (4000, 48, 4096, 30000, 64, 200, 100000, 1000),
    # a window of 10,000 completions: once it holds more than 8,192 the quantile is
    # taken by the cooperative calibration kernel inside the loop
    (30000, 8, 16384, 262144, 512, 10000, 100000, 1000),
])
def test_stream_prefix(M, ws, oracle, N, D, H, cap, B, Wn, a, mw):
    w = W.make_stream(n_requests=N)
    qo, so = check_stream(M, ws, oracle, N, D, H, cap, B, Wn, a, mw, w)
    assert (qo >= 0).any() or N < 1000


def test_stream_full_workload(M, ws, oracle):
    """All 1,000,000 requests of the streaming workload, bit for bit."""
    w = W.make_stream()
    c = W.WORKLOADS["stream"]
    qo, so = check_stream(M, ws, oracle, w["N"], w["D"], w["H"], w["cap"], w["batch"],
                          w["window"], w["alpha_ppm"], w["max_wait"], w)
    assert len(qo) == (w["N"] + c["batch"] - 1) // c["batch"]
