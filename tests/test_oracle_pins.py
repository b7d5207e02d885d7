"""Pins of the CPU oracle against what the paper and mathematics fix.

None of these compares the oracle with itself: each check goes through an
independent route (exact rational arithmetic, numpy's sort / lexsort, closed
forms of special cases, invariants, brute-force placement with
re-projection, the conformal coverage theorem, hand-derived goldens).
"""
from fractions import Fraction
import math

import numpy as np
import pytest

from paper_2609_15359_gb300 import workloads as W

I32_MAX = 2**31 - 1


# --------------------------------------------------------------------------
# A1 / A2: calibration (Sec. 3.2)
# --------------------------------------------------------------------------

def exact_rank(n, alpha_ppm):
    """ceil((1 - alpha)(n + 1)) in exact rational arithmetic."""
    return math.ceil((1 - Fraction(alpha_ppm, 10**6)) * (n + 1))


def test_rank_matches_exact_rational(oracle):
    rng = np.random.default_rng(1)
    cases = [(9, 700000), (9, 200000), (9, 100000), (9, 50000), (0, 100000),
             (499, 100000), (10**6, 100000), (10**12, 1), (10**12, 999999)]
    cases += [(int(n), int(a)) for n, a in zip(rng.integers(0, 10**7, 300),
                                               rng.integers(1, 10**6, 300))]
    for n, a in cases:
        assert oracle.rank(n, a) == exact_rank(n, a), (n, a)


def test_calibration_golden(oracle, golden):
    c = golden["calibration"]
    s = np.maximum(0, np.array(c["true_len"]) - np.array(c["pred_len"]))
    assert s.tolist() == c["scores"]
    for case in c["cases"]:
        assert oracle.rank(len(s), case["alpha_ppm"]) == case["rank"]
        st, q = oracle.calibrate(c["true_len"], c["pred_len"], case["alpha_ppm"])
        assert st == case["status"]
        if st == 0:
            assert q == case["q"]
    m = c["misround_case"]
    # the naive floating-point rank would be 4 here
    assert math.ceil((1 - 0.7) * 10) == 4
    assert oracle.rank(9, m["alpha_ppm"]) == m["rank"]
    assert oracle.calibrate(m["true_len"], m["pred_len"], m["alpha_ppm"]) == (0, m["q"])
    b = c["bound"]
    st, U = oracle.bound(b["pred"], b["q"])
    assert st == 0 and U.tolist() == b["U"]


@pytest.mark.parametrize("n", [1, 2, 9, 10, 57, 500, 4096, 100000])
def test_quantile_is_sorted_order_statistic(oracle, n):
    rng = np.random.default_rng(n)
    L = rng.integers(-50, 2000, n).astype(np.int32)
    P = rng.integers(-50, 2000, n).astype(np.int32)
    if n > 20:
        P[: n // 3] = L[: n // 3] + 7  # many exact zeros and duplicates
    s = np.maximum(0, L.astype(np.int64) - P)
    for a in (1, 50000, 100000, 200000, 500000, 900000, 999999):
        k = exact_rank(n, a)
        st, q = oracle.calibrate(L, P, a)
        if k > n:
            assert st == -3
            continue
        assert st == 0
        assert q == np.sort(s)[k - 1]
        # order-statistic definition of the k-th smallest
        assert np.count_nonzero(s <= q) >= k
        assert np.count_nonzero(s < q) < k


@pytest.mark.parametrize("seed", [0, 1])
def test_quantile_full_int32_range(oracle, seed):
    """Scores of full-range int32 lengths reach 2^32 - 1 (the difference of two
    int32 values clamped at 0).  The quantile is still the k-th smallest of them
    (numpy's sort in int64), and a quantile above INT32_MAX cannot be an int32
    bound: MAPS_E_RANGE."""
    rng = np.random.default_rng(100 + seed)
    n = 3001
    L = rng.integers(-(2**31), 2**31, n, dtype=np.int64)
    P = rng.integers(-(2**31), 2**31, n, dtype=np.int64)
    # powers of two and their neighbours among the scores
    e = rng.integers(0, 32, n // 3)
    P[: n // 3] = -(2**31)
    L[: n // 3] = np.minimum(P[: n // 3] + (1 << e) + rng.integers(-1, 2, n // 3), 2**31 - 1)
    L, P = L.astype(np.int32), P.astype(np.int32)
    s = np.maximum(0, L.astype(np.int64) - P)
    assert s.max() > 2**31  # some scores above INT32_MAX
    seen = set()
    for a in (1000, 100000, 300000, 500000, 700000, 900000, 999000):
        k = exact_rank(n, a)
        st, q = oracle.calibrate(L, P, a)
        want = np.sort(s)[k - 1]
        if want > 2**31 - 1:
            assert st == -2, a
        else:
            assert st == 0 and q == want, a
        seen.add(st)
    assert seen == {0, -2}


def test_calibration_unbounded_and_invalid(oracle):
    e = np.zeros(0, np.int32)
    assert oracle.calibrate(e, e, 100000)[0] == -3  # n = 0: rank 1 > 0
    # n < ceil((1-alpha)/alpha) -> rank exceeds n
    L = np.arange(8, dtype=np.int32)
    assert oracle.calibrate(L, L, 100000)[0] == -3
    assert oracle.calibrate(np.arange(9, dtype=np.int32), np.zeros(9, np.int32),
                            100000) == (0, 8)
    assert oracle.calibrate(L, L, 0)[0] == -1
    assert oracle.calibrate(L, L, 10**6)[0] == -1


def test_coverage_theorem_on_held_out_residuals(oracle):
    """Sec. 3.2: P(L <= Lhat + q) >= 1 - alpha under exchangeability.  With
    continuous positive scores (ties only at 0, below the quantile) the
    coverage of one exchangeable test point is exactly k/(n+1)."""
    rng = np.random.default_rng(2024)
    n, a, draws, tests = 99, 100000, 600, 200
    k = exact_rank(n, a)
    cov = np.empty(draws)
    for d in range(draws):
        L = np.rint(rng.lognormal(12.0, 1.0, n + tests)).astype(np.int32)
        P = np.rint(L * np.exp(rng.normal(0, 0.4, n + tests))).astype(np.int32)
        st, q = oracle.calibrate(L[:n], P[:n], a)
        assert st == 0
        st, U = oracle.bound(P[n:], q)
        assert st == 0
        cov[d] = np.mean(L[n:] <= U)
    se = cov.std(ddof=1) / math.sqrt(draws)
    target = k / (n + 1)
    assert cov.mean() >= 1 - a / 1e6 - 4 * se
    assert abs(cov.mean() - target) <= 4 * se, (cov.mean(), target, se)


def test_bound_closed_form_and_range(oracle):
    pred = np.array([0, 1, 5, 1000, I32_MAX - 10], np.int32)
    st, U = oracle.bound(pred[:4], 7)
    assert st == 0 and U.tolist() == [7, 8, 12, 1007]
    st, _ = oracle.bound(pred, 11)
    assert st == -2


# --------------------------------------------------------------------------
# A3 / A4: projected occupancy
# --------------------------------------------------------------------------

def _end_and_base(H, p, g, U):
    e = np.clip(U.astype(np.int64) - g, 1, H)
    b = p.astype(np.int64) + g + 1
    return e, b


def test_occupancy_golden(oracle, golden):
    d = golden["decoders"]
    st, K = oracle.occupancy(d["D"], d["H"], d["res_off"], d["res_prompt"],
                             d["res_gen"], d["res_bound"])
    assert st == 0 and K.tolist() == d["K"]


def test_single_resident_ramp_closed_form(oracle):
    """One resident on an empty decoder: the footprint ramp p+g+1+t for the
    steps it is live; with g = 0 and U <= H the last value is p + U, the
    footprint M(r) = L_p + L_out of Eq. (kv_demand)."""
    rng = np.random.default_rng(5)
    for _ in range(300):
        H = int(rng.integers(1, 64))
        p, g, U = (int(x) for x in rng.integers(0, 80, 3))
        st, K = oracle.occupancy(1, H, [0, 1], [p], [g], [U])
        assert st == 0
        live = [t for t in range(H) if K[0, t] != 0]
        e = len(live)
        assert live == list(range(e))  # live on a prefix of the horizon
        assert e == min(max(U - g, 1), H)
        assert K[0, 0] == p + g + 1
        assert np.all(np.diff(K[0, :e]) == 1)
        assert K[0].sum() == e * (p + g + 1) + e * (e - 1) // 2
        if g == 0 and 1 <= U <= H:
            assert K[0].max() == p + U


@pytest.mark.parametrize("name", ["tiny", "d16"])
def test_occupancy_mass_first_step_and_linearity(oracle, name):
    w = W.make(name)
    D, H = w["D"], w["H"]
    st, q = oracle.calibrate(w["cal_true"], w["cal_pred"], w["alphas_ppm"][0])
    U = w["res_pred"].astype(np.int64) + q
    p, g = w["res_prompt"], w["res_gen"]
    st, K = oracle.occupancy(D, H, w["res_off"], p, g, U)
    assert st == 0
    e, b = _end_and_base(H, p, g, U)
    off = w["res_off"]
    for k in range(D):
        sl = slice(off[k], off[k + 1])
        # total token-steps: closed-form sum of each resident's ramp
        assert K[k].sum() == np.sum(e[sl] * b[sl] + e[sl] * (e[sl] - 1) // 2)
        # every resident is live at t = 0
        assert K[k, 0] == b[sl].sum()
        # after the last end step nothing is left
        assert np.all(K[k, int(e[sl].max()):] == 0)
    # linearity: occupancy of a union is the sum of the parts
    half = np.zeros(len(p), bool)
    half[::2] = True
    offA = np.concatenate([[0], np.cumsum([half[off[k]:off[k + 1]].sum() for k in range(D)])])
    offB = np.concatenate([[0], np.cumsum([(~half[off[k]:off[k + 1]]).sum() for k in range(D)])])
    stA, KA = oracle.occupancy(D, H, offA, p[half], g[half], U[half])
    stB, KB = oracle.occupancy(D, H, offB, p[~half], g[~half], U[~half])
    assert stA == stB == 0
    assert np.array_equal(KA.astype(np.int64) + KB, K)
    # sampled cells by the per-cell sum definition agree
    rng = np.random.default_rng(3)
    for _ in range(50):
        k, t = int(rng.integers(D)), int(rng.integers(H))
        assert oracle.occupancy_cell(H, off, k, t, p, g, U) == K[k, t]


def test_occupancy_domain_and_range(oracle):
    assert oracle.occupancy(1, 8, [0, 1], [-1], [0], [3])[0] == -2
    assert oracle.occupancy(1, 8, [0, 1], [1], [0], [-3])[0] == -2
    assert oracle.occupancy(2, 8, [0, 2, 1], [1, 1], [0, 0], [3, 3])[0] == -2
    big = I32_MAX // 2
    assert oracle.occupancy(1, 4, [0, 2], [big, big], [0, 0], [4, 4])[0] == -2
    st, K = oracle.occupancy(1, 4, [0, 1], [I32_MAX - 4], [0], [4])
    assert st == 0 and K[0].tolist() == [I32_MAX - 3, I32_MAX - 2, I32_MAX - 1, I32_MAX]
    assert oracle.occupancy(1, 4, [0, 1], [I32_MAX - 3], [0], [4])[0] == -2


# --------------------------------------------------------------------------
# A5 / A6 / A7: dispatch (Sec. 3.3, Alg. 1)
# --------------------------------------------------------------------------

def test_dispatch_golden(oracle, golden):
    d, c = golden["decoders"], golden["candidates"]
    K = np.array(d["K"], np.int32)
    res = (d["res_off"], d["res_prompt"], d["res_gen"], d["res_bound"])
    st, ch, hr, Ka, Qa = oracle.dispatch(0, 2, 8, 1, K, d["cap"], d["Q"],
                                         c["prompt"], c["bound"], *res)
    assert st == 0 and ch.tolist() == golden["snapshot"]["choice"]
    assert hr.tolist() == golden["snapshot"]["headroom"]
    assert np.array_equal(Ka, K) and Qa.tolist() == d["Q"]
    s = golden["sequential"]
    st, ch, hr, Ka, Qa = oracle.dispatch(1, 2, 8, 1, K, d["cap"], d["Q"],
                                         c["prompt"], c["bound"], *res)
    assert st == 0 and ch.tolist() == s["choice"] and hr.tolist() == s["headroom"]
    assert Ka.tolist() == s["K_after"] and Qa.tolist() == s["Q_after"]
    a = golden["alg1"]
    st, ch, hr, _, _ = oracle.dispatch(2, 2, 8, a["S"], None, d["cap"], d["Q"],
                                       c["prompt"], c["bound"], *res)
    assert st == 0 and ch.tolist() == a["choice"] and hr.tolist() == a["headroom"]
    st, ch, hr, _, Qa = oracle.dispatch(3, 2, 8, a["S"], None, d["cap"], d["Q"],
                                        c["prompt"], c["bound"], *res)
    assert st == 0 and ch.tolist() == a["sequential_choice"]
    assert hr.tolist() == a["sequential_headroom"]
    assert Qa.tolist() == a["sequential_Q_after"]


def _rule(keys_feasible, h):
    """Reference selection: lowest Q among h >= 0, else highest h; ties to
    the lowest decoder index (Alg. 1)."""
    feas = [k for k in range(len(h)) if h[k] >= 0]
    if feas:
        return min(feas, key=lambda k: (keys_feasible[k], k))
    return min(range(len(h)), key=lambda k: (-h[k], k))


def test_dispatch_empty_decoders_reduce_to_admission_test(oracle):
    """With no residents and H >= U the peak is p + U = M(r) (Eq. kv_demand)
    and feasibility is the admission test K + M(r) <= C of Eq. (admission)
    with K = 0."""
    rng = np.random.default_rng(11)
    for _ in range(200):
        D = int(rng.integers(1, 9))
        H = 256
        cap = rng.integers(0, 400, D).astype(np.int32)
        Q = rng.integers(0, 4, D).astype(np.int32)
        J = int(rng.integers(1, 20))
        cp = rng.integers(0, 200, J).astype(np.int32)
        cb = rng.integers(1, H + 1, J).astype(np.int32)
        K = np.zeros((D, H), np.int32)
        st, ch, hr, _, _ = oracle.dispatch(0, D, H, 1, K, cap, Q, cp, cb)
        assert st == 0
        for j in range(J):
            h = cap.astype(np.int64) - (int(cp[j]) + int(cb[j]))
            k = _rule(Q, h)
            assert ch[j] == k and hr[j] == h[k]


def _tiny_instance(rng, D, H):
    R_per = rng.integers(0, 4, D)
    off = np.concatenate([[0], np.cumsum(R_per)]).astype(np.int64)
    R = int(off[-1])
    p = rng.integers(0, 12, R).astype(np.int32)
    g = rng.integers(0, 6, R).astype(np.int32)
    U = rng.integers(0, H + 4, R).astype(np.int32)
    cap = rng.integers(0, 120, D).astype(np.int32)
    Q = rng.integers(0, 3, D).astype(np.int32)
    return off, p, g, U, cap, Q


def _with_extra(off, p, g, U, k, pj, Uj):
    """Resident arrays with one more resident (pj, g=0, Uj) on decoder k."""
    pos = int(off[k + 1])
    off2 = off.copy()
    off2[k + 1:] += 1
    return (off2, np.insert(p, pos, pj), np.insert(g, pos, 0),
            np.insert(U, pos, Uj))


def test_dispatch_snapshot_by_placement_enumeration(oracle):
    """Brute force over placements: put the candidate on each decoder as a
    fresh resident, re-project that decoder's occupancy, take its peak over
    the candidate's live steps, and apply the rule."""
    rng = np.random.default_rng(7)
    for _ in range(150):
        D, H = int(rng.integers(1, 5)), int(rng.integers(1, 24))
        off, p, g, U, cap, Q = _tiny_instance(rng, D, H)
        st, K = oracle.occupancy(D, H, off, p, g, U)
        assert st == 0
        J = int(rng.integers(1, 6))
        cp = rng.integers(0, 12, J).astype(np.int32)
        cb = rng.integers(0, H + 4, J).astype(np.int32)
        st, ch, hr, _, _ = oracle.dispatch(0, D, H, 1, K, cap, Q, cp, cb)
        assert st == 0
        for j in range(J):
            u = min(max(int(cb[j]), 1), H)
            h = []
            for k in range(D):
                o2, p2, g2, U2 = _with_extra(off, p, g, U, k, cp[j], cb[j])
                st2, K2 = oracle.occupancy(D, H, o2, p2, g2, U2)
                assert st2 == 0
                h.append(int(cap[k]) - int(K2[k, :u].max()))
            k = _rule(Q, h)
            assert ch[j] == k and hr[j] == h[k]


def test_dispatch_sequential_equals_reprojection(oracle):
    """Sec. 3.3 reservation: after each commit the state equals the
    re-projection of residents plus every committed candidate, and each
    choice is the snapshot choice against that state."""
    rng = np.random.default_rng(9)
    for _ in range(100):
        D, H = int(rng.integers(1, 5)), int(rng.integers(1, 24))
        off, p, g, U, cap, Q = _tiny_instance(rng, D, H)
        st, K = oracle.occupancy(D, H, off, p, g, U)
        J = int(rng.integers(1, 7))
        cp = rng.integers(0, 12, J).astype(np.int32)
        cb = rng.integers(0, H + 4, J).astype(np.int32)
        st, ch, hr, Ka, Qa = oracle.dispatch(1, D, H, 1, K, cap, Q, cp, cb)
        assert st == 0
        o2, p2, g2, U2, Q2 = off, p, g, U, Q.copy()
        for j in range(J):
            st1, K1 = oracle.occupancy(D, H, o2, p2, g2, U2)
            st1, c1, h1, _, _ = oracle.dispatch(0, D, H, 1, K1, cap, Q2,
                                                cp[j:j + 1], cb[j:j + 1])
            assert c1[0] == ch[j] and h1[0] == hr[j]
            o2, p2, g2, U2 = _with_extra(o2, p2, g2, U2, int(ch[j]), cp[j], cb[j])
            Q2[ch[j]] += 1
        st1, Kf = oracle.occupancy(D, H, o2, p2, g2, U2)
        assert np.array_equal(Ka, Kf) and np.array_equal(Qa, Q2)


def test_alg1_feasible_implies_horizon_feasible(oracle):
    """A decoder that Algorithm 1 deems feasible (block budget covers the
    demand) is also feasible in the horizon form, for any block size."""
    rng = np.random.default_rng(13)
    checked = 0
    for _ in range(200):
        D = int(rng.integers(1, 5))
        H = 64
        off, p, g, U, cap, Q = _tiny_instance(rng, D, H - 8)
        cap = (cap * 2).astype(np.int32)
        S = int(rng.choice([1, 2, 16]))
        st, K = oracle.occupancy(D, H, off, p, g, U)
        J = 4
        cp = rng.integers(0, 12, J).astype(np.int32)
        cb = rng.integers(0, H, J).astype(np.int32)
        for k in range(D):
            sl = slice(off[k], off[k + 1])
            o1 = np.array([0, off[k + 1] - off[k]])
            st, _, h_alg, _, _ = oracle.dispatch(2, 1, H, S, None, cap[k:k + 1],
                                                 Q[k:k + 1], cp, cb, o1, p[sl],
                                                 g[sl], U[sl])
            st2, _, h_hor, _, _ = oracle.dispatch(0, 1, H, 1, K[k:k + 1],
                                                  cap[k:k + 1], Q[k:k + 1], cp, cb)
            assert st == st2 == 0
            for j in range(J):
                if h_alg[j] >= 0:
                    checked += 1
                    assert h_hor[j] >= 0
    assert checked > 50


def test_alg1_block_rounding_example(oracle):
    """Eq. (feasibility) with S = 16: B_need = ceil((p+U)/16); B_eff =
    floor(C/16) - sum ceil((p + max(U, g+1))/16).  Worked by hand:
    decoder 0 C=100 -> 6 blocks; resident (p=17, g=3, U=2) holds
    ceil((17+4)/16) = 2 -> B_eff = 4.  Decoder 1 C=64 -> 4 blocks, empty.
    Candidate (p=30, U=33): need ceil(63/16) = 4 -> both feasible -> min Q.
    Candidate (p=30, U=35): need ceil(65/16) = 5 -> none -> argmax B_eff =
    d0 (4 == 4, lowest index), headroom -1."""
    st, ch, hr, _, Qa = oracle.dispatch(2, 2, 8, 16, None, [100, 64], [3, 1],
                                        [30, 30], [33, 35], [0, 1, 1], [17],
                                        [3], [2])
    assert st == 0 and ch.tolist() == [1, 0] and hr.tolist() == [0, -1]


# --------------------------------------------------------------------------
# A8: local order
# --------------------------------------------------------------------------

def test_order_golden(oracle, golden):
    o = golden["order"]
    st, perm, seg = oracle.order_local(o["D"], o["dec"], o["bound"], o["wait"],
                                       o["arrival"], o["max_wait"])
    assert st == 0 and perm.tolist() == o["perm"] and seg.tolist() == o["seg_off"]
    assert [o["ids"][i] for i in perm] == o["order_ids"]


@pytest.mark.parametrize("N,D", [(1, 1), (17, 3), (1000, 8), (50000, 64)])
def test_order_matches_lexsort(oracle, N, D):
    rng = np.random.default_rng(N)
    dec = rng.integers(0, D, N).astype(np.int32)
    U = rng.integers(0, 40, N).astype(np.int32)
    wait = rng.integers(-5, 3000, N).astype(np.int32)
    arr = rng.integers(0, max(2, N // 2), N).astype(np.int32)
    mw = 1000
    st, perm, seg = oracle.order_local(D, dec, U, wait, arr, mw)
    assert st == 0
    prom = wait > mw
    prim = np.where(prom, arr, U)
    idx = np.arange(N)
    ref = np.lexsort((idx, arr, prim, ~prom, dec))
    assert np.array_equal(perm, ref)
    assert np.array_equal(seg, np.concatenate([[0], np.cumsum(np.bincount(dec, minlength=D))]))


def test_order_domain(oracle):
    assert oracle.order_local(2, [2], [1], [0], [0], 10)[0] == -2
    assert oracle.order_local(2, [0], [-1], [0], [0], 10)[0] == -2
    assert oracle.order_local(2, [0], [1], [0], [-1], 10)[0] == -2
    st, perm, seg = oracle.order_local(3, [], [], [], [], 10)
    assert st == 0 and seg.tolist() == [0, 0, 0, 0]


# --------------------------------------------------------------------------
# A9: streaming loop
# --------------------------------------------------------------------------

def test_stream_golden(oracle, stream_golden):
    c, r = stream_golden["config"], stream_golden["requests"]
    st, ch, q, stats = oracle.stream(c["N"], c["D"], c["H"], c["cap"], c["batch"],
                                     c["window"], c["alpha_ppm"], c["max_wait"],
                                     np.array(r["arrival_ms"]), np.array(r["prompt"]),
                                     np.array(r["true_len"]), np.array(r["pred"]))
    assert st == 0
    assert ch.tolist() == stream_golden["choice"]
    assert q.tolist() == stream_golden["q"]
    assert stats.tolist() == stream_golden["stats"]


@pytest.mark.parametrize("Wn,a", [(500, 100000), (20, 100000), (7, 500000)])
def test_stream_unconstrained_closed_form(oracle, Wn, a):
    """With capacity and horizon large enough that every request fits, all
    queues drain at every batch: each bounded batch is dispatched by min-Q
    with the per-commit reservation (Q += 1), i.e. cyclically from decoder 0,
    and unbounded batches round-robin on the arrival index.  Every request
    runs from its batch's step for exactly its true length, so the window at
    each batch is the last `window` requests completed by then, ordered by
    (completion step, id), and q is their conformal quantile."""
    w = W.make_stream(n_requests=30000)
    N, D, B = 30000, 32, 256
    H, cap = 16384, 2**30
    st, ch, q, stats = oracle.stream(N, D, H, cap, B, Wn, a, 1000,
                                     w["arrival_ms"], w["prompt"], w["true"], w["pred"])
    assert st == 0
    nb = (N + B - 1) // B
    bidx = np.arange(N) // B
    s = w["arrival_ms"][np.minimum((np.arange(nb) + 1) * B, N) - 1]
    comp = s[bidx] + w["true"]
    ids = np.arange(N)
    n_rr = 0
    for b in range(nb):
        lo, hi = b * B, min(N, (b + 1) * B)
        elig = ids[(bidx < b) & (comp <= s[b])]
        order = np.lexsort((elig, comp[elig]))
        win = elig[order][-Wn:]
        k = exact_rank(len(win), a)
        if k > len(win):
            assert q[b] == -1
            assert np.array_equal(ch[lo:hi], ids[lo:hi] % D)
            n_rr += 1
        else:
            sc = np.maximum(0, w["true"][win].astype(np.int64) - w["pred"][win])
            assert q[b] == np.sort(sc)[k - 1]
            assert np.array_equal(ch[lo:hi], np.arange(hi - lo) % D)
        assert stats[b, 2] == 0 and stats[b, 3] == 0
    assert 0 < n_rr < nb
    assert stats[:, 1].sum() == N


def test_stream_conservation_under_pressure(oracle):
    """Tight capacity: requests wait and block; counts must still balance."""
    w = W.make_stream(n_requests=20000)
    N, D, B = 20000, 4, 256
    st, ch, q, stats = oracle.stream(N, D, 4096, 12000, B, 500, 100000, 1000,
                                     w["arrival_ms"], w["prompt"], w["true"], w["pred"])
    assert st == 0
    assert ch.min() >= 0 and ch.max() < D
    admitted = np.cumsum(stats[:, 1])
    completed = np.cumsum(stats[:, 0])
    dispatched = np.minimum((np.arange(len(q)) + 1) * B, N)
    waiting = dispatched - admitted
    assert np.array_equal(waiting, stats[:, 2])
    assert np.all(completed <= admitted)
    assert stats[:, 2].max() > 0  # the queues did back up
