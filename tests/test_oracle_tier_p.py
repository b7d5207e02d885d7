"""Pins of the plain (tier P) oracle, oracle_p.cpp.

Tier P computes the same integers as the by-definition oracle (oracle.c) by
another route: a selection instead of a full sort, an end-step count and one
pass down the horizon instead of adding every footprint to every step, prefix
maxima instead of a maximum per (candidate, decoder) pair, grouping by decoder
instead of one comparison sort.  So each check below compares two independent
implementations, on the hand-derived worked example, on the benchmark
workloads (a candidate sample on the largest ones) and on random tiny
instances with their error cases, and checks that the thread count does not
change a result.
"""
import numpy as np
import pytest

from paper_2609_15359_gb300 import workloads as W


def test_tier_p_worked_example(oracle, golden):
    c = golden["calibration"]
    for case in c["cases"]:
        st, q = oracle.p_calibrate(c["true_len"], c["pred_len"], case["alpha_ppm"])
        if case["q"] is None:
            assert st == -3  # unbounded: the rank exceeds n
        else:
            assert st == 0 and q == case["q"]
    d = golden["decoders"]
    st, K = oracle.p_occupancy(d["D"], d["H"], d["res_off"], d["res_prompt"], d["res_gen"],
                               d["res_bound"])
    assert st == 0 and K.tolist() == d["K"]
    cands, snap = golden["candidates"], golden["snapshot"]
    st, ch, hr = oracle.p_dispatch_snapshot(d["D"], d["H"], K, d["cap"], d["Q"],
                                            cands["prompt"], cands["bound"])
    assert st == 0 and ch.tolist() == snap["choice"] and hr.tolist() == snap["headroom"]
    r = golden["order"]
    st, perm, seg = oracle.p_order_local(r["D"], r["dec"], r["bound"], r["wait"], r["arrival"],
                                         r["max_wait"])
    assert st == 0 and perm.tolist() == r["perm"] and seg.tolist() == r["seg_off"]


@pytest.mark.parametrize("name", ["tiny", "d16", "d64"])
@pytest.mark.parametrize("feasible", [False, True])
def test_tier_p_equals_tier_b_on_workloads(oracle, name, feasible):
    w = W.make(name, feasible=feasible)
    D, H = w["D"], w["H"]
    for a in w["alphas_ppm"]:
        stb, qb = oracle.calibrate(w["cal_true"], w["cal_pred"], a)
        stp, qp = oracle.p_calibrate(w["cal_true"], w["cal_pred"], a)
        assert stb == stp == 0 and qb == qp
        pred = np.concatenate([w["res_pred"], w["cand_pred"]])
        _, Ub = oracle.bound(pred, qb)
        _, Up = oracle.p_bound(pred, qp)
        assert np.array_equal(Ub, Up)
        R = w["R"]
        stb, Kb = oracle.occupancy(D, H, w["res_off"], w["res_prompt"], w["res_gen"], Ub[:R])
        stp, Kp = oracle.p_occupancy(D, H, w["res_off"], w["res_prompt"], w["res_gen"], Up[:R])
        assert stb == stp == 0 and np.array_equal(Kb, Kp)
        cp, cb = w["cand_prompt"], Ub[R:]
        if len(cp) > 2000:  # the by-definition scores are O(J * D * H): a sample
            idx = np.random.default_rng(D).choice(len(cp), 2000, replace=False)
            cp, cb = cp[idx], cb[idx]
        stb, chb, hrb, _, _ = oracle.dispatch(0, D, H, 1, Kb, w["cap"], w["Q"], cp, cb)
        stp, chp, hrp = oracle.p_dispatch_snapshot(D, H, Kp, w["cap"], w["Q"], cp, cb)
        assert stb == stp == 0
        assert np.array_equal(chb, chp) and np.array_equal(hrb, hrp)
        dec = np.concatenate([w["res_dec"], chb if len(chb) == w["J"] else
                              np.resize(chb, w["J"]).astype(np.int32)])
        wait = np.concatenate([w["res_wait"], np.zeros(w["J"], np.int32)])
        arr = np.arange(R + w["J"], dtype=np.int32)
        stb, pb, sb = oracle.order_local(D, dec, Ub, wait, arr, w["max_wait"])
        stp, pp, sp = oracle.p_order_local(D, dec, Up, wait, arr, w["max_wait"])
        assert stb == stp == 0 and np.array_equal(pb, pp) and np.array_equal(sb, sp)


def test_tier_p_equals_tier_b_on_random_tiny_instances(oracle):
    rng = np.random.default_rng(2024)
    for it in range(10_000):
        n = int(rng.integers(0, 40))
        L = rng.integers(0, 60, n).astype(np.int32)
        P = rng.integers(0, 60, n).astype(np.int32)
        a = int(rng.integers(1, 10**6))
        stb, qb = oracle.calibrate(L, P, a)
        stp, qp = oracle.p_calibrate(L, P, a)
        assert stb == stp and (stb != 0 or qb == qp), (it, stb, stp)
        D, H = int(rng.integers(1, 6)), int(rng.integers(1, 40))
        per = rng.integers(0, 6, D)
        off = np.concatenate([[0], np.cumsum(per)]).astype(np.int64)
        R = int(off[-1])
        p = rng.integers(0, 30, R).astype(np.int32)
        g = rng.integers(0, 2 * H + 2, R).astype(np.int32)
        U = rng.integers(0, 3 * H + 2, R).astype(np.int32)
        if R and it % 10 == 0:
            [p, g, U][it % 3][int(rng.integers(0, R))] = -1  # a length outside the domain
        stb, Kb = oracle.occupancy(D, H, off, p, g, U)
        stp, Kp = oracle.p_occupancy(D, H, off, p, g, U)
        assert stb == stp, it
        if stb == 0:
            assert np.array_equal(Kb, Kp), it
            J = int(rng.integers(0, 12))
            cp = rng.integers(0, 50, J).astype(np.int32)
            cb = rng.integers(0, 2 * H + 3, J).astype(np.int32)
            if J and it % 7 == 0:
                cb[0] = -2
            cap = (Kb.max(axis=1) + rng.integers(-40, 80, D)).clip(0).astype(np.int32)
            Q = rng.integers(0, 3, D).astype(np.int32)
            stb, chb, hrb, _, _ = oracle.dispatch(0, D, H, 1, Kb, cap, Q, cp, cb)
            stp, chp, hrp = oracle.p_dispatch_snapshot(D, H, Kp, cap, Q, cp, cb)
            assert stb == stp and np.array_equal(chb, chp) and np.array_equal(hrb, hrp), it
        N = int(rng.integers(0, 30))
        dec = rng.integers(0, D, N).astype(np.int32)
        bnd = rng.integers(0, 8, N).astype(np.int32)
        wait = rng.integers(0, 6, N).astype(np.int32)
        arr = rng.integers(0, 10, N).astype(np.int32)
        if N and it % 11 == 0:
            dec[0] = D  # a decoder outside the domain
        stb, pb, sb = oracle.order_local(D, dec, bnd, wait, arr, 2)
        stp, pp, sp = oracle.p_order_local(D, dec, bnd, wait, arr, 2)
        assert stb == stp, it
        if stb == 0:
            assert np.array_equal(pb, pp) and np.array_equal(sb, sp), it


def test_tier_p_results_do_not_depend_on_threads(oracle):
    w = W.make("d16")
    q = oracle.p_calibrate(w["cal_true"], w["cal_pred"], w["alphas_ppm"][0])[1]
    U = oracle.p_bound(np.concatenate([w["res_pred"], w["cand_pred"]]), q)[1]
    out = []
    for th in (1, 4):
        oracle.p_threads(th)
        _, K = oracle.p_occupancy(w["D"], w["H"], w["res_off"], w["res_prompt"], w["res_gen"],
                                  U[:w["R"]])
        _, ch, hr = oracle.p_dispatch_snapshot(w["D"], w["H"], K, w["cap"], w["Q"],
                                               w["cand_prompt"], U[w["R"]:])
        dec = np.concatenate([w["res_dec"], ch])
        wait = np.concatenate([w["res_wait"], np.zeros(w["J"], np.int32)])
        _, perm, _ = oracle.p_order_local(w["D"], dec, U, wait,
                                          np.arange(len(dec), dtype=np.int32), w["max_wait"])
        out.append((K, ch, hr, perm))
    oracle.p_threads(1)
    for a, b in zip(out[0], out[1]):
        assert np.array_equal(a, b)
