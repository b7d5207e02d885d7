"""Pins of the App. A round-robin KV-pressure oracle (oracle_rr.c).

Each pin comes from somewhere other than the oracle: the processor-sharing
completion formula for requests that arrive together (a textbook closed form,
and with integer lengths the token rounds reach it exactly), the FIFO capacity
gate that serialises requests too large to share a decoder, round-robin
routing when nothing contends, the high-pressure interval definition on
cases whose occupancy is known in advance, and conservation invariants.
"""
import numpy as np
import pytest

TOK = 1000          # t_tok = 1 ms in microseconds
THETA = 850000      # theta = 0.85


def ps_closed_form(t0, lengths):
    """Completion times of k requests that start together on one processor-
    sharing server of rate one token per TOK: sorted l_1 <= ... <= l_k, the
    i-th completes at t0 + TOK * (l_1 + ... + l_i + (k - i) * l_i)."""
    order = np.argsort(lengths, kind="stable")
    ls = np.asarray(lengths)[order]
    k = len(ls)
    done = np.empty(k, dtype=np.int64)
    acc = 0
    for i in range(k):
        acc += int(ls[i])
        done[order[i]] = t0 + TOK * (acc + (k - 1 - i) * int(ls[i]))
    return done


def test_single_request(oracle):
    st, a, d, s, ts = oracle.rr_pressure(4, 50000, TOK, THETA, [5], [45000], [7])
    assert st == 0 and a.tolist() == [5] and d.tolist() == [5 + 7 * TOK] and ts == 7 * TOK
    # footprint 45,007 >= 0.85 * 50,000: one high-pressure interval, the whole run
    assert s[0].tolist() == [7 * TOK, 7 * TOK, 1, 1, 0, 0]
    assert s[1:].sum() == 0


@pytest.mark.parametrize("seed", range(6))
def test_processor_sharing_closed_form(oracle, seed):
    rng = np.random.default_rng(seed)
    k = int(rng.integers(1, 40))
    lengths = rng.integers(1, 300, k)
    t0 = int(rng.integers(0, 10**6))
    # one decoder, everything arrives at t0 and fits: pure processor sharing
    st, a, d, s, ts = oracle.rr_pressure(1, 10**9, TOK, THETA, np.full(k, t0),
                                         np.zeros(k), lengths)
    assert st == 0 and (a == t0).all()
    assert np.array_equal(d, ps_closed_form(t0, lengths))
    assert ts == d.max() - t0 and s[0, 3] == k


def test_fifo_gate_serialises_large_requests(oracle):
    # every request needs 0.6 C: one at a time, in arrival order
    C, k = 100000, 5
    lengths = np.array([30, 10, 50, 20, 40])
    prompt = 60000 - lengths
    st, a, d, s, ts = oracle.rr_pressure(1, C, TOK, THETA, np.zeros(k), prompt, lengths)
    assert st == 0
    ends = np.cumsum(lengths) * TOK
    assert np.array_equal(d, ends) and np.array_equal(a, np.concatenate([[0], ends[:-1]]))
    # all arrive at 0, the first is admitted at once: k - 1 wait at the last arrival
    assert s[0, 4] == k - 1 and s[0, 5] == a.sum()
    assert s[0, 0] == 0 and s[0, 2] == 0  # 0.6 < 0.85: never under pressure
    # 0.9 C each: the decoder stays above the threshold through every hand-over
    prompt9 = 90000 - lengths
    st, a, d, s, ts = oracle.rr_pressure(1, C, TOK, THETA, np.zeros(k), prompt9, lengths)
    assert st == 0 and s[0, 0] == ends[-1] and s[0, 1] == ends[-1] and s[0, 2] == 1


def test_round_robin_routing_without_contention(oracle):
    rng = np.random.default_rng(3)
    N, n = 4, 40
    arr = np.arange(n) * 10**7  # far apart: every request runs alone
    lengths = rng.integers(1, 100, n)
    st, a, d, s, ts = oracle.rr_pressure(N, 50000, TOK, THETA, arr, np.full(n, 100), lengths)
    assert st == 0 and np.array_equal(a, arr) and np.array_equal(d, arr + lengths * TOK)
    assert s[:, 3].tolist() == [n // N] * N  # request i on decoder i mod N
    assert (s[:, 0] == 0).all() and (s[:, 4] == 0).all() and (s[:, 5] == 0).all()


def test_light_load_never_reaches_the_threshold(oracle):
    rng = np.random.default_rng(5)
    n = 2000
    arr = np.cumsum(rng.integers(0, 5000, n))
    st, a, d, s, ts = oracle.rr_pressure(4, 50000, TOK, THETA, arr, rng.integers(1, 100, n),
                                         rng.integers(1, 50, n))
    assert st == 0 and (s[:, 0] == 0).all() and (s[:, 2] == 0).all()
    assert s[:, 3].sum() == n


@pytest.mark.parametrize("rho", [0.8, 1.0, 1.1])
def test_conservation_and_metric_invariants(oracle, rho):
    rng = np.random.default_rng(int(rho * 10))
    N, C, n = 4, 50000, 3000
    out = np.clip(np.rint(rng.lognormal(5.5, 1.0, n)), 1, 8192).astype(np.int64)
    prompt = rng.integers(32, 2049, n)
    lam = rho * N / (out.mean() * TOK * 1e-6)  # requests per second
    arr = np.rint(np.cumsum(rng.exponential(1.0, n)) * 1e6 / lam).astype(np.int64)
    st, a, d, s, ts = oracle.rr_pressure(N, C, TOK, THETA, arr, prompt, out)
    assert st == 0
    assert s[:, 3].sum() == n                       # every request completes
    assert (a >= arr).all() and (d >= a + out * TOK).all()
    for dd in range(N):
        idx = np.arange(dd, n, N)
        assert (np.diff(a[idx]) >= 0).all()         # FIFO: admitted in arrival order
        assert s[dd, 5] == (a[idx] - arr[idx]).sum()
    assert ts == d.max() - arr[0]
    assert (s[:, 0] <= ts).all() and (s[:, 1] <= s[:, 0]).all()
    assert ((s[:, 2] > 0) == (s[:, 0] > 0)).all()


def test_domain(oracle):
    # a footprint above C can never be admitted; out_len < 1; decreasing arrival
    assert oracle.rr_pressure(1, 100, TOK, THETA, [0], [60], [41])[0] == -2
    assert oracle.rr_pressure(1, 100, TOK, THETA, [0], [6], [0])[0] == -2
    assert oracle.rr_pressure(2, 100, TOK, THETA, [5, 4], [6, 6], [1, 1])[0] == -2
    assert oracle.rr_pressure(0, 100, TOK, THETA, [0], [6], [1])[0] == -1
