"""Pins of the streaming-loop oracle's policy variants: the Sec. 4 ablations
(MQ->MC, SJF->FCFS), the round-robin and least-requests baselines, the App. C
reservation accountings, and the per-decoder statistics.

Each pin holds by the policies' definitions, independently of the oracle's
code: round robin is i mod D; least requests reduces to round robin while
every request stays in the system; MC and MAPS agree when no decoder is ever
feasible (both take the most headroom); SJF and FCFS agree when every bound
is equal (SJF breaks ties by arrival, and promotion keeps arrival order); a
hand-worked two-request case separates the three accountings; the per-decoder
sums equal the per-batch totals.
"""
import numpy as np
import pytest

from paper_2609_15359_gb300 import workloads as W


def run(oracle, w, n, **kw):
    cfg = dict(N=n, D=w["D"], H=w["H"], cap=w["cap"], batch=w["batch"], window=w["window"],
               alpha_ppm=w["alpha_ppm"], max_wait=w["max_wait"])
    cfg.update({k: kw.pop(k) for k in list(kw) if k in cfg})
    return oracle.stream(cfg["N"], cfg["D"], cfg["H"], cfg["cap"], cfg["batch"], cfg["window"],
                         cfg["alpha_ppm"], cfg["max_wait"], w["arrival_ms"], w["prompt"],
                         w["true"], w["pred"], with_dec_stats=True, **kw)


@pytest.fixture(scope="module")
def w():
    return W.make_stream(n_requests=30000)


def test_round_robin_baseline(oracle, w):
    st, ch, q, stats, ds = run(oracle, w, 20000, dispatch=oracle.DISPATCH_RR)
    assert st == 0 and np.array_equal(ch, np.arange(20000) % w["D"])
    assert ds[:, 2].sum() == stats[:, 1].sum()


def test_least_requests_is_round_robin_while_nothing_completes(oracle, w):
    n = 3000
    long = dict(w, true=np.full(len(w["true"]), 10**6, np.int32))  # nobody completes
    assert w["arrival_ms"][n - 1] < 10**6
    st_l, ch_l, *_ = run(oracle, long, n, dispatch=oracle.DISPATCH_LR)
    assert st_l == 0 and np.array_equal(ch_l, np.arange(n) % w["D"])


def test_mc_equals_maps_when_nothing_is_feasible(oracle, w):
    # capacity 1: no decoder is ever feasible and nothing is ever admitted
    a = run(oracle, w, 8000, cap=1)
    b = run(oracle, w, 8000, cap=1, dispatch=oracle.DISPATCH_MC)
    assert a[0] == b[0] == 0 and np.array_equal(a[1], b[1]) and np.array_equal(a[3], b[3])
    # with room to spare the two rules differ
    c = run(oracle, w, 8000, dispatch=oracle.DISPATCH_MC)
    d = run(oracle, w, 8000)
    assert not np.array_equal(c[1], d[1])


def test_fcfs_equals_sjf_when_every_bound_is_equal(oracle, w):
    same = dict(w, pred=np.full(len(w["pred"]), 200, np.int32))
    a = run(oracle, same, 10000, cap=10000)
    b = run(oracle, same, 10000, cap=10000, local=oracle.LOCAL_FCFS)
    assert a[0] == b[0] == 0
    for x, y in zip(a[1:], b[1:]):
        assert np.array_equal(x, y)
    # with different bounds the local order matters
    c = run(oracle, w, 10000, cap=10000)
    d = run(oracle, w, 10000, cap=10000, local=oracle.LOCAL_FCFS)
    assert not np.array_equal(c[3], d[3])


@pytest.mark.parametrize("cap,admitted", [(260, [1, 0, 0]), (290, [1, 1, 0]), (400, [1, 1, 1])])
def test_accountings_on_a_hand_worked_case(oracle, cap, admitted):
    """One decoder, batches of one.  A (p 100, true 50, pred 40) arrives at
    step 0 and is admitted at once (the quantile is still unbounded, so the
    bound is the prediction).  B (the same) arrives at step 10, when A has 10
    tokens: admission counts A as 110 tokens (occupancy), 100 + max(40, 10) =
    140 (staged release), or 100 + 100 + 40 = 240 (held), and B needs
    100 + 40 = 140."""
    for acc, want in zip((oracle.ACCOUNT_OCCUPANCY, oracle.ACCOUNT_STAGED, oracle.ACCOUNT_HELD),
                         admitted):
        st, ch, q, stats = oracle.stream(2, 1, 64, cap, 1, 4, 100000, 1000, np.array([0, 10]),
                                         np.array([100, 100]), np.array([50, 50]),
                                         np.array([40, 40]), accounting=acc)
        assert st == 0 and q.tolist() == [-1, -1]
        assert stats[0].tolist() == [0, 1, 0, 0]
        assert stats[1, 1] == want and stats[1, 2] == 1 - want


@pytest.mark.parametrize("dispatch,local,acc", [(0, 0, 0), (1, 0, 1), (2, 1, 2), (3, 0, 0),
                                                (0, 1, 2)])
def test_per_decoder_statistics_sum_to_the_batch_totals(oracle, w, dispatch, local, acc):
    n = 20000
    st, ch, q, stats, ds = run(oracle, w, n, cap=10000, dispatch=dispatch, local=local,
                               accounting=acc)
    assert st == 0 and ch.min() >= 0 and ch.max() < w["D"]
    assert ds[:, 2].sum() == stats[:, 1].sum()   # admissions
    assert ds[:, 1].sum() == stats[:, 3].sum()   # over-capacity events
    B = w["batch"]
    s = w["arrival_ms"][np.minimum(np.arange(1, stats.shape[0] + 1) * B, n) - 1]
    span = np.append(np.diff(s), 0)
    assert ds[:, 0].sum() == (stats[:, 2] * span).sum()  # waiting x steps
    assert (ds >= 0).all()
