"""Pins of the streaming loop's fidelity modes in the oracle: per-step
admission with preemption, and the deferral of a request until its bound is
available with the round-robin timeout beta (Sec. 3.3, memory-aware
scheduler; App. D).

Each pin is a hand-traced case or a property the model's definition fixes:
with capacity to spare, per-step admission changes nothing; a reservation
that covers every true length (staged accounting, predictions exact) never
preempts; zero prediction delays make the deferral a no-op; beta = 0 with
late predictions sends everything round robin; the sums of the per-decoder
statistics equal the per-batch totals.
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
                         w["true"], w.get("pred_override", w["pred"]), with_dec_stats=True, **kw)


@pytest.fixture(scope="module")
def w():
    return W.make_stream(n_requests=20000)


def tiny(oracle, arr, p, true, pred, cap, D=1, per_step=1, beta=-1, delay=None, acc=0):
    return oracle.stream(len(arr), D, 64, cap, 1, 4, 100000, 1000, np.array(arr), np.array(p),
                         np.array(true), np.array(pred), accounting=acc, with_dec_stats=True,
                         per_step=per_step, beta=beta, pred_delay=None if delay is None else
                         np.array(delay))


def test_preemption_hand_trace(oracle):
    """One decoder of capacity 40, batches of one, the quantile unbounded
    throughout (U = prediction).  A (p 10, true 50, pred 5) is admitted at
    step 0; B (p 10, true 20, pred 5) at step 3 (13 + 15 <= 40).  At step t
    the two hold 20 + (t - 1) + (t - 4) tokens before taking one each, which
    passes 40 at t = 12: B, the later admitted, is preempted and re-admitted
    at once (22 + 15 <= 40); at t = 17 the pair would hold 42 and B is
    preempted again, and now 27 + 15 > 40 keeps it waiting until A completes
    at step 50.  B then runs steps 51..70.  C (step 100) drives the loop to
    step 100.  B waits through steps 17..49: 33 request-steps."""
    st, ch, q, stats, ds = tiny(oracle, [0, 3, 100], [10, 10, 1], [50, 20, 1], [5, 5, 1], 40)
    assert st == 0 and ch.tolist() == [0, 0, 0] and q.tolist() == [-1, -1, -1]
    assert stats.tolist() == [[0, 1, 0, 0], [0, 1, 0, 0], [2, 3, 0, 0]]
    assert ds.tolist() == [[33, 0, 5, 2]]
    # admission only at dispatch steps: nobody is preempted, B completes at 23
    st, ch, q, stats, ds = tiny(oracle, [0, 3, 100], [10, 10, 1], [50, 20, 1], [5, 5, 1], 40,
                                per_step=0)
    assert stats.tolist() == [[0, 1, 0, 0], [0, 1, 0, 0], [2, 1, 0, 0]]
    assert ds.tolist() == [[0, 0, 3, 0]]


def test_deferral_hand_trace(oracle):
    """One decoder of capacity 70, batches of one, beta = 5.  B (arrives at 1)
    has its prediction 50 steps late: at step 1 it waits, at step 20 it has
    waited past beta and goes round robin with the horizon (64) as its bound,
    so 1 + 10 + 64 > 70 keeps it behind C; at step 60 its prediction is in
    (U = 5) and it is admitted."""
    arr, p, true, pred = [0, 1, 20, 60], [10, 10, 1, 1], [5, 5, 1, 1], [5, 5, 1, 1]
    st, ch, q, stats, ds = tiny(oracle, arr, p, true, pred, 70, per_step=0, beta=5,
                                delay=[0, 50, 0, 0])
    assert st == 0 and ch.tolist() == [0, 0, 0, 0]
    assert stats.tolist() == [[0, 1, 0, 0], [0, 0, 0, 0], [1, 1, 1, 0], [1, 2, 0, 0]]
    assert ds[0, 0] == 40  # B waits from step 20 to step 60
    # without deferral B is dispatched and admitted at step 1
    st, ch, q, stats, ds = tiny(oracle, arr, p, true, pred, 70, per_step=0)
    assert stats.tolist() == [[0, 1, 0, 0], [0, 1, 0, 0], [2, 1, 0, 0], [1, 1, 0, 0]]
    # a beta the delay never reaches: B waits for its bound and is dispatched
    # at step 60 with U = 5 (the last dispatch step also forces the rest out)
    st, ch, q, stats, ds = tiny(oracle, arr, p, true, pred, 70, per_step=0, beta=1000,
                                delay=[0, 50, 0, 0])
    assert stats.tolist() == [[0, 1, 0, 0], [0, 0, 0, 0], [1, 1, 0, 0], [1, 2, 0, 0]]


def test_per_step_equals_batch_mode_with_room_to_spare(oracle, w):
    a = run(oracle, w, 20000, cap=10**9)
    b = run(oracle, w, 20000, cap=10**9, per_step=1)
    assert a[0] == b[0] == 0
    for x, y in zip(a[1:4], b[1:4]):
        assert np.array_equal(x, y)
    assert np.array_equal(a[4][:, :3], b[4][:, :3]) and b[4][:, 3].sum() == 0
    assert a[3][:, 2].sum() == 0  # nothing ever waits


def test_reservations_covering_true_lengths_never_preempt(oracle, w):
    exact = dict(w, pred_override=w["true"])
    for cap in (6000, 12000):
        st, ch, q, stats, ds = run(oracle, exact, 20000, cap=cap, per_step=1, accounting=1)
        assert st == 0 and ds[:, 3].sum() == 0 and stats[:, 3].sum() == 0
        assert stats[:, 2].sum() > 0  # the capacity binds
    # occupancy accounting admits against current tokens only: it preempts
    st, ch, q, stats, ds = run(oracle, exact, 20000, cap=6000, per_step=1)
    assert st == 0 and ds[:, 3].sum() > 0


def test_zero_delays_defer_nothing(oracle, w):
    a = run(oracle, w, 20000, cap=10000, per_step=1)
    b = run(oracle, w, 20000, cap=10000, per_step=1, beta=0,
            pred_delay=np.zeros(20000, np.int32))
    for x, y in zip(a, b):
        assert np.array_equal(np.asarray(x), np.asarray(y))


def test_late_predictions_with_zero_timeout_go_round_robin(oracle, w):
    late = np.full(20000, 10**6, np.int32)
    st, ch, q, stats, ds = run(oracle, w, 20000, beta=0, pred_delay=late)
    assert st == 0 and np.array_equal(ch, np.arange(20000) % w["D"])


@pytest.mark.parametrize("per_step,acc,beta", [(1, 0, -1), (1, 1, 300), (0, 2, 300), (1, 2, 1000)])
def test_statistics_sum_to_the_batch_totals(oracle, w, per_step, acc, beta):
    rng = np.random.default_rng(7)
    delay = rng.integers(0, 1500, 20000).astype(np.int32)
    st, ch, q, stats, ds = run(oracle, w, 20000, cap=10000, per_step=per_step, accounting=acc,
                               beta=beta, pred_delay=delay)
    assert st == 0 and ch.min() >= 0 and ch.max() < w["D"]
    assert ds[:, 2].sum() == stats[:, 1].sum()   # admissions
    assert ds[:, 1].sum() == stats[:, 3].sum()   # over-capacity batches
    assert (ds >= 0).all()
    # conservation: every request is dispatched by the last batch; each
    # admission starts a run that ends in a completion, a preemption or the
    # end, so admissions - preemptions = completed + running, and the rest
    # wait after the last admission
    assert ds[:, 2].sum() - ds[:, 3].sum() + stats[-1, 2] == 20000
