"""A bounded device wait that runs out is reported, and the device stays usable.

The calibration's cooperative kernel (calibration sets above 8,192 residuals)
waits at a bounded grid barrier after each select pass; the test aid
maps_test_calibrate_absent_block makes one of its blocks return at once, so
the others' wait runs out.

The local order's global form (arrival not in index order) sorts with
decoupled look-back between tiles: each tile waits, bounded, for its
predecessors' published counts.  The test aid maps_test_withhold_lookback
makes one tile publish nothing, so the next tile's wait runs out after a short
limit.  The call must then report MAPS_E_TIMEOUT through maps_check, write
only inside its outputs, and the next call on a fresh workspace must give the
oracle's order exactly.  Nothing faults, traps or hangs.
"""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


def test_order_lookback_timeout_is_reported_and_the_next_call_is_exact(oracle):
    if not torch.cuda.is_available():
        pytest.fail("CUDA device required")
    from paper_2609_15359_gb300 import maps as M
    rng = np.random.default_rng(11)
    N, D, mw = 200_000, 64, 1000
    dec = rng.integers(0, D, N).astype(np.int32)
    U = rng.integers(0, 40000, N).astype(np.int32)
    wait = rng.integers(0, 3000, N).astype(np.int32)
    arr = rng.integers(0, 2**31 - 1, N, dtype=np.int64).astype(np.int32)  # not in index order
    ins = [torch.from_numpy(x).cuda() for x in (dec, U, wait, arr)]
    perm = torch.full((N,), -1, dtype=torch.int32, device="cuda")
    seg = torch.full((D + 1,), -1, dtype=torch.int64, device="cuda")
    ws = M.Workspace()
    try:
        assert M.lib.maps_test_withhold_lookback(3, 2000) == 0
        assert M.maps_order_local(D, *ins, mw, perm, seg, ws=ws) == 0
        assert M.maps_check(ws) == M.MAPS_E_TIMEOUT
    finally:
        assert M.lib.maps_test_withhold_lookback(-1, 0) == 0
    p = perm.cpu().numpy()
    assert p.min() >= -1 and p.max() < N  # written only inside the output
    sto, po, so = oracle.order_local(D, dec, U, wait, arr, mw)
    ws2 = M.Workspace()
    perm.fill_(-1)
    assert M.maps_order_local(D, *ins, mw, perm, seg, ws=ws2) == 0
    assert M.maps_check(ws2) == 0 and sto == 0
    assert np.array_equal(perm.cpu().numpy(), po)
    assert np.array_equal(seg.cpu().numpy(), so)


@pytest.mark.parametrize("form", ["long_queue", "global"])
def test_order_grid_barrier_timeout_is_reported_and_the_next_call_is_exact(oracle, form):
    """Block 0 of the order's finishing kernel is made absent
    (maps_test_absent_block), so the others' first grid barrier runs out after
    a short limit: the call reports MAPS_E_TIMEOUT, every block ends at that
    barrier (what it wrote before stays inside the outputs and workspace), and
    the next call on a fresh workspace gives the oracle's order exactly.
    long_queue: arrival in index order and one queue of 20,000 entries (5 runs
    ranked pairwise, one barrier before the placement); global: arrival out of
    index order (the radix passes; the plan block 0 would write is never read,
    since every other block ends at the barrier after it)."""
    if not torch.cuda.is_available():
        pytest.fail("CUDA device required")
    from paper_2609_15359_gb300 import maps as M
    rng = np.random.default_rng(13)
    N, D, mw = 60_000, 8, 1000
    dec = np.where(np.arange(N) < 20_000, 0, rng.integers(1, D, N)).astype(np.int32)
    U = rng.integers(0, 40000, N).astype(np.int32)
    wait = rng.integers(0, 3000, N).astype(np.int32)
    if form == "long_queue":
        arr = np.arange(N, dtype=np.int32)
    else:
        arr = rng.integers(0, 2**31 - 1, N, dtype=np.int64).astype(np.int32)
    ins = [torch.from_numpy(x).cuda() for x in (dec, U, wait, arr)]
    perm = torch.full((N,), -1, dtype=torch.int32, device="cuda")
    seg = torch.full((D + 1,), -1, dtype=torch.int64, device="cuda")
    ws = M.Workspace()
    try:
        assert M.lib.maps_test_withhold_lookback(-1, 2000) == 0  # the waits' short limit
        assert M.lib.maps_test_absent_block(0) == 0
        assert M.maps_order_local(D, *ins, mw, perm, seg, ws=ws) == 0
        assert M.maps_check(ws) == M.MAPS_E_TIMEOUT
    finally:
        assert M.lib.maps_test_absent_block(-1) == 0
        assert M.lib.maps_test_withhold_lookback(-1, 0) == 0
    p = perm.cpu().numpy()
    assert p.min() >= -1 and p.max() < N  # written only inside the output
    sto, po, so = oracle.order_local(D, dec, U, wait, arr, mw)
    ws2 = M.Workspace()
    perm.fill_(-1)
    assert M.maps_order_local(D, *ins, mw, perm, seg, ws=ws2) == 0
    assert M.maps_check(ws2) == 0 and sto == 0
    assert np.array_equal(perm.cpu().numpy(), po)
    assert np.array_equal(seg.cpu().numpy(), so)


def test_calibrate_grid_barrier_timeout_is_reported_and_the_next_call_is_exact(oracle):
    """Block 0 of the calibration's cooperative kernel is made absent, so the
    other blocks' barrier after the first select pass runs out after a short
    limit: the call reports MAPS_E_TIMEOUT and writes no bound, and the next
    call on a fresh workspace gives the oracle's q and bounds exactly."""
    if not torch.cuda.is_available():
        pytest.fail("CUDA device required")
    from paper_2609_15359_gb300 import maps as M
    rng = np.random.default_rng(17)
    n, m, a = 200_000, 5_000, 100_000
    L = rng.integers(0, 40000, n).astype(np.int32)
    P = rng.integers(0, 40000, n).astype(np.int32)
    pred = rng.integers(0, 5000, m).astype(np.int32)
    Ld, Pd, pd = (torch.from_numpy(x).cuda() for x in (L, P, pred))
    U = torch.full((m + 1,), -9, dtype=torch.int32, device="cuda")
    qd = torch.full((1,), -9, dtype=torch.int32, device="cuda")
    ws = M.Workspace()
    try:
        assert M.lib.maps_test_calibrate_absent_block(0, 2000) == 0
        st, _ = M.maps_calibrate(Ld, Pd, a, pd, U[:m], qd, ws=ws)
        assert st == 0
        assert M.maps_check(ws) == M.MAPS_E_TIMEOUT
    finally:
        assert M.lib.maps_test_calibrate_absent_block(-1, 0) == 0
    assert (U.cpu().numpy() == -9).all() and int(qd.item()) == -9  # nothing written
    sto, qo = oracle.calibrate(L, P, a)
    _, Uo = oracle.bound(pred, qo)
    ws2 = M.Workspace()
    st, q = M.maps_calibrate(Ld, Pd, a, pd, U[:m], qd, q_host=True, ws=ws2)
    assert st == sto == 0 and q == qo == int(qd.item())
    assert np.array_equal(U[:m].cpu().numpy(), Uo) and int(U[m].item()) == -9
