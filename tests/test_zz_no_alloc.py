"""The allocation-free local order (maps_order_local_static).

Callers that cannot allocate device memory -- a scheduler inside a process
whose allocator it does not own, or one that must not allocate while
serving -- use this entry point: its scratch is an array compiled into the
library.  Call after call it must give the oracle's order exactly, although
the array keeps the previous call's contents.  The cases alternate between
the one-block form and the multi-kernel forms (counters, look-back state and
plan carved from the array), so every multi-kernel call but the first reuses
state a larger call left behind; one case has more than 1,024 decoders (the
scatter that claims slots by atomics).  Named to be collected last.
"""
import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


def _inputs(rng, N, D, sorted_arrival):
    dec = rng.integers(0, D, N).astype(np.int32)
    U = rng.integers(0, 5000, N).astype(np.int32)
    wait = rng.integers(0, 3000, N).astype(np.int32)
    if sorted_arrival:
        arr = np.arange(N, dtype=np.int32)
    else:
        arr = rng.integers(0, 2**31 - 1, N, dtype=np.int64).astype(np.int32)
    return dec, U, wait, arr


def _static(M, D, host_ins, mw):
    ins = [torch.from_numpy(x).cuda() for x in host_ins]
    N = ins[0].numel()
    perm = torch.full((max(N, 1),), -1, dtype=torch.int32, device="cuda")
    seg = torch.full((D + 1,), -1, dtype=torch.int64, device="cuda")
    st = ctypes.c_int32(-99)
    rc = M.lib.maps_order_local_static(N, D, M._ptr(ins[0]), M._ptr(ins[1]), M._ptr(ins[2]),
                                       M._ptr(ins[3]), mw, M._ptr(perm), M._ptr(seg),
                                       ctypes.byref(st), M._stream(None))
    torch.cuda.synchronize()
    return rc, st.value, perm[:N].cpu().numpy(), seg.cpu().numpy()


# (N, D, arrival in index order, max_wait): one-block and multi-kernel forms
# alternate; consecutive multi-kernel calls of different sizes and forms
CASES = [(65536, 256, False, 1000), (3000, 7, True, 500), (20000, 2000, False, 800),
         (65536, 256, True, 1000), (50000, 4096, True, 0), (4608, 4096, False, 300),
         (40000, 3, False, 2000), (1, 1, True, 0)]


def test_static_order_equals_the_oracle_on_consecutive_calls(oracle):
    if not torch.cuda.is_available():
        pytest.fail("CUDA device required")
    from paper_2609_15359_gb300 import maps as M
    rng = np.random.default_rng(42)
    for N, D, srt, mw in CASES:
        host_ins = _inputs(rng, N, D, srt)
        sto, po, so = oracle.order_local(D, *host_ins, mw)
        rc, st, perm, seg = _static(M, D, host_ins, mw)
        assert rc == 0 and st == 0 and sto == 0, (N, D, rc, st)
        assert np.array_equal(perm, po), (N, D)
        assert np.array_equal(seg, so), (N, D)


def test_static_order_reports_a_data_error_then_recovers(oracle):
    """A decoder index out of range is MAPS_E_RANGE through status_host; the
    next call on the same array starts from a clear status and is exact."""
    from paper_2609_15359_gb300 import maps as M
    rng = np.random.default_rng(7)
    dec, U, wait, arr = _inputs(rng, 20000, 300, True)
    bad = dec.copy()
    bad[123] = 300
    rc, st, _, _ = _static(M, 300, (bad, U, wait, arr), 1000)
    assert st == M.MAPS_E_RANGE
    sto, po, so = oracle.order_local(300, dec, U, wait, arr, 1000)
    rc, st, perm, seg = _static(M, 300, (dec, U, wait, arr), 1000)
    assert rc == 0 and st == 0 and sto == 0
    assert np.array_equal(perm, po) and np.array_equal(seg, so)


def test_static_order_rejects_sizes_beyond_its_array():
    from paper_2609_15359_gb300 import maps as M
    assert M.lib.maps_order_local_static(65537, 4, None, None, None, None, 0, None, None, None,
                                         None) == M.MAPS_E_WORKSPACE
    assert M.lib.maps_order_local_static(10, 4097, None, None, None, None, 0, None, None, None,
                                         None) == M.MAPS_E_WORKSPACE
