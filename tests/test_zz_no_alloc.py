"""The allocation-free local order (maps_order_local_static).

Callers that cannot allocate device memory -- a scheduler inside a process
whose allocator it does not own, or one that must not allocate while
serving -- use this entry point: its scratch is an array compiled into the
library.  It must give exactly what maps_order_local gives with a caller
workspace, call after call (the array keeps the previous call's contents).
Named to be collected last.
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
    return [torch.from_numpy(x).cuda() for x in (dec, U, wait, arr)]


def _reference(M, D, ins, mw):
    N = ins[0].numel()
    perm = torch.full((N,), -1, dtype=torch.int32, device="cuda")
    seg = torch.full((D + 1,), -1, dtype=torch.int64, device="cuda")
    ws = M.Workspace()
    assert M.maps_order_local(D, *ins, mw, perm, seg, ws=ws) == 0
    assert M.maps_check(ws) == 0
    return perm.cpu().numpy(), seg.cpu().numpy()


def _static(M, D, ins, mw):
    N = ins[0].numel()
    perm = torch.full((N,), -1, dtype=torch.int32, device="cuda")
    seg = torch.full((D + 1,), -1, dtype=torch.int64, device="cuda")
    st = ctypes.c_int32(-99)
    rc = M.lib.maps_order_local_static(N, D, M._ptr(ins[0]), M._ptr(ins[1]), M._ptr(ins[2]),
                                       M._ptr(ins[3]), mw, M._ptr(perm), M._ptr(seg),
                                       ctypes.byref(st), M._stream(None))
    assert rc == 0 and st.value == 0
    torch.cuda.synchronize()
    return perm.cpu().numpy(), seg.cpu().numpy()


def test_static_order_matches_workspace_order_on_consecutive_calls():
    if not torch.cuda.is_available():
        pytest.fail("CUDA device required")
    from paper_2609_15359_gb300 import maps as M
    rng = np.random.default_rng(42)
    cases = [(65536, 256, False, 1000), (3000, 7, True, 500)]
    for N, D, srt, mw in cases:  # two calls in a row on the shared array
        ins = _inputs(rng, N, D, srt)
        p_ref, s_ref = _reference(M, D, ins, mw)
        p_st, s_st = _static(M, D, ins, mw)
        assert np.array_equal(p_st, p_ref)
        assert np.array_equal(s_st, s_ref)


def test_static_order_rejects_sizes_beyond_its_array():
    from paper_2609_15359_gb300 import maps as M
    assert M.lib.maps_order_local_static(65537, 4, None, None, None, None, 0, None, None, None,
                                         None) == M.MAPS_E_WORKSPACE
    assert M.lib.maps_order_local_static(10, 4097, None, None, None, None, 0, None, None, None,
                                         None) == M.MAPS_E_WORKSPACE
