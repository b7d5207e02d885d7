"""Thin Python binding of the MAPS C ABI (``include/maps.h``).

Argument marshalling only: every function passes torch tensors' device
pointers and the current CUDA stream to the function of the same name in
``libmaps.so`` and returns its status.  Every step of the computation runs in
the library's CUDA kernels; there is no CPU path.  Importing this module
loads the library and fails loudly when it is missing.
"""
from __future__ import annotations

import ctypes
import os

import torch

MAPS_OK = 0
MAPS_E_INVALID = -1
MAPS_E_RANGE = -2
MAPS_E_UNBOUNDED = -3
MAPS_E_TIMEOUT = -4
MAPS_E_CUDA = -5
MAPS_E_WORKSPACE = -6

MODE_SNAPSHOT = 0
MODE_SEQUENTIAL = 1
MODE_ALG1_SNAPSHOT = 2
MODE_ALG1_SEQUENTIAL = 3

STATUS_NAMES = {0: "MAPS_OK", -1: "MAPS_E_INVALID", -2: "MAPS_E_RANGE",
                -3: "MAPS_E_UNBOUNDED", -4: "MAPS_E_TIMEOUT", -5: "MAPS_E_CUDA",
                -6: "MAPS_E_WORKSPACE"}

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libmaps.so")


class StreamCfg(ctypes.Structure):
    """``maps_stream_cfg`` of include/maps.h."""
    _fields_ = [("N", ctypes.c_int64), ("D", ctypes.c_int32), ("H", ctypes.c_int32),
                ("cap", ctypes.c_int32), ("batch", ctypes.c_int32), ("window", ctypes.c_int32),
                ("alpha_ppm", ctypes.c_uint32), ("max_wait", ctypes.c_int32),
                ("dispatch_policy", ctypes.c_int32), ("local_order", ctypes.c_int32),
                ("accounting", ctypes.c_int32), ("per_step", ctypes.c_int32),
                ("beta", ctypes.c_int32)]


# maps_stream_cfg policy fields
STREAM_MAPS, STREAM_MC, STREAM_RR, STREAM_LR = 0, 1, 2, 3
STREAM_SJF, STREAM_FCFS = 0, 1
STREAM_OCCUPANCY, STREAM_STAGED, STREAM_HELD = 0, 1, 2


class RRCfg(ctypes.Structure):
    """``maps_rr_cfg`` of include/maps.h."""
    _fields_ = [("n_req", ctypes.c_int64), ("N", ctypes.c_int32), ("C", ctypes.c_int32),
                ("t_tok_us", ctypes.c_int32), ("theta_ppm", ctypes.c_uint32)]


class MapsError(RuntimeError):
    def __init__(self, status: int, what: str = ""):
        super().__init__(f"{what}: {STATUS_NAMES.get(status, status)}")
        self.status = status


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(
            f"{LIB_PATH} is missing: build it with paper_2609_15359_gb300.build.build() "
            "(nvcc, sm_103a). There is no CPU fallback.")
    lib = ctypes.CDLL(LIB_PATH)
    i32, i64, u32, sz, vp = (ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32,
                             ctypes.c_size_t, ctypes.c_void_p)
    sigs = {
        "maps_version": ([], ctypes.c_int),
        "maps_last_cuda_error": ([], ctypes.c_int),
        "maps_check": ([vp, vp], ctypes.c_int),
        "maps_set_dispatch_events": ([vp, vp], ctypes.c_int),
        "maps_test_withhold_lookback": ([i32, u32], ctypes.c_int),
        "maps_test_absent_block": ([i32], ctypes.c_int),
        "maps_test_calibrate_absent_block": ([i32, u32], ctypes.c_int),
        "maps_calibrate_workspace_size": ([i64, i64], sz),
        "maps_calibrate": ([vp, vp, i64, u32, vp, i64, vp, vp, vp, vp, sz, vp], ctypes.c_int),
        "maps_project_occupancy_workspace_size": ([i32, i32, i64], sz),
        "maps_project_occupancy": ([i32, i32, vp, i64, vp, vp, vp, vp, vp, vp, sz, vp], ctypes.c_int),
        "maps_dispatch_workspace_size": ([i32, i32, i32, i64], sz),
        "maps_dispatch": ([i32, i32, i32, i32, vp, vp, vp, vp, vp, i64, vp, vp, vp, i64, vp, vp,
                           vp, vp, vp, sz, vp], ctypes.c_int),
        "maps_order_local_workspace_size": ([i64, i32], sz),
        "maps_order_local": ([i64, i32, vp, vp, vp, vp, i32, vp, vp, vp, sz, vp], ctypes.c_int),
        "maps_order_local_static": ([i64, i32, vp, vp, vp, vp, i32, vp, vp, vp, vp], ctypes.c_int),
        "maps_rr_pressure_workspace_size": ([ctypes.POINTER(RRCfg), i64], sz),
        "maps_rr_pressure": ([ctypes.POINTER(RRCfg), i64, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp],
                             ctypes.c_int),
        "maps_stream_workspace_size": ([ctypes.POINTER(StreamCfg)], sz),
        "maps_stream_run": ([ctypes.POINTER(StreamCfg), vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz,
                             vp],
                            ctypes.c_int),
    }
    for name, (args, res) in sigs.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    return lib


lib = _load()
EXPORTS = ("maps_version", "maps_last_cuda_error", "maps_check", "maps_set_dispatch_events",
           "maps_test_withhold_lookback", "maps_test_absent_block",
           "maps_test_calibrate_absent_block", "maps_calibrate_workspace_size", "maps_calibrate",
           "maps_project_occupancy_workspace_size", "maps_project_occupancy",
           "maps_dispatch_workspace_size", "maps_dispatch",
           "maps_order_local_workspace_size", "maps_order_local", "maps_order_local_static",
           "maps_stream_workspace_size", "maps_stream_run",
           "maps_rr_pressure_workspace_size", "maps_rr_pressure")


def _stream(stream) -> ctypes.c_void_p:
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _ptr(t, dtype=None) -> ctypes.c_void_p:
    if t is None:
        return ctypes.c_void_p(0)
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError("expected a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"expected {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise TypeError("expected a contiguous tensor")
    return ctypes.c_void_p(t.data_ptr())


class Workspace:
    """Zero-filled device scratch owned by the caller, grown on demand."""

    def __init__(self, nbytes: int = 0, device=None):
        self.device = torch.device("cuda") if device is None else torch.device(device)
        self.buf = torch.zeros(max(int(nbytes), 256), dtype=torch.uint8, device=self.device)

    def ensure(self, nbytes: int) -> "Workspace":
        if nbytes > self.buf.numel():
            self.buf = torch.zeros(int(nbytes), dtype=torch.uint8, device=self.device)
        return self

    @property
    def ptr(self) -> ctypes.c_void_p:
        return ctypes.c_void_p(self.buf.data_ptr())

    @property
    def nbytes(self) -> int:
        return self.buf.numel()


def maps_check(ws: Workspace, stream=None) -> int:
    return lib.maps_check(ws.ptr, _stream(stream))


def maps_set_dispatch_events(before=None, after=None) -> int:
    """Benchmarking aid: torch.cuda.Event objects that later SNAPSHOT
    maps_dispatch calls of this thread record around their scoring kernel
    (None, None turns it off).  The events must already exist on the device:
    record each once first."""
    h = lambda e: None if e is None else ctypes.c_void_p(e.cuda_event)  # noqa: E731
    return lib.maps_set_dispatch_events(h(before), h(after))


def maps_calibrate(true_len, pred_len, alpha_ppm: int, query_pred=None, bound_out=None,
                   q_dev_out=None, q_host: bool = False, ws: Workspace | None = None,
                   stream=None):
    """Returns (status, q) where q is the host quantile when ``q_host``."""
    n = true_len.numel()
    m = 0 if query_pred is None else query_pred.numel()
    ws = ws or Workspace()
    ws.ensure(lib.maps_calibrate_workspace_size(n, m))
    qh = ctypes.c_int32(0)
    st = lib.maps_calibrate(_ptr(true_len, torch.int32), _ptr(pred_len, torch.int32), n,
                            int(alpha_ppm), _ptr(query_pred, torch.int32), m,
                            _ptr(bound_out, torch.int32), _ptr(q_dev_out, torch.int32),
                            ctypes.byref(qh) if q_host else None, ws.ptr, ws.nbytes,
                            _stream(stream))
    return st, (int(qh.value) if q_host else None)


def kmax_shape(D: int, H: int) -> tuple[int, int]:
    """Shape of the 16-step summary of K (uint32 values, stored as int32)."""
    return D, (H + 15) // 16


def maps_project_occupancy(D: int, H: int, res_off, prompt, gen, bound, K_out, kmax_out=None,
                           ws: Workspace | None = None, stream=None) -> int:
    R = prompt.numel()
    ws = ws or Workspace()
    ws.ensure(lib.maps_project_occupancy_workspace_size(D, H, R))
    return lib.maps_project_occupancy(D, H, _ptr(res_off, torch.int64), R,
                                      _ptr(prompt, torch.int32), _ptr(gen, torch.int32),
                                      _ptr(bound, torch.int32), _ptr(K_out, torch.int32),
                                      _ptr(kmax_out, torch.int32), ws.ptr, ws.nbytes,
                                      _stream(stream))


def maps_dispatch(mode: int, D: int, H: int, S: int, K, cap, Q, cand_prompt, cand_bound,
                  choice_out, headroom_out=None, res_off=None, prompt=None, gen=None,
                  bound=None, kmax=None, ws: Workspace | None = None, stream=None) -> int:
    J = cand_prompt.numel()
    R = 0 if prompt is None else prompt.numel()
    ws = ws or Workspace()
    ws.ensure(lib.maps_dispatch_workspace_size(mode, D, H, J))
    return lib.maps_dispatch(mode, D, H, S, _ptr(K, torch.int32), _ptr(kmax, torch.int32),
                             _ptr(cap, torch.int32),
                             _ptr(Q, torch.int32), _ptr(res_off, torch.int64), R,
                             _ptr(prompt, torch.int32), _ptr(gen, torch.int32),
                             _ptr(bound, torch.int32), J, _ptr(cand_prompt, torch.int32),
                             _ptr(cand_bound, torch.int32), _ptr(choice_out, torch.int32),
                             _ptr(headroom_out, torch.int64), ws.ptr, ws.nbytes,
                             _stream(stream))


def maps_order_local(D: int, dec, bound, wait, arrival, max_wait: int, perm_out, seg_off_out,
                     ws: Workspace | None = None, stream=None) -> int:
    N = dec.numel()
    ws = ws or Workspace()
    ws.ensure(lib.maps_order_local_workspace_size(N, D))
    return lib.maps_order_local(N, D, _ptr(dec, torch.int32), _ptr(bound, torch.int32),
                                _ptr(wait, torch.int32), _ptr(arrival, torch.int32),
                                int(max_wait), _ptr(perm_out, torch.int32),
                                _ptr(seg_off_out, torch.int64), ws.ptr, ws.nbytes,
                                _stream(stream))


def maps_order_local_static(D: int, dec, bound, wait, arrival, max_wait: int, perm_out,
                            seg_off_out, sync_status: bool = True, stream=None) -> int:
    """maps_order_local with the library's fixed scratch array: no workspace,
    no allocation.  N <= 65,536 and D <= 4,096."""
    N = dec.numel()
    st = ctypes.c_int32(0)
    return lib.maps_order_local_static(N, D, _ptr(dec, torch.int32), _ptr(bound, torch.int32),
                                       _ptr(wait, torch.int32), _ptr(arrival, torch.int32),
                                       int(max_wait), _ptr(perm_out, torch.int32),
                                       _ptr(seg_off_out, torch.int64),
                                       ctypes.byref(st) if sync_status else None,
                                       _stream(stream))


def stream_cfg(N: int, D: int, H: int, cap: int, batch: int, window: int, alpha_ppm: int,
               max_wait: int, dispatch_policy: int = STREAM_MAPS, local_order: int = STREAM_SJF,
               accounting: int = STREAM_OCCUPANCY, per_step: int = 0,
               beta: int = -1) -> StreamCfg:
    return StreamCfg(int(N), int(D), int(H), int(cap), int(batch), int(window), int(alpha_ppm),
                     int(max_wait), int(dispatch_policy), int(local_order), int(accounting),
                     int(per_step), int(beta))


def maps_stream_run(cfg: StreamCfg, arrival_ms, prompt, true_len, pred, choice_out, q_out,
                    stats_out, dec_stats_out=None, ws: Workspace | None = None,
                    stream=None, pred_delay=None) -> int:
    """The whole streaming loop on the device; returns the full status.
    dec_stats_out: optional [D][4] int64 per-decoder statistics; pred_delay:
    [N] int32 prediction delays (required when cfg.beta >= 0)."""
    ws = ws or Workspace()
    ws.ensure(lib.maps_stream_workspace_size(ctypes.byref(cfg)))
    return lib.maps_stream_run(ctypes.byref(cfg), _ptr(arrival_ms, torch.int64),
                               _ptr(prompt, torch.int32), _ptr(true_len, torch.int32),
                               _ptr(pred, torch.int32), _ptr(pred_delay, torch.int32),
                               _ptr(choice_out, torch.int32),
                               _ptr(q_out, torch.int32), _ptr(stats_out, torch.int64),
                               _ptr(dec_stats_out, torch.int64), ws.ptr, ws.nbytes,
                               _stream(stream))


def maps_rr_pressure(N: int, C: int, t_tok_us: int, theta_ppm: int, arrival_us, prompt, out_len,
                     admit_out, done_out, stats_out, t_sim_out, ws: Workspace | None = None,
                     stream=None) -> int:
    """The App. A round-robin simulation of n_real realisations at once.
    arrival_us [n_real][n_req] int64, prompt / out_len [n_real][n_req] int32;
    outputs admit / done [n_real][n_req] int64, stats [n_real][N][6] int64,
    t_sim [n_real] int64."""
    n_real, n_req = arrival_us.shape
    cfg = RRCfg(int(n_req), int(N), int(C), int(t_tok_us), int(theta_ppm))
    ws = ws or Workspace()
    ws.ensure(lib.maps_rr_pressure_workspace_size(ctypes.byref(cfg), n_real))
    return lib.maps_rr_pressure(ctypes.byref(cfg), n_real, _ptr(arrival_us, torch.int64),
                                _ptr(prompt, torch.int32), _ptr(out_len, torch.int32),
                                _ptr(admit_out, torch.int64), _ptr(done_out, torch.int64),
                                _ptr(stats_out, torch.int64), _ptr(t_sim_out, torch.int64),
                                ws.ptr, ws.nbytes, _stream(stream))
