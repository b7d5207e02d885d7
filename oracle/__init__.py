"""ctypes front end of the plain-C oracle (``oracle.c``).

TEST INFRASTRUCTURE ONLY: imported by the test suite, the smoke check and the
benchmark's CPU-baseline leg.  The product package never imports it.

Functions take and return numpy arrays.  Each returns ``(status, outputs...)``
with the same status codes as the product library (0 ok, -1 invalid, -2 range,
-3 unbounded).
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_SRC_RR = os.path.join(_HERE, "oracle_rr.c")
_LIB = os.path.join(_HERE, "liboracle.so")

MODE_SNAPSHOT, MODE_SEQUENTIAL, MODE_ALG1_SNAPSHOT, MODE_ALG1_SEQUENTIAL = 0, 1, 2, 3


_SRC_P = os.path.join(_HERE, "oracle_p.cpp")
_LIB_P = os.path.join(_HERE, "liboracle_p.so")


def build(force: bool = False) -> str:
    """Compile ``liboracle.so`` (plain C11, -O2) and ``liboracle_p.so`` (the
    tier-P oracle, C++17 -O2, with OpenMP where the compiler has it) with the
    host compilers."""
    if force or not os.path.exists(_LIB) or (
            os.path.getmtime(_LIB) < max(os.path.getmtime(_SRC), os.path.getmtime(_SRC_RR),
                                         os.path.getmtime(os.path.join(_HERE, "oracle.h")))):
        tmp = _LIB + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-shared", "-fPIC",
                               "-o", tmp, _SRC, _SRC_RR])
        os.replace(tmp, _LIB)
    if force or not os.path.exists(_LIB_P) or os.path.getmtime(_LIB_P) < os.path.getmtime(_SRC_P):
        tmp = _LIB_P + f".{os.getpid()}.tmp"
        base = ["g++", "-O2", "-std=c++17", "-shared", "-fPIC", "-o", tmp, _SRC_P]
        r = subprocess.run(base[:1] + ["-fopenmp"] + base[1:], capture_output=True, text=True)
        if r.returncode != 0:  # no OpenMP: the same code, one thread
            subprocess.check_call(base)
        os.replace(tmp, _LIB_P)
    return _LIB


_lib = None

_i32p = np.ctypeslib.ndpointer(np.int32, flags="C_CONTIGUOUS")
_i64p = np.ctypeslib.ndpointer(np.int64, flags="C_CONTIGUOUS")


class StreamCfg(ctypes.Structure):
    _fields_ = [("N", ctypes.c_int64), ("D", ctypes.c_int32),
                ("H", ctypes.c_int32), ("cap", ctypes.c_int32),
                ("batch", ctypes.c_int32), ("window", ctypes.c_int32),
                ("alpha_ppm", ctypes.c_uint32), ("max_wait", ctypes.c_int32),
                ("dispatch", ctypes.c_int32), ("local", ctypes.c_int32),
                ("accounting", ctypes.c_int32), ("per_step", ctypes.c_int32),
                ("beta", ctypes.c_int32)]


# streaming-loop policies (the Sec. 4 ablations, the baselines, App. C)
DISPATCH_MAPS, DISPATCH_MC, DISPATCH_RR, DISPATCH_LR = 0, 1, 2, 3
LOCAL_SJF, LOCAL_FCFS = 0, 1
ACCOUNT_OCCUPANCY, ACCOUNT_STAGED, ACCOUNT_HELD = 0, 1, 2


class RRCfg(ctypes.Structure):
    _fields_ = [("n_req", ctypes.c_int64), ("N", ctypes.c_int32), ("C", ctypes.c_int32),
                ("t_tok_us", ctypes.c_int32), ("theta_ppm", ctypes.c_uint32)]


def lib():
    global _lib
    if _lib is None:
        L = ctypes.CDLL(build())
        L.oracle_rank.restype = ctypes.c_int64
        L.oracle_rank.argtypes = [ctypes.c_int64, ctypes.c_uint32]
        L.oracle_calibrate.argtypes = [_i32p, _i32p, ctypes.c_int64,
                                       ctypes.c_uint32,
                                       ctypes.POINTER(ctypes.c_int64)]
        L.oracle_bound.argtypes = [_i32p, ctypes.c_int64, ctypes.c_int64, _i32p]
        L.oracle_occupancy.argtypes = [ctypes.c_int32, ctypes.c_int32, _i64p,
                                       ctypes.c_int64, _i32p, _i32p, _i32p,
                                       _i32p]
        L.oracle_occupancy_cell.restype = ctypes.c_int64
        L.oracle_occupancy_cell.argtypes = [ctypes.c_int32, _i64p,
                                            ctypes.c_int32, ctypes.c_int32,
                                            _i32p, _i32p, _i32p]
        vp = ctypes.c_void_p
        L.oracle_dispatch.argtypes = [ctypes.c_int32, ctypes.c_int32,
                                      ctypes.c_int32, ctypes.c_int32, vp, vp,
                                      vp, vp, ctypes.c_int64, vp, vp, vp,
                                      ctypes.c_int64, vp, vp, vp, vp]
        L.oracle_order_local.argtypes = [ctypes.c_int64, ctypes.c_int32, vp, vp,
                                         vp, vp, ctypes.c_int32, vp, vp]
        L.oracle_stream.argtypes = [ctypes.POINTER(StreamCfg), _i64p, _i32p,
                                    _i32p, _i32p, ctypes.c_void_p, _i32p, _i32p, _i64p,
                                    _i64p]
        L.oracle_rr_pressure.argtypes = [ctypes.POINTER(RRCfg), _i64p, _i32p, _i32p,
                                         _i64p, _i64p, _i64p, ctypes.POINTER(ctypes.c_int64)]
        _lib = L
    return _lib


_libp = None


def libp():
    """The tier-P oracle (``oracle_p.cpp``)."""
    global _libp
    if _libp is None:
        build()
        L = ctypes.CDLL(_LIB_P)
        vp, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
        L.oraclep_threads.argtypes = [ctypes.c_int]
        L.oraclep_calibrate.argtypes = [vp, vp, i64, ctypes.c_uint32, ctypes.POINTER(i64)]
        L.oraclep_bound.argtypes = [vp, i64, i64, vp]
        L.oraclep_occupancy.argtypes = [i32, i32, vp, i64, vp, vp, vp, vp]
        L.oraclep_dispatch_snapshot.argtypes = [i32, i32, vp, vp, vp, i64, vp, vp, vp, vp]
        L.oraclep_order_local.argtypes = [i64, i32, vp, vp, vp, vp, i32, vp, vp]
        _libp = L
    return _libp


def _c32(a):
    return np.ascontiguousarray(a, dtype=np.int32)


def _c64(a):
    return np.ascontiguousarray(a, dtype=np.int64)


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def rank(n: int, alpha_ppm: int) -> int:
    return int(lib().oracle_rank(n, alpha_ppm))


def calibrate(true_len, pred_len, alpha_ppm: int):
    t, p = _c32(true_len), _c32(pred_len)
    q = ctypes.c_int64(0)
    st = lib().oracle_calibrate(t, p, t.shape[0], alpha_ppm, ctypes.byref(q))
    return st, int(q.value)


def bound(pred, q: int):
    p = _c32(pred)
    out = np.empty_like(p)
    st = lib().oracle_bound(p, p.shape[0], q, out)
    return st, out


def occupancy(D: int, H: int, res_off, prompt, gen, bnd):
    off = _c64(res_off)
    p, g, u = _c32(prompt), _c32(gen), _c32(bnd)
    K = np.empty((D, H), dtype=np.int32)
    st = lib().oracle_occupancy(D, H, off, p.shape[0], p, g, u, K.reshape(-1))
    return st, K


def occupancy_cell(H: int, res_off, k: int, t: int, prompt, gen, bnd) -> int:
    return int(lib().oracle_occupancy_cell(H, _c64(res_off), k, t, _c32(prompt),
                                           _c32(gen), _c32(bnd)))


def dispatch(mode: int, D: int, H: int, S: int, K, cap, Q, cand_prompt,
             cand_bound, res_off=None, prompt=None, gen=None, bnd=None):
    """Returns (status, choice, headroom, K_after, Q_after).  K and Q are
    copied; SEQUENTIAL modes update the copies in place."""
    Kc = None if K is None else _c32(K).copy()
    Qc = _c32(Q).copy()
    capc = _c32(cap)
    cp, cb = _c32(cand_prompt), _c32(cand_bound)
    J = cp.shape[0]
    choice = np.empty(J, dtype=np.int32)
    head = np.empty(J, dtype=np.int64)
    off = None if res_off is None else _c64(res_off)
    pr = None if prompt is None else _c32(prompt)
    ge = None if gen is None else _c32(gen)
    bo = None if bnd is None else _c32(bnd)
    R = 0 if pr is None else pr.shape[0]
    st = lib().oracle_dispatch(mode, D, H, S, _ptr(Kc), _ptr(capc), _ptr(Qc),
                               _ptr(off), R, _ptr(pr), _ptr(ge), _ptr(bo), J,
                               _ptr(cp), _ptr(cb), _ptr(choice), _ptr(head))
    return st, choice, head, Kc, Qc


def order_local(D: int, dec, bnd, wait, arrival, max_wait: int):
    d, b, w, a = _c32(dec), _c32(bnd), _c32(wait), _c32(arrival)
    N = d.shape[0]
    perm = np.empty(N, dtype=np.int32)
    seg = np.empty(D + 1, dtype=np.int64)
    st = lib().oracle_order_local(N, D, _ptr(d), _ptr(b), _ptr(w), _ptr(a),
                                  max_wait, _ptr(perm), _ptr(seg))
    return st, perm, seg


def stream(N, D, H, cap, batch, window, alpha_ppm, max_wait, arrival_ms,
           prompt, true_len, pred, dispatch=DISPATCH_MAPS, local=LOCAL_SJF,
           accounting=ACCOUNT_OCCUPANCY, with_dec_stats=False, per_step=0, beta=-1,
           pred_delay=None):
    """Returns (status, choice, q, stats [nb][4]) and, with with_dec_stats,
    the per-decoder statistics [D][4] as a fifth item.  per_step=1 admits on
    every step with preemption; beta >= 0 with pred_delay [N] defers a
    request until its bound is available, round robin after beta steps."""
    cfg = StreamCfg(N, D, H, cap, batch, window, alpha_ppm, max_wait, dispatch, local,
                    accounting, per_step, beta)
    nb = (N + batch - 1) // batch
    choice = np.empty(N, dtype=np.int32)
    q = np.empty(nb, dtype=np.int32)
    stats = np.empty(4 * nb, dtype=np.int64)
    dstats = np.zeros(4 * D, dtype=np.int64)
    pdl = None if pred_delay is None else _c32(pred_delay[:N])
    st = lib().oracle_stream(ctypes.byref(cfg), _c64(arrival_ms[:N]),
                             _c32(prompt[:N]), _c32(true_len[:N]),
                             _c32(pred[:N]),
                             None if pdl is None else pdl.ctypes.data_as(ctypes.c_void_p),
                             choice, q, stats, dstats)
    if with_dec_stats:
        return st, choice, q, stats.reshape(nb, 4), dstats.reshape(D, 4)
    return st, choice, q, stats.reshape(nb, 4)


def rr_pressure(N: int, C: int, t_tok_us: int, theta_ppm: int, arrival_us, prompt, out_len):
    """The App. A round-robin simulation of one realisation.  Returns (status,
    admit_us, done_us, stats [N][6] = T_hp, B_hp, C_hp, completed, longest
    queue, total wait (times in microseconds), t_sim)."""
    a, p, o = _c64(arrival_us), _c32(prompt), _c32(out_len)
    n = a.shape[0]
    cfg = RRCfg(n, N, C, t_tok_us, theta_ppm)
    admit = np.zeros(n, dtype=np.int64)
    done = np.zeros(n, dtype=np.int64)
    stats = np.zeros(6 * N, dtype=np.int64)
    tsim = ctypes.c_int64(0)
    st = lib().oracle_rr_pressure(ctypes.byref(cfg), a, p, o, admit, done, stats,
                                  ctypes.byref(tsim))
    return st, admit, done, stats.reshape(N, 6), int(tsim.value)


# ---------------------------------------------------------------------------
# tier P: the same results computed the plain way (oracle_p.cpp)
# ---------------------------------------------------------------------------

def p_threads(n: int = 1) -> int:
    """Host threads for the tier-P loops (n <= 0: every core); returns the
    number used (1 when the library was built without OpenMP)."""
    return int(libp().oraclep_threads(n))


def p_calibrate(true_len, pred_len, alpha_ppm: int):
    t, p = _c32(true_len), _c32(pred_len)
    q = ctypes.c_int64(0)
    st = libp().oraclep_calibrate(_ptr(t), _ptr(p), t.shape[0], alpha_ppm, ctypes.byref(q))
    return st, int(q.value)


def p_bound(pred, q: int):
    p = _c32(pred)
    out = np.empty_like(p)
    st = libp().oraclep_bound(_ptr(p), p.shape[0], q, _ptr(out))
    return st, out


def p_occupancy(D: int, H: int, res_off, prompt, gen, bnd, out=None):
    """``out``: an optional [D][H] int32 array to write K into (reused)."""
    off = _c64(res_off)
    p, g, u = _c32(prompt), _c32(gen), _c32(bnd)
    K = np.empty((D, H), dtype=np.int32) if out is None else out
    st = libp().oraclep_occupancy(D, H, _ptr(off), p.shape[0], _ptr(p), _ptr(g), _ptr(u),
                                  _ptr(K))
    return st, K


def p_dispatch_snapshot(D: int, H: int, K, cap, Q, cand_prompt, cand_bound):
    Kc, capc, Qc = _c32(K), _c32(cap), _c32(Q)
    cp, cb = _c32(cand_prompt), _c32(cand_bound)
    J = cp.shape[0]
    choice = np.empty(J, dtype=np.int32)
    head = np.empty(J, dtype=np.int64)
    st = libp().oraclep_dispatch_snapshot(D, H, _ptr(Kc), _ptr(capc), _ptr(Qc), J, _ptr(cp),
                                          _ptr(cb), _ptr(choice), _ptr(head))
    return st, choice, head


def p_order_local(D: int, dec, bnd, wait, arrival, max_wait: int, out=None):
    """``out``: an optional [N] int32 array for the order (reused)."""
    d, b, w, a = _c32(dec), _c32(bnd), _c32(wait), _c32(arrival)
    N = d.shape[0]
    perm = np.empty(N, dtype=np.int32) if out is None else out
    seg = np.empty(D + 1, dtype=np.int64)
    st = libp().oraclep_order_local(N, D, _ptr(d), _ptr(b), _ptr(w), _ptr(a), max_wait,
                                    _ptr(perm), _ptr(seg))
    return st, perm, seg
