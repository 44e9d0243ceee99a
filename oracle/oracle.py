"""fp64 CPU oracle for the Frac selective fractional SSM scan (arXiv 2609.36314).

TEST INFRASTRUCTURE ONLY: imported by tests/, ``__graft_entry__.smoke()`` and
the ``cpu_baseline`` / ``--impl reference`` legs of ``bench.py``.  Nothing in
the product path (``paper_2609_36314_gb300``) imports it, and it imports
nothing from there.

The arithmetic lives in ``frac_oracle.c`` (plain C, fp64, sequential in t,
OpenMP over independent (batch, head) streams).  This module compiles it with
gcc on first use and marshals numpy arrays; every input is converted to
float64 first, so the oracle sees exactly the values the GPU path sees
(bf16 inputs are exactly representable in fp64).

Parity status: forward, backward and decode are pinned by tests/test_oracle_*.py
(closed-form impulse response, Mittag-Leffler tracking through the finite
sum-of-exponentials bank of Theorem 2, literal Algorithm 1, K=1 textbook SSM,
brute-force materialised kernel, chunked == sequential, finite differences,
an independent autograd implementation, invariances).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "frac_oracle.c")
_LIB_PATH = os.path.join(_HERE, "_build", "libfrac_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile frac_oracle.c into a shared library (gcc, -O2, OpenMP)."""
    os.makedirs(os.path.dirname(_LIB_PATH), exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-fopenmp", "-shared", "-fPIC", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            i64, dp, ci = ctypes.c_int64, ctypes.c_void_p, ctypes.c_int
            lib.frac_oracle_fwd.argtypes = [i64] * 7 + [dp] * 13 + [ci]
            lib.frac_oracle_fwd.restype = ci
            lib.frac_oracle_bwd.argtypes = [i64] * 7 + [dp] * 24 + [i64, ci]
            lib.frac_oracle_bwd.restype = ci
            lib.frac_oracle_decode.argtypes = [i64] * 6 + [dp] * 12
            lib.frac_oracle_decode.restype = ci
            lib.frac_oracle_max_threads.argtypes = []
            lib.frac_oracle_max_threads.restype = ci
            _lib = lib
    return _lib


def max_threads() -> int:
    return int(_load().frac_oracle_max_threads())


def _f64(a):
    if a is None:
        return None
    return np.ascontiguousarray(a, dtype=np.float64)


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _dims(x, Bm, tau):
    Bsz, L, H, P = x.shape
    G, N = Bm.shape[2], Bm.shape[3]
    K = tau.shape[1]
    return Bsz, L, H, P, G, N, K


def fwd(x, dt, alpha, lam, tau, Bm, Cm, w_read, w_write, D, h0=None, nthreads=None):
    """Sequential fp64 forward.  Returns (y [B,L,H,P], h_final [B,H,K,P,N])."""
    x, dt, alpha, lam, tau, Bm, Cm, w_read, w_write, D, h0 = map(
        _f64, (x, dt, alpha, lam, tau, Bm, Cm, w_read, w_write, D, h0))
    Bsz, L, H, P, G, N, K = _dims(x, Bm, tau)
    y = np.empty((Bsz, L, H, P))
    hf = np.empty((Bsz, H, K, P, N))
    nt = nthreads or max_threads()
    rc = _load().frac_oracle_fwd(Bsz, L, H, P, G, N, K, _ptr(x), _ptr(dt), _ptr(alpha), _ptr(lam),
                                 _ptr(tau), _ptr(Bm), _ptr(Cm), _ptr(w_read), _ptr(w_write),
                                 _ptr(D), _ptr(h0), _ptr(y), _ptr(hf), nt)
    if rc:
        raise RuntimeError(f"frac_oracle_fwd failed with code {rc}")
    return y, hf


def bwd(x, dt, alpha, lam, tau, Bm, Cm, w_read, w_write, D, dy, h0=None, dh_final=None,
        seg=32, nthreads=None):
    """fp64 adjoint of the sequential recurrence.

    Returns a dict with dx, ddt, dalpha, dlam, dB, dC, dw_read, dw_write, dD, dh0 and dtau
    (the gradient of the timescales tau [H, K]).
    """
    x, dt, alpha, lam, tau, Bm, Cm, w_read, w_write, D, dy, h0, dh_final = map(
        _f64, (x, dt, alpha, lam, tau, Bm, Cm, w_read, w_write, D, dy, h0, dh_final))
    Bsz, L, H, P, G, N, K = _dims(x, Bm, tau)
    out = dict(dx=np.empty_like(x), ddt=np.empty_like(dt), dalpha=np.empty_like(alpha),
               dlam=np.empty_like(lam), dB=np.empty_like(Bm), dC=np.empty_like(Cm),
               dw_read=np.empty_like(w_read), dw_write=np.empty_like(w_write),
               dD=np.empty_like(D), dh0=np.empty((Bsz, H, K, P, N)), dtau=np.empty_like(tau))
    nt = nthreads or max_threads()
    rc = _load().frac_oracle_bwd(
        Bsz, L, H, P, G, N, K, _ptr(x), _ptr(dt), _ptr(alpha), _ptr(lam), _ptr(tau), _ptr(Bm),
        _ptr(Cm), _ptr(w_read), _ptr(w_write), _ptr(D), _ptr(h0), _ptr(dy), _ptr(dh_final),
        _ptr(out["dx"]), _ptr(out["ddt"]), _ptr(out["dalpha"]), _ptr(out["dlam"]),
        _ptr(out["dB"]), _ptr(out["dC"]), _ptr(out["dw_read"]), _ptr(out["dw_write"]),
        _ptr(out["dD"]), _ptr(out["dh0"]), _ptr(out["dtau"]), int(seg), nt)
    if rc:
        raise RuntimeError(f"frac_oracle_bwd failed with code {rc}")
    return out


def decode(x_t, dt, alpha, lam, tau, B_t, C_t, w_read, w_write, D, state):
    """One recurrence step on a cached state.  Returns (y_t [B,H,P], new_state)."""
    x_t, dt, alpha, lam, tau, B_t, C_t, w_read, w_write, D = map(
        _f64, (x_t, dt, alpha, lam, tau, B_t, C_t, w_read, w_write, D))
    st = np.array(state, dtype=np.float64, copy=True, order="C")
    Bsz, H, P = x_t.shape
    G, N = B_t.shape[1], B_t.shape[2]
    K = tau.shape[1]
    y = np.empty((Bsz, H, P))
    rc = _load().frac_oracle_decode(Bsz, H, P, G, N, K, _ptr(x_t), _ptr(dt), _ptr(alpha),
                                    _ptr(lam), _ptr(tau), _ptr(B_t), _ptr(C_t), _ptr(w_read),
                                    _ptr(w_write), _ptr(D), _ptr(st), _ptr(y))
    if rc:
        raise RuntimeError(f"frac_oracle_decode failed with code {rc}")
    return y, st
