"""ctypes loader for libfrac.so (the C ABI declared in include/frac.h).

No fallback: if the library cannot be loaded, every call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

from . import build as _build

_lock = threading.Lock()
_lib = None

# Every symbol include/frac.h declares.
EXPORTS = (
    "frac_scan_fwd_workspace_size",
    "frac_scan_fwd",
    "frac_scan_bwd_workspace_size",
    "frac_scan_bwd",
    "frac_decode_step",
    "frac_scan_fwd_static",
    "frac_scan_fwd_static_status",
    "frac_workspace_status",
    "frac_param_prep_fwd",
    "frac_param_prep_bwd",
    "frac_conv1d_fwd",
    "frac_conv1d_bwd",
    "frac_conv1d_step",
    "frac_gated_rmsnorm_fwd",
    "frac_gated_rmsnorm_bwd",
    "frac_trace_enable",
    "frac_trace_collect",
    "frac_trace_reset",
    "frac_status_string",
    "frac_last_error",
)

FRAC_OK = 0
FRAC_DTYPE_F32 = 0
FRAC_DTYPE_BF16 = 1
FRAC_FLAG_FORCE_SIMT = 1
FRAC_FLAG_BWD_REUSE_FWD_STATES = 2
FRAC_FLAG_TEST_EXPIRE_WAIT = 4
FRAC_SCAN_FWD_STATIC_SCRATCH_BYTES = 64 << 20


class FracDims(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int64), ("seqlen", ctypes.c_int64),
                ("nheads", ctypes.c_int64), ("headdim", ctypes.c_int64),
                ("ngroups", ctypes.c_int64), ("dstate", ctypes.c_int64),
                ("nmodes", ctypes.c_int64), ("chunk", ctypes.c_int64),
                ("dtype", ctypes.c_int32), ("flags", ctypes.c_int32)]


class FracPrepConfig(ctypes.Structure):
    _fields_ = [("dt_min", ctypes.c_float), ("dt_max", ctypes.c_float),
                ("lam_min", ctypes.c_float), ("lam_max", ctypes.c_float),
                ("flags", ctypes.c_int32), ("reserved", ctypes.c_int32)]


FRAC_PREP_ZOH_INJECTION = 1
FRAC_PREP_NO_SOFTMAX = 2
FRAC_PREP_NO_READ_PRIOR = 4
FRAC_PREP_NO_WRITE_PRIOR = 8
FRAC_PREP_ALPHA_ONE = 16


class FracConvDims(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int64), ("seqlen", ctypes.c_int64),
                ("channels", ctypes.c_int64), ("width", ctypes.c_int64),
                ("dtype", ctypes.c_int32), ("flags", ctypes.c_int32)]


FRAC_CONV_SILU = 1


class FracNormDims(ctypes.Structure):
    _fields_ = [("rows", ctypes.c_int64), ("dim", ctypes.c_int64),
                ("group_size", ctypes.c_int64), ("eps", ctypes.c_float),
                ("dtype", ctypes.c_int32), ("flags", ctypes.c_int32)]


class FracTraceEntry(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 64), ("launches", ctypes.c_int32),
                ("total_ms", ctypes.c_double)]


class FracError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str):
        super().__init__(f"{where} failed with status {status}: {detail}")
        self.status = status


def library_path() -> str:
    return _build.LIB_PATH


def load(build_if_missing: bool = True) -> ctypes.CDLL:
    """Load (building first if needed) the in-tree libfrac.so."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = _build.LIB_PATH
        if build_if_missing and not _build.up_to_date():
            _build.build()
        if not os.path.exists(path):
            raise RuntimeError(f"libfrac.so not found at {path}; run paper_2609_36314_gb300.build")
        lib = ctypes.CDLL(path)
        P = ctypes.c_void_p
        dims_p = ctypes.POINTER(FracDims)
        st = ctypes.c_int
        lib.frac_scan_fwd_workspace_size.argtypes = [dims_p, ctypes.POINTER(ctypes.c_size_t)]
        lib.frac_scan_fwd_workspace_size.restype = st
        lib.frac_scan_bwd_workspace_size.argtypes = [dims_p, ctypes.POINTER(ctypes.c_size_t)]
        lib.frac_scan_bwd_workspace_size.restype = st
        lib.frac_scan_fwd.argtypes = [dims_p] + [P] * 13 + [P, ctypes.c_size_t, P]
        lib.frac_scan_fwd.restype = st
        lib.frac_scan_bwd.argtypes = [dims_p] + [P] * 24 + [P, ctypes.c_size_t, P]
        lib.frac_scan_bwd.restype = st
        lib.frac_decode_step.argtypes = [dims_p] + [P] * 12 + [P]
        lib.frac_decode_step.restype = st
        lib.frac_scan_fwd_static.argtypes = [dims_p] + [P] * 13 + [P]
        lib.frac_scan_fwd_static.restype = st
        lib.frac_scan_fwd_static_status.argtypes = [P]
        lib.frac_scan_fwd_static_status.restype = st
        cfg_p = ctypes.POINTER(FracPrepConfig)
        lib.frac_param_prep_fwd.argtypes = [dims_p, cfg_p] + [P] * 12 + [P]
        lib.frac_param_prep_fwd.restype = st
        lib.frac_param_prep_bwd.argtypes = [dims_p, cfg_p] + [P] * 19 + [P]
        lib.frac_param_prep_bwd.restype = st
        conv_p = ctypes.POINTER(FracConvDims)
        norm_p = ctypes.POINTER(FracNormDims)
        lib.frac_conv1d_fwd.argtypes = [conv_p] + [P] * 6 + [P]
        lib.frac_conv1d_fwd.restype = st
        lib.frac_conv1d_bwd.argtypes = [conv_p] + [P] * 9 + [P]
        lib.frac_conv1d_bwd.restype = st
        lib.frac_conv1d_step.argtypes = [conv_p] + [P] * 5 + [P]
        lib.frac_conv1d_step.restype = st
        lib.frac_gated_rmsnorm_fwd.argtypes = [norm_p] + [P] * 4 + [P]
        lib.frac_gated_rmsnorm_fwd.restype = st
        lib.frac_gated_rmsnorm_bwd.argtypes = [norm_p] + [P] * 7 + [P]
        lib.frac_gated_rmsnorm_bwd.restype = st
        lib.frac_workspace_status.argtypes = [P, P]
        lib.frac_workspace_status.restype = st
        lib.frac_trace_enable.argtypes = [ctypes.c_int]
        lib.frac_trace_enable.restype = st
        lib.frac_trace_collect.argtypes = [ctypes.POINTER(FracTraceEntry), ctypes.c_int,
                                           ctypes.POINTER(ctypes.c_int)]
        lib.frac_trace_collect.restype = st
        lib.frac_trace_reset.argtypes = []
        lib.frac_trace_reset.restype = st
        lib.frac_status_string.argtypes = [st]
        lib.frac_status_string.restype = ctypes.c_char_p
        lib.frac_last_error.argtypes = []
        lib.frac_last_error.restype = ctypes.c_char_p
        _lib = lib
        return lib


def check(status: int, where: str) -> None:
    if status != FRAC_OK:
        lib = load()
        raise FracError(status, where, lib.frac_last_error().decode() or
                        lib.frac_status_string(status).decode())


def trace_enable(on: bool) -> None:
    load().frac_trace_enable(1 if on else 0)


def trace_reset() -> None:
    load().frac_trace_reset()


def trace_collect() -> dict:
    """{kernel name: (launches, total_ms)} recorded since the last reset (waits for the events)."""
    lib = load()
    n = ctypes.c_int(0)
    lib.frac_trace_collect(None, 0, ctypes.byref(n))
    buf = (FracTraceEntry * max(1, n.value))()
    lib.frac_trace_collect(buf, n.value, ctypes.byref(n))
    return {buf[i].name.decode(): (int(buf[i].launches), float(buf[i].total_ms))
            for i in range(n.value)}
