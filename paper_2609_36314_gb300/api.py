"""Python binding of the Frac scan C ABI (argument marshalling only).

PyTorch provides device memory and the current CUDA stream; every step of the scan
runs in libfrac.so.  Tensors must be CUDA, contiguous, in the dtypes include/frac.h
states (x, B, C, w_read, w_write, y and their gradients in one dtype: float32 or
bfloat16; controls, tau, D and mode states float32).
"""
from __future__ import annotations

import ctypes

import torch

from . import _lib

_DT = {torch.float32: _lib.FRAC_DTYPE_F32, torch.bfloat16: _lib.FRAC_DTYPE_BF16}


def make_dims(batch, seqlen, nheads, headdim, ngroups, dstate, nmodes, dtype, chunk=0,
              force_simt=False, reuse_fwd_states=False, extra_flags=0) -> _lib.FracDims:
    flags = (_lib.FRAC_FLAG_FORCE_SIMT if force_simt else 0) | (
        _lib.FRAC_FLAG_BWD_REUSE_FWD_STATES if reuse_fwd_states else 0) | int(extra_flags)
    return _lib.FracDims(batch, seqlen, nheads, headdim, ngroups, dstate, nmodes, chunk,
                         _DT[dtype], flags)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _need(t, name, dtype, shape=None):
    if t is None:
        raise ValueError(f"{name} is required")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")
    return t


def _need_out(t, name, dtype, shape):
    """An output the caller supplied: the kernels write exactly `shape` elements of `dtype`."""
    if t is not None:
        _need(t, name, dtype, shape)
    return t


def _need_scan_inputs(x, dt, alpha, lam, tau, B, C, w_read, w_write, D, h0, dims):
    Bz, L, H, P, G, N, K = dims
    dt_, f32 = x.dtype, torch.float32
    _need(x, "x", dt_, (Bz, L, H, P))
    for name, t in (("dt", dt), ("alpha", alpha), ("lam", lam)):
        _need(t, name, f32, (Bz, L, H))
    _need(tau, "tau", f32, (H, K))
    _need(B, "B", dt_, (Bz, L, G, N))
    _need(C, "C", dt_, (Bz, L, G, N))
    _need(w_read, "w_read", dt_, (Bz, L, H, K))
    _need(w_write, "w_write", dt_, (Bz, L, H, K))
    _need(D, "D", f32, (H,))
    if h0 is not None:
        _need(h0, "h0", f32, (Bz, H, K, P, N))


def _scan_dims(x, B, tau, chunk, force_simt, reuse_fwd_states=False):
    if x.dim() != 4 or B.dim() != 4 or tau.dim() != 2:
        raise ValueError("x [B,L,H,P], B/C [B,L,G,N], tau [H,K] expected")
    Bz, L, H, P = x.shape
    G, N = B.shape[2], B.shape[3]
    K = tau.shape[1]
    return (make_dims(Bz, L, H, P, G, N, K, x.dtype, chunk, force_simt, reuse_fwd_states),
            (Bz, L, H, P, G, N, K))


def fwd_workspace_size(dims: _lib.FracDims) -> int:
    n = ctypes.c_size_t(0)
    _lib.check(_lib.load().frac_scan_fwd_workspace_size(ctypes.byref(dims), ctypes.byref(n)),
               "frac_scan_fwd_workspace_size")
    return int(n.value)


def bwd_workspace_size(dims: _lib.FracDims) -> int:
    n = ctypes.c_size_t(0)
    _lib.check(_lib.load().frac_scan_bwd_workspace_size(ctypes.byref(dims), ctypes.byref(n)),
               "frac_scan_bwd_workspace_size")
    return int(n.value)


def _workspace(nbytes, device, given):
    if given is not None:
        if given.numel() * given.element_size() < nbytes:
            raise ValueError("workspace too small")
        return given
    return torch.empty(max(nbytes, 1), dtype=torch.uint8, device=device)


def scan_fwd(x, dt, alpha, lam, tau, B, C, w_read, w_write, D, h0=None, *, chunk=0,
             force_simt=False, want_final_state=True, y=None, h_final=None, workspace=None,
             stream=None):
    """Chunked forward scan.  Returns (y [B,L,H,P], h_final [B,H,K,P,N] or None)."""
    dims, shp = _scan_dims(x, B, tau, chunk, force_simt)
    Bz, L, H, P, G, N, K = shp
    f32 = torch.float32
    _need_scan_inputs(x, dt, alpha, lam, tau, B, C, w_read, w_write, D, h0, shp)
    _need_out(y, "y", x.dtype, (Bz, L, H, P))
    if want_final_state:
        _need_out(h_final, "h_final", f32, (Bz, H, K, P, N))
    if y is None:
        y = torch.empty_like(x)
    if want_final_state and h_final is None:
        h_final = torch.empty((Bz, H, K, P, N), dtype=f32, device=x.device)
    ws = _workspace(fwd_workspace_size(dims), x.device, workspace)
    _lib.check(_lib.load().frac_scan_fwd(
        ctypes.byref(dims), _ptr(x), _ptr(dt), _ptr(alpha), _ptr(lam), _ptr(tau), _ptr(B),
        _ptr(C), _ptr(w_read), _ptr(w_write), _ptr(D), _ptr(h0), _ptr(y),
        _ptr(h_final if want_final_state else None), _ptr(ws), ws.numel(), _stream(stream)),
        "frac_scan_fwd")
    return y, (h_final if want_final_state else None)


def scan_fwd_static(x, dt, alpha, lam, tau, B, C, w_read, w_write, D, h0=None, *, chunk=0,
                    force_simt=False, want_final_state=True, y=None, h_final=None, stream=None):
    """scan_fwd for callers that cannot provide scratch memory: the library's own fixed device
    array (FRAC_SCAN_FWD_STATIC_SCRATCH_BYTES) holds the per-chunk states, so this call
    allocates nothing besides the outputs it is not given.  Calls that overlap on the GPU
    race on that array."""
    dims, shp = _scan_dims(x, B, tau, chunk, force_simt)
    Bz, L, H, P, G, N, K = shp
    _need_scan_inputs(x, dt, alpha, lam, tau, B, C, w_read, w_write, D, h0, shp)
    _need_out(y, "y", x.dtype, (Bz, L, H, P))
    if want_final_state:
        _need_out(h_final, "h_final", torch.float32, (Bz, H, K, P, N))
    if y is None:
        y = torch.empty_like(x)
    if want_final_state and h_final is None:
        h_final = torch.empty((Bz, H, K, P, N), dtype=torch.float32, device=x.device)
    _lib.check(_lib.load().frac_scan_fwd_static(
        ctypes.byref(dims), _ptr(x), _ptr(dt), _ptr(alpha), _ptr(lam), _ptr(tau), _ptr(B),
        _ptr(C), _ptr(w_read), _ptr(w_write), _ptr(D), _ptr(h0), _ptr(y),
        _ptr(h_final if want_final_state else None), _stream(stream)), "frac_scan_fwd_static")
    return y, (h_final if want_final_state else None)


def scan_bwd(x, dt, alpha, lam, tau, B, C, w_read, w_write, D, dy, h0=None, dh_final=None, *,
             chunk=0, force_simt=False, want_dh0=True, want_dtau=False, workspace=None, out=None,
             stream=None, reuse_fwd_states=False):
    """Backward of scan_fwd.  Returns a dict of gradients (dx, ddt, dalpha, dlam, dB, dC,
    dw_read, dw_write, dD, dh0, dtau; dh0 / dtau None when not wanted).  With reuse_fwd_states,
    `workspace` must be the buffer a scan_fwd call on the same inputs just used (sized with
    bwd_workspace_size)."""
    if reuse_fwd_states and workspace is None:
        raise ValueError("reuse_fwd_states needs the workspace of the forward call")
    dims, shp = _scan_dims(x, B, tau, chunk, force_simt, reuse_fwd_states)
    Bz, L, H, P, G, N, K = shp
    dt_ = x.dtype
    f32 = torch.float32
    _need_scan_inputs(x, dt, alpha, lam, tau, B, C, w_read, w_write, D, h0, shp)
    _need(dy, "dy", dt_, (Bz, L, H, P))
    if dh_final is not None:
        _need(dh_final, "dh_final", f32, (Bz, H, K, P, N))
    if out is not None:
        for name, dtype, shape in (("dx", dt_, (Bz, L, H, P)), ("ddt", f32, (Bz, L, H)),
                                   ("dalpha", f32, (Bz, L, H)), ("dlam", f32, (Bz, L, H)),
                                   ("dB", dt_, (Bz, L, G, N)), ("dC", dt_, (Bz, L, G, N)),
                                   ("dw_read", dt_, (Bz, L, H, K)), ("dw_write", dt_, (Bz, L, H, K)),
                                   ("dD", f32, (H,))):
            _need(out.get(name), name, dtype, shape)
        _need_out(out.get("dh0"), "dh0", f32, (Bz, H, K, P, N))
        _need_out(out.get("dtau"), "dtau", f32, (H, K))
    g = out if out is not None else dict(
        dx=torch.empty_like(x), ddt=torch.empty_like(dt), dalpha=torch.empty_like(alpha),
        dlam=torch.empty_like(lam), dB=torch.empty_like(B), dC=torch.empty_like(C),
        dw_read=torch.empty_like(w_read), dw_write=torch.empty_like(w_write),
        dD=torch.empty_like(D),
        dh0=torch.empty((Bz, H, K, P, N), dtype=f32, device=x.device) if want_dh0 else None,
        dtau=torch.empty((H, K), dtype=f32, device=x.device) if want_dtau else None)
    ws = _workspace(bwd_workspace_size(dims), x.device, workspace)
    _lib.check(_lib.load().frac_scan_bwd(
        ctypes.byref(dims), _ptr(x), _ptr(dt), _ptr(alpha), _ptr(lam), _ptr(tau), _ptr(B),
        _ptr(C), _ptr(w_read), _ptr(w_write), _ptr(D), _ptr(h0), _ptr(dy), _ptr(dh_final),
        _ptr(g["dx"]), _ptr(g["ddt"]), _ptr(g["dalpha"]), _ptr(g["dlam"]), _ptr(g["dB"]),
        _ptr(g["dC"]), _ptr(g["dw_read"]), _ptr(g["dw_write"]), _ptr(g["dD"]),
        _ptr(g.get("dh0")), _ptr(g.get("dtau")), _ptr(ws), ws.numel(), _stream(stream)),
        "frac_scan_bwd")
    return g


def decode_step(x_t, dt, alpha, lam, tau, B_t, C_t, w_read, w_write, D, state, y_t=None,
                stream=None):
    """One decode step: updates `state` in place and returns y_t [B,H,P]."""
    if x_t.dim() != 3 or B_t.dim() != 3:
        raise ValueError("x_t [B,H,P], B_t/C_t [B,G,N] expected")
    Bz, H, P = x_t.shape
    G, N = B_t.shape[1], B_t.shape[2]
    K = tau.shape[1]
    dt_ = x_t.dtype
    f32 = torch.float32
    _need(x_t, "x_t", dt_)
    _need(B_t, "B_t", dt_, (Bz, G, N))
    _need(C_t, "C_t", dt_, (Bz, G, N))
    _need(w_read, "w_read", dt_, (Bz, H, K))
    _need(w_write, "w_write", dt_, (Bz, H, K))
    for name, t in (("dt", dt), ("alpha", alpha), ("lam", lam)):
        _need(t, name, f32, (Bz, H))
    _need(tau, "tau", f32, (H, K))
    _need(D, "D", f32, (H,))
    _need(state, "state", f32, (Bz, H, K, P, N))
    _need_out(y_t, "y_t", dt_, (Bz, H, P))
    if y_t is None:
        y_t = torch.empty_like(x_t)
    dims = make_dims(Bz, 1, H, P, G, N, K, dt_)
    _lib.check(_lib.load().frac_decode_step(
        ctypes.byref(dims), _ptr(x_t), _ptr(dt), _ptr(alpha), _ptr(lam), _ptr(tau), _ptr(B_t),
        _ptr(C_t), _ptr(w_read), _ptr(w_write), _ptr(D), _ptr(state), _ptr(y_t),
        _stream(stream)), "frac_decode_step")
    return y_t


def prep_config(dt_min=1e-4, dt_max=1.0, lam_min=0.25, lam_max=4.0, zoh_injection=False,
                no_softmax=False, no_read_prior=False, no_write_prior=False,
                alpha_one=False) -> _lib.FracPrepConfig:
    """Clip ranges (defaults: the language-modelling setting) and variant flags of the
    scan-parameter construction."""
    flags = ((_lib.FRAC_PREP_ZOH_INJECTION if zoh_injection else 0) |
             (_lib.FRAC_PREP_NO_SOFTMAX if no_softmax else 0) |
             (_lib.FRAC_PREP_NO_READ_PRIOR if no_read_prior else 0) |
             (_lib.FRAC_PREP_NO_WRITE_PRIOR if no_write_prior else 0) |
             (_lib.FRAC_PREP_ALPHA_ONE if alpha_one else 0))
    return _lib.FracPrepConfig(dt_min, dt_max, lam_min, lam_max, flags, 0)


def _prep_dims(dt_raw, g_read, tau):
    if dt_raw.dim() < 1 or g_read.dim() != dt_raw.dim() + 1 or tau.dim() != 2:
        raise ValueError("dt_raw [..., H], g_read [..., H, K], tau [H, K] expected")
    H, K = tau.shape
    if dt_raw.shape[-1] != H or g_read.shape[-1] != K or tuple(g_read.shape[:-1]) != tuple(dt_raw.shape):
        raise ValueError("dt_raw [..., H], g_read [..., H, K] (the same leading dims) and tau [H, K] expected")
    rows = dt_raw.numel() // H
    return make_dims(1, rows, H, 1, 1, 1, K, g_read.dtype)


def _need_prep_inputs(dt_raw, alpha_raw, lam_raw, g_read, g_write, tau, dt_bias):
    f32 = torch.float32
    _need(dt_raw, "dt_raw", f32)
    _need(tau, "tau", f32)
    if alpha_raw is not None:
        _need(alpha_raw, "alpha_raw", f32, dt_raw.shape)
    _need(lam_raw, "lam_raw", f32, dt_raw.shape)
    _need(g_read, "g_read", g_read.dtype)
    _need(g_write, "g_write", g_read.dtype, g_read.shape)
    if dt_bias is not None:
        _need(dt_bias, "dt_bias", f32, (tau.shape[0],))


def param_prep_fwd(dt_raw, alpha_raw, lam_raw, g_read, g_write, tau, dt_bias=None, cfg=None,
                   out=None, stream=None):
    """Scan controls and mode weights from the projections' outputs.  Returns a dict with
    dt, alpha, lam (float32, shape of dt_raw) and w_read, w_write (dtype of g_read)."""
    cfg = cfg or prep_config()
    dims = _prep_dims(dt_raw, g_read, tau)
    f32 = torch.float32
    _need_prep_inputs(dt_raw, alpha_raw, lam_raw, g_read, g_write, tau, dt_bias)
    if out is not None:
        for name in ("dt", "alpha", "lam"):
            _need(out.get(name), name, f32, dt_raw.shape)
        for name in ("w_read", "w_write"):
            _need(out.get(name), name, g_read.dtype, g_read.shape)
    o = out if out is not None else dict(
        dt=torch.empty_like(dt_raw), alpha=torch.empty_like(dt_raw), lam=torch.empty_like(dt_raw),
        w_read=torch.empty_like(g_read), w_write=torch.empty_like(g_read))
    _lib.check(_lib.load().frac_param_prep_fwd(
        ctypes.byref(dims), ctypes.byref(cfg), _ptr(dt_raw), _ptr(dt_bias), _ptr(alpha_raw),
        _ptr(lam_raw), _ptr(g_read), _ptr(g_write), _ptr(tau), _ptr(o["dt"]), _ptr(o["alpha"]),
        _ptr(o["lam"]), _ptr(o["w_read"]), _ptr(o["w_write"]), _stream(stream)),
        "frac_param_prep_fwd")
    return o


def param_prep_bwd(dt_raw, alpha_raw, lam_raw, g_read, g_write, tau, ddt, dalpha, dlam, dw_read,
                   dw_write, dt_bias=None, cfg=None, want_dt_bias=True, want_dtau=True,
                   stream=None):
    """Backward of param_prep_fwd.  Returns a dict with ddt_raw, dalpha_raw, dlam_raw,
    dg_read, dg_write, and ddt_bias [H] / dtau [H, K] (None when not wanted)."""
    cfg = cfg or prep_config()
    dims = _prep_dims(dt_raw, g_read, tau)
    f32 = torch.float32
    _need_prep_inputs(dt_raw, alpha_raw, lam_raw, g_read, g_write, tau, dt_bias)
    for name, t in (("ddt", ddt), ("dalpha", dalpha), ("dlam", dlam)):
        _need(t, name, f32, dt_raw.shape)
    for name, t in (("dw_read", dw_read), ("dw_write", dw_write)):
        _need(t, name, g_read.dtype, g_read.shape)
    H, K = tau.shape
    g = dict(ddt_raw=torch.empty_like(dt_raw), dalpha_raw=torch.empty_like(dt_raw),
             dlam_raw=torch.empty_like(dt_raw), dg_read=torch.empty_like(g_read),
             dg_write=torch.empty_like(g_read),
             ddt_bias=torch.empty(H, dtype=f32, device=tau.device) if want_dt_bias else None,
             dtau=torch.empty((H, K), dtype=f32, device=tau.device) if want_dtau else None)
    _lib.check(_lib.load().frac_param_prep_bwd(
        ctypes.byref(dims), ctypes.byref(cfg), _ptr(dt_raw), _ptr(dt_bias), _ptr(alpha_raw),
        _ptr(lam_raw), _ptr(g_read), _ptr(g_write), _ptr(tau), _ptr(ddt), _ptr(dalpha),
        _ptr(dlam), _ptr(dw_read), _ptr(dw_write), _ptr(g["ddt_raw"]), _ptr(g["dalpha_raw"]),
        _ptr(g["dlam_raw"]), _ptr(g["dg_read"]), _ptr(g["dg_write"]), _ptr(g["ddt_bias"]),
        _ptr(g["dtau"]), _stream(stream)), "frac_param_prep_bwd")
    return g


# ----------------------------------------------------------------------------- mixer glue
def _conv_dims(x, w, silu):
    if x.dim() != 3 or w.dim() != 2 or w.shape[0] != x.shape[2]:
        raise ValueError("x [B, L, C], w [C, W] expected")
    return _lib.FracConvDims(x.shape[0], x.shape[1], x.shape[2], w.shape[1], _DT[x.dtype],
                             _lib.FRAC_CONV_SILU if silu else 0)


def _need_conv_inputs(x, w, bias, state):
    B, L, C = x.shape
    W = w.shape[1]
    _need(x, "x", x.dtype)
    _need(w, "w", torch.float32, (C, W))
    if bias is not None:
        _need(bias, "bias", torch.float32, (C,))
    if state is not None:
        _need(state, "state", x.dtype, (B, C, W - 1))
    return B, L, C, W


def conv1d_fwd(x, w, bias=None, state=None, *, silu=False, want_state=False, stream=None):
    """Depthwise causal conv1d over [B, L, C] (optionally SiLU).  Returns (u, final state
    [B, C, W-1] or None)."""
    dims = _conv_dims(x, w, silu)
    B, L, C, W = _need_conv_inputs(x, w, bias, state)
    u = torch.empty_like(x)
    fin = torch.empty((B, C, W - 1), dtype=x.dtype, device=x.device) if want_state else None
    _lib.check(_lib.load().frac_conv1d_fwd(ctypes.byref(dims), _ptr(x), _ptr(w), _ptr(bias),
                                           _ptr(state), _ptr(u), _ptr(fin), _stream(stream)),
               "frac_conv1d_fwd")
    return u, fin


def conv1d_bwd(x, w, du, bias=None, state=None, *, silu=False, want_dstate=False, stream=None):
    """Backward of conv1d_fwd.  Returns dict(dx, dw, dbias, dstate)."""
    dims = _conv_dims(x, w, silu)
    B, L, C, W = _need_conv_inputs(x, w, bias, state)
    _need(du, "du", x.dtype, x.shape)
    g = dict(dx=torch.empty_like(x), dw=torch.empty_like(w),
             dbias=torch.empty(C, dtype=torch.float32, device=x.device) if bias is not None else None,
             dstate=torch.empty((B, C, W - 1), dtype=x.dtype, device=x.device) if want_dstate else None)
    _lib.check(_lib.load().frac_conv1d_bwd(
        ctypes.byref(dims), _ptr(x), _ptr(w), _ptr(bias), _ptr(state), _ptr(du), _ptr(g["dx"]),
        _ptr(g["dw"]), _ptr(g["dbias"]), _ptr(g["dstate"]), _stream(stream)), "frac_conv1d_bwd")
    return g


def conv1d_step(x_t, w, state, bias=None, *, silu=False, u_t=None, stream=None):
    """One decode step of the conv: x_t [B, C]; state [B, C, W-1] shifts in place."""
    if x_t.dim() != 2 or w.dim() != 2:
        raise ValueError("x_t [B, C], w [C, W] expected")
    B, C = x_t.shape
    W = w.shape[1]
    _need(x_t, "x_t", x_t.dtype)
    _need(w, "w", torch.float32, (C, W))
    if bias is not None:
        _need(bias, "bias", torch.float32, (C,))
    _need(state, "state", x_t.dtype, (B, C, W - 1))
    _need_out(u_t, "u_t", x_t.dtype, (B, C))
    dims = _lib.FracConvDims(B, 1, C, W, _DT[x_t.dtype], _lib.FRAC_CONV_SILU if silu else 0)
    if u_t is None:
        u_t = torch.empty_like(x_t)
    _lib.check(_lib.load().frac_conv1d_step(ctypes.byref(dims), _ptr(x_t), _ptr(w), _ptr(bias),
                                            _ptr(state), _ptr(u_t), _stream(stream)),
               "frac_conv1d_step")
    return u_t


def _norm_dims(y, group_size, eps):
    if y.dim() != 2:
        raise ValueError("y [rows, dim] expected")
    R, D = y.shape
    return _lib.FracNormDims(R, D, group_size or D, float(eps), _DT[y.dtype], 0)


def gated_rmsnorm_fwd(y, z, weight, group_size=0, eps=1e-5, stream=None):
    """RMSNorm(y * silu(z)) * weight over groups of group_size features (0: the whole row)."""
    dims = _norm_dims(y, group_size, eps)
    _need(y, "y", y.dtype)
    if z is not None:
        _need(z, "z", y.dtype, y.shape)
    _need(weight, "weight", torch.float32, (y.shape[1],))
    out = torch.empty_like(y)
    _lib.check(_lib.load().frac_gated_rmsnorm_fwd(ctypes.byref(dims), _ptr(y), _ptr(z),
                                                  _ptr(weight), _ptr(out), _stream(stream)),
               "frac_gated_rmsnorm_fwd")
    return out


def gated_rmsnorm_bwd(y, z, weight, dout, group_size=0, eps=1e-5, stream=None):
    """Backward of gated_rmsnorm_fwd.  Returns dict(dy, dz, dweight)."""
    dims = _norm_dims(y, group_size, eps)
    _need(y, "y", y.dtype)
    if z is not None:
        _need(z, "z", y.dtype, y.shape)
    _need(weight, "weight", torch.float32, (y.shape[1],))
    _need(dout, "dout", y.dtype, y.shape)
    g = dict(dy=torch.empty_like(y), dz=torch.empty_like(y) if z is not None else None,
             dweight=torch.empty_like(weight))
    _lib.check(_lib.load().frac_gated_rmsnorm_bwd(
        ctypes.byref(dims), _ptr(y), _ptr(z), _ptr(weight), _ptr(dout), _ptr(g["dy"]),
        _ptr(g["dz"]), _ptr(g["dweight"]), _stream(stream)), "frac_gated_rmsnorm_bwd")
    return g
