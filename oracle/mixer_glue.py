"""fp64 CPU oracle of the two FracMixer operations around the scan, and their backwards.

TEST INFRASTRUCTURE ONLY: imported by tests/, ``__graft_entry__.smoke()`` and bench.py's
``cpu_baseline`` leg.  Nothing in the product path imports it, and it imports nothing from the
product path.

1. Depthwise causal 1-D convolution along the sequence (Sec. 3.3: the content branch produces
   u_t by a local depthwise causal convolution; width d_conv = 4 in App. E.2 and E.4):
       pre[b, t, c] = bias_c + sum_{j=0}^{W-1} w[c, j] x[b, t - (W-1) + j, c]
   where positions before the sequence start read the W-1 previous inputs of a carried state
   (zeros by default), and u = pre, or u = silu(pre) with the activation on.  The paper names
   only the convolution; the SiLU after it is the convention of the Mamba-family mixers the
   layer follows (Sec. 3.3), kept as an option.  One decode step is the same with the state
   window shifted by one input.
2. Gated RMS normalisation of the scan output (Sec. 3.3: "gated normalization" before the output
   projection), read as the Mamba2 form: with v = y * silu(z) (or v = y without a gate),
       out = v / sqrt(mean_group(v^2) + eps) * weight
   the mean taken over consecutive groups of `group_size` features of each row.

silu(a) = a * sigmoid(a).  Layouts: x, u [B, L, C]; w [C, W]; bias [C]; state [B, C, W-1]
(oldest input first); y, z, out [rows, D]; weight [D].
"""
from __future__ import annotations

import numpy as np


def _sigmoid(a):
    a = np.asarray(a, dtype=np.float64)
    e = np.exp(-np.abs(a))
    return np.where(a >= 0, 1.0 / (1.0 + e), e / (1.0 + e))


def silu(a):
    return a * _sigmoid(a)


def silu_grad(a):
    s = _sigmoid(a)
    return s * (1.0 + a * (1.0 - s))


def _padded(x, state):
    """[B, W-1 + L, C]: the carried inputs (state, oldest first) then the sequence."""
    Bz, L, C = x.shape
    W1 = state.shape[2]
    return np.concatenate([np.transpose(state, (0, 2, 1)), x], axis=1)


def conv1d_fwd(x, w, bias=None, state=None, activation=False):
    """Returns (u [B, L, C], final state [B, C, W-1])."""
    x = np.asarray(x, np.float64)
    w = np.asarray(w, np.float64)
    Bz, L, C = x.shape
    W = w.shape[1]
    st = np.zeros((Bz, C, W - 1)) if state is None else np.asarray(state, np.float64)
    xp = _padded(x, st)
    pre = np.zeros((Bz, L, C)) + (0.0 if bias is None else np.asarray(bias, np.float64))
    for j in range(W):                       # tap j reads input t - (W-1) + j
        pre += w[:, j] * xp[:, j:j + L, :]
    u = silu(pre) if activation else pre
    final = np.transpose(xp[:, L:L + W - 1, :], (0, 2, 1)).copy()
    return u, final


def conv1d_bwd(x, w, du, bias=None, state=None, activation=False):
    """Returns dict(dx, dw, dbias, dstate): the adjoint of conv1d_fwd's u (its final state is
    a copy of inputs and carries no upstream gradient here)."""
    x = np.asarray(x, np.float64)
    w = np.asarray(w, np.float64)
    du = np.asarray(du, np.float64)
    Bz, L, C = x.shape
    W = w.shape[1]
    st = np.zeros((Bz, C, W - 1)) if state is None else np.asarray(state, np.float64)
    xp = _padded(x, st)
    pre = np.zeros((Bz, L, C)) + (0.0 if bias is None else np.asarray(bias, np.float64))
    for j in range(W):
        pre += w[:, j] * xp[:, j:j + L, :]
    g = du * silu_grad(pre) if activation else du
    dxp = np.zeros_like(xp)
    dw = np.zeros_like(w)
    for j in range(W):
        dxp[:, j:j + L, :] += w[:, j] * g
        dw[:, j] = np.sum(g * xp[:, j:j + L, :], axis=(0, 1))
    return dict(dx=dxp[:, W - 1:], dw=dw, dbias=g.sum(axis=(0, 1)),
                dstate=np.transpose(dxp[:, :W - 1], (0, 2, 1)).copy())


def conv1d_step(x_t, w, state, bias=None, activation=False):
    """One decode step: x_t [B, C], state [B, C, W-1] -> (u_t [B, C], new state)."""
    u, final = conv1d_fwd(np.asarray(x_t, np.float64)[:, None, :], w, bias, state, activation)
    return u[:, 0], final


def gated_rmsnorm_fwd(y, z, weight, group_size, eps=1e-5):
    y = np.asarray(y, np.float64)
    v = y * silu(np.asarray(z, np.float64)) if z is not None else y
    R, D = v.shape
    vg = v.reshape(R, D // group_size, group_size)
    r = np.sqrt(np.mean(vg * vg, axis=-1, keepdims=True) + eps)
    return (vg / r).reshape(R, D) * np.asarray(weight, np.float64)


def gated_rmsnorm_bwd(y, z, weight, dout, group_size, eps=1e-5):
    """Returns dict(dy, dz, dweight)."""
    y = np.asarray(y, np.float64)
    dout = np.asarray(dout, np.float64)
    weight = np.asarray(weight, np.float64)
    zz = None if z is None else np.asarray(z, np.float64)
    v = y * silu(zz) if zz is not None else y
    R, D = v.shape
    G = D // group_size
    vg = v.reshape(R, G, group_size)
    r = np.sqrt(np.mean(vg * vg, axis=-1, keepdims=True) + eps)
    n = vg / r
    dn = (dout * weight).reshape(R, G, group_size)
    # n = v / r(v):  dv = (dn - n mean(dn n)) / r
    dv = ((dn - n * np.mean(dn * n, axis=-1, keepdims=True)) / r).reshape(R, D)
    out = dict(dweight=np.sum(dout * n.reshape(R, D), axis=0))
    if zz is None:
        out.update(dy=dv, dz=None)
    else:
        out.update(dy=dv * silu(zz), dz=dv * y * silu_grad(zz))
    return out
