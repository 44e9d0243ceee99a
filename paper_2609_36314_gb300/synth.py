"""Seeded synthetic inputs for the Frac scan (host, numpy).

This module holds input recipes only -- no step of the scan itself.  The same
host arrays feed the CUDA path and the fp64 oracle, so both see identical bytes.

Recipe (one independent numpy PCG64 stream per tensor, keyed by (seed, tensor id)):
  x, B, C, dy ~ N(0, 1)
  Delta  = clip(softplus(z - shift), 1e-4, 1),  z ~ N(0,1); shift 1 (3 for the
           long-context prefill workload).  The clip range is the paper's
           (language-modelling setup, App. E.3).
  alpha  = sigmoid(z)                           (Sec. 3.3: sigmoid keeps alpha in (0,1))
  lambda = clip(softplus(z), 0.25, 4)           (Sec. 3.3 softplus; clip of App. E.3)
  tau_m  = 2^(17 (m-1)/(K-1)), m = 1..K         (geometric bank from 1 to 2^17, App. E.3;
                                                 endpoints included)
  w_read, w_write = softmax_m(-alpha ln tau_m + 0.5 z_m),  z ~ N(0,1) i.i.d.
           (Eq. read-softmax with the log-timescale prior; the learned logit maps
            are replaced by sigma(0) * z = 0.5 z.)
  D ~ N(0, 1) per head.
bf16 tensors are rounded once, round-to-nearest-even, from the float32 draw and
kept as uint16 bit patterns; ``to_f64`` widens them exactly for the oracle.
"""
from __future__ import annotations

import dataclasses


import numpy as np

# tensor ids for the per-tensor streams
_IDS = dict(x=0, dt=1, alpha=2, lam=3, B=4, C=5, w_read=6, w_write=7, D=8, dy=9, h0=10,
            dh_final=11, up_dt=12, up_alpha=13, up_lam=14, up_w_read=15, up_w_write=16,
            u=17, conv_w=18, conv_b=19, z=20, norm_w=21, dout=22, conv_state=23)


@dataclasses.dataclass(frozen=True)
class Shape:
    batch: int
    seqlen: int
    nheads: int
    headdim: int
    ngroups: int
    dstate: int
    nmodes: int
    chunk: int
    dtype: str          # "f32" or "bf16": dtype of x, B, C, w_read, w_write, y and their grads
    dt_shift: float = 1.0

    def replace(self, **kw):
        return dataclasses.replace(self, **kw)


# The five workloads (synthetic, seed 0).
WORKLOADS = {
    "fwd_f32_small": Shape(1, 256, 2, 32, 1, 16, 4, 64, "f32"),
    "fwd_bf16_b4_l2048": Shape(4, 2048, 16, 64, 1, 64, 8, 128, "bf16"),
    "train_bf16_b8_l4096": Shape(8, 4096, 64, 64, 1, 128, 8, 0, "bf16"),
    "prefill_bf16_l65536": Shape(1, 65536, 64, 64, 1, 128, 8, 256, "bf16", dt_shift=3.0),
    # decode: 512-token prefill then 1024 single-token steps
    "decode_b128": Shape(128, 512, 64, 64, 1, 128, 8, 0, "bf16"),
}
DECODE_STEPS = 1024


def rng_for(seed: int, name: str, sub: int = 0) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, _IDS[name], sub])))


def normal(seed: int, name: str, shape, sub: int = 0) -> np.ndarray:
    return rng_for(seed, name, sub).standard_normal(size=shape, dtype=np.float32)


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round float32 to bfloat16 (nearest even); returns uint16 bit patterns."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)
    rounding = ((u >> 16) & 1) + np.uint32(0x7FFF)
    out = ((u + rounding) >> 16).astype(np.uint16)
    nan = np.isnan(a)
    if nan.any():
        out[nan] = 0x7FC0
    return out


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def to_f64(a: np.ndarray) -> np.ndarray:
    """Widen a host tensor (float32, float64 or bf16 bits) to float64 exactly."""
    if a.dtype == np.uint16:
        return bf16_bits_to_f32(a).astype(np.float64)
    return a.astype(np.float64)


def cast(a: np.ndarray, dtype: str) -> np.ndarray:
    if dtype == "bf16":
        return f32_to_bf16_bits(a.astype(np.float32))
    if dtype == "f32":
        return np.ascontiguousarray(a, dtype=np.float32)
    raise ValueError(dtype)


def softplus(z):
    return np.logaddexp(0.0, z)


def timescales(nmodes: int, nheads: int) -> np.ndarray:
    """Geometric bank from 1 to 2^17 inclusive, the same for every head: [H, K] float32."""
    if nmodes == 1:
        t = np.ones(1)
    else:
        t = 2.0 ** (17.0 * np.arange(nmodes) / (nmodes - 1))
    return np.ascontiguousarray(np.broadcast_to(t.astype(np.float32), (nheads, nmodes)))


def mode_weights(alpha: np.ndarray, tau: np.ndarray, z: np.ndarray) -> np.ndarray:
    """softmax_m(-alpha ln tau_m + 0.5 z_m) in fp64; alpha [..., H], tau [H, K], z [..., H, K]."""
    logits = -alpha.astype(np.float64)[..., None] * np.log(tau.astype(np.float64)) + 0.5 * z
    logits -= logits.max(axis=-1, keepdims=True)
    w = np.exp(logits)
    return w / w.sum(axis=-1, keepdims=True)


def controls(seed: int, shape_blh, dt_shift: float):
    """Delta, alpha, lambda as float32 arrays of shape shape_blh."""
    dt = np.clip(softplus(normal(seed, "dt", shape_blh).astype(np.float64) - dt_shift), 1e-4, 1.0)
    alpha = 1.0 / (1.0 + np.exp(-normal(seed, "alpha", shape_blh).astype(np.float64)))
    lam = np.clip(softplus(normal(seed, "lam", shape_blh).astype(np.float64)), 0.25, 4.0)
    return dt.astype(np.float32), alpha.astype(np.float32), lam.astype(np.float32)


def make_scan_inputs(s: Shape, seed: int = 0, with_dy: bool = False, with_h0: bool = False,
                     with_dh_final: bool = False) -> dict:
    """Inputs of one scan call, in the dtypes the C-ABI takes (bf16 as uint16 bits)."""
    Bz, L, H, P, G, N, K = s.batch, s.seqlen, s.nheads, s.headdim, s.ngroups, s.dstate, s.nmodes
    dt, alpha, lam = controls(seed, (Bz, L, H), s.dt_shift)
    tau = timescales(K, H)
    out = dict(
        x=cast(normal(seed, "x", (Bz, L, H, P)), s.dtype),
        dt=dt, alpha=alpha, lam=lam, tau=tau,
        B=cast(normal(seed, "B", (Bz, L, G, N)), s.dtype),
        C=cast(normal(seed, "C", (Bz, L, G, N)), s.dtype),
        w_read=cast(mode_weights(alpha, tau, normal(seed, "w_read", (Bz, L, H, K))), s.dtype),
        w_write=cast(mode_weights(alpha, tau, normal(seed, "w_write", (Bz, L, H, K))), s.dtype),
        D=normal(seed, "D", (H,)),
    )
    if with_dy:
        out["dy"] = cast(normal(seed, "dy", (Bz, L, H, P)), s.dtype)
    if with_h0:
        out["h0"] = (0.5 * normal(seed, "h0", (Bz, H, K, P, N))).astype(np.float32)
    if with_dh_final:
        out["dh_final"] = (0.5 * normal(seed, "dh_final", (Bz, H, K, P, N))).astype(np.float32)
    return out


def make_decode_inputs(s: Shape, steps: int, seed: int = 0) -> dict:
    """Per-step decode inputs, stacked over steps: x_t [T,B,H,P], B_t/C_t [T,B,G,N], ..."""
    Bz, H, P, G, N, K = s.batch, s.nheads, s.headdim, s.ngroups, s.dstate, s.nmodes
    sub = 1  # a separate stream family from the prefill inputs
    dt = np.clip(softplus(normal(seed, "dt", (steps, Bz, H), sub).astype(np.float64) - s.dt_shift),
                 1e-4, 1.0).astype(np.float32)
    alpha = (1.0 / (1.0 + np.exp(-normal(seed, "alpha", (steps, Bz, H), sub).astype(np.float64)))
             ).astype(np.float32)
    lam = np.clip(softplus(normal(seed, "lam", (steps, Bz, H), sub).astype(np.float64)),
                  0.25, 4.0).astype(np.float32)
    tau = timescales(K, H)
    return dict(
        x=cast(normal(seed, "x", (steps, Bz, H, P), sub), s.dtype),
        dt=dt, alpha=alpha, lam=lam, tau=tau,
        B=cast(normal(seed, "B", (steps, Bz, G, N), sub), s.dtype),
        C=cast(normal(seed, "C", (steps, Bz, G, N), sub), s.dtype),
        w_read=cast(mode_weights(alpha, tau, normal(seed, "w_read", (steps, Bz, H, K), sub)), s.dtype),
        w_write=cast(mode_weights(alpha, tau, normal(seed, "w_write", (steps, Bz, H, K), sub)), s.dtype),
        D=normal(seed, "D", (H,)),
    )


def make_prep_inputs(s: Shape, seed: int = 0, with_grads: bool = False) -> dict:
    """Inputs of the scan-parameter construction with the same distributions as the scan recipe
    above: the raw controls are the z draws (Delta's shift is the per-head bias), the logits
    0.5 z (sigma(0) z).  With with_grads, upstream gradients of its five outputs ~ N(0, 1)."""
    Bz, L, H, K = s.batch, s.seqlen, s.nheads, s.nmodes
    out = dict(
        dt_raw=normal(seed, "dt", (Bz, L, H)),
        alpha_raw=normal(seed, "alpha", (Bz, L, H)),
        lam_raw=normal(seed, "lam", (Bz, L, H)),
        g_read=cast(0.5 * normal(seed, "w_read", (Bz, L, H, K)), s.dtype),
        g_write=cast(0.5 * normal(seed, "w_write", (Bz, L, H, K)), s.dtype),
        tau=timescales(K, H),
        dt_bias=np.full((H,), -s.dt_shift, dtype=np.float32),
    )
    if with_grads:
        out.update(
            ddt=normal(seed, "up_dt", (Bz, L, H)), dalpha=normal(seed, "up_alpha", (Bz, L, H)),
            dlam=normal(seed, "up_lam", (Bz, L, H)),
            dw_read=cast(normal(seed, "up_w_read", (Bz, L, H, K)), s.dtype),
            dw_write=cast(normal(seed, "up_w_write", (Bz, L, H, K)), s.dtype))
    return out


def make_conv_inputs(batch, seqlen, channels, width, dtype, seed=0, with_state=True):
    """Inputs of the causal conv1d: x, du ~ N(0,1) [B, L, C] and a carried state ~ N(0,1)
    [B, C, W-1] in dtype; w ~ N(0, 1/W) [C, W] and bias ~ N(0, 0.01) [C] in float32."""
    out = dict(
        x=cast(normal(seed, "u", (batch, seqlen, channels)), dtype),
        w=(normal(seed, "conv_w", (channels, width)) / np.sqrt(width)).astype(np.float32),
        bias=(0.1 * normal(seed, "conv_b", (channels,))).astype(np.float32),
        du=cast(normal(seed, "dout", (batch, seqlen, channels)), dtype))
    if with_state:
        out["state"] = cast(normal(seed, "conv_state", (batch, channels, width - 1)), dtype)
    return out


def make_norm_inputs(rows, dim, dtype, seed=0):
    """Inputs of the gated RMSNorm: y, z, dout ~ N(0,1) [rows, dim] in dtype; weight
    1 + N(0, 0.01) [dim] in float32."""
    return dict(y=cast(normal(seed, "x", (rows, dim)), dtype), z=cast(normal(seed, "z", (rows, dim)), dtype),
                weight=(1.0 + 0.1 * normal(seed, "norm_w", (dim,))).astype(np.float32),
                dout=cast(normal(seed, "dout", (rows, dim)), dtype))


def rel_l2(a, b) -> float:
    """||a - b||_2 / max(||b||_2, 1e-30), in fp64."""
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    den = max(float(np.linalg.norm(b.ravel())), 1e-30)
    return float(np.linalg.norm((a - b).ravel())) / den


def algorithmic_flops_per_token_head(s: Shape) -> float:
    """State update + readout: 4 K P N."""
    return 4.0 * s.nmodes * s.headdim * s.dstate




def make_scan_inputs_torch(s: Shape, seed: int, device, with_dy: bool = False) -> dict:
    """The same recipe drawn with torch's generator on `device` (fast inputs for timing runs;
    the parity tests use the numpy recipe above so that the oracle reads identical bytes)."""
    import torch
    import torch.nn.functional as F
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    Bz, L, H, P, G, N, K = s.batch, s.seqlen, s.nheads, s.headdim, s.ngroups, s.dstate, s.nmodes
    dty = torch.bfloat16 if s.dtype == "bf16" else torch.float32

    def n(*shape):
        return torch.randn(shape, generator=g, device=device, dtype=torch.float32)

    dt = torch.clamp(F.softplus(n(Bz, L, H) - s.dt_shift), 1e-4, 1.0)
    alpha = torch.sigmoid(n(Bz, L, H))
    lam = torch.clamp(F.softplus(n(Bz, L, H)), 0.25, 4.0)
    tau = torch.from_numpy(timescales(K, H)).to(device)
    ltau = torch.log(tau)

    def weights():
        return torch.softmax(-alpha[..., None] * ltau + 0.5 * n(Bz, L, H, K), dim=-1).to(dty)

    out = dict(x=n(Bz, L, H, P).to(dty), dt=dt, alpha=alpha, lam=lam, tau=tau,
               B=n(Bz, L, G, N).to(dty), C=n(Bz, L, G, N).to(dty), w_read=weights(),
               w_write=weights(), D=n(H))
    if with_dy:
        out["dy"] = n(Bz, L, H, P).to(dty)
    return out
