"""fp64 CPU oracle of the Frac scan-parameter construction and its backward.

TEST INFRASTRUCTURE ONLY: imported by tests/, ``__graft_entry__.smoke()`` and bench.py's
``cpu_baseline`` leg.  Nothing in the product path imports it, and it imports nothing from the
product path.

What it computes, per position (b, t) and head h, from the outputs of the layer's projections
(Sec. 3.3 and Algorithm 1 of App. D):

  Delta   = clip(softplus(dt_raw + dt_bias_h), dt_min, dt_max)     Sec. 3.3 (linear projection with
                                                                    learned bias, then softplus);
                                                                    clip range of App. E.3
  alpha   = sigmoid(alpha_raw)                                     Sec. 3.3 (0 < alpha < 1)
  lambda  = clip(softplus(lam_raw), lam_min, lam_max)              Sec. 3.3; clip of App. E.3
  c_{t,m} = softmax_m(-alpha ln tau_m + g_read_{t,m})              Eq. read-softmax
  b_{t,m} = softmax_m(-alpha ln tau_m + g_write_{t,m})             the write weights of Sec. 3.2
                                                                    (same functional form)

g_read / g_write are the mode-wise residual logits (the learned maps applied to the content
signal); they are inputs.  Variants (flags), each an ablation or an alternative the paper
states:
  ZOH_INJECTION   the write weight becomes b / lambda, so that the scan's kappa = (1 - rho) b /
                  lambda is the exact zero-order-hold injection of Eq. rho-beta-def-frac
  NO_SOFTMAX      the weights are the logits themselves, without the softmax (App. G ablation
                  "w/o softmax R/W"; reading: the normalisation is removed, nothing replaces it)
  NO_READ_PRIOR   the read logits omit -alpha ln tau (with NO_WRITE_PRIOR: App. G "pure
                  multiscale bank")
  NO_WRITE_PRIOR  the write logits omit -alpha ln tau (App. G ablation "w/o write prior")
  ALPHA_ONE       alpha = 1 for every token (App. G ablation "alpha = 1")

The backward is the adjoint of the same formulas (chain rule, written out below).  Clipping
passes the gradient where the clipped value lies inside [min, max] (bounds included) and stops
it outside.  Arrays: raw controls [..., H], logits [..., H, K], tau [H, K], dt_bias [H].
"""
from __future__ import annotations

import dataclasses

import numpy as np

ZOH_INJECTION = 1
NO_SOFTMAX = 2
NO_READ_PRIOR = 4
NO_WRITE_PRIOR = 8
ALPHA_ONE = 16


@dataclasses.dataclass(frozen=True)
class PrepConfig:
    dt_min: float = 1e-4   # App. E.3: Delta in [1e-4, 1]
    dt_max: float = 1.0
    lam_min: float = 0.25  # App. E.3: lambda in [0.25, 4]
    lam_max: float = 4.0
    flags: int = 0


def softplus(x):
    """log(1 + e^x), written without overflow: max(x, 0) + log1p(e^-|x|)."""
    x = np.asarray(x, dtype=np.float64)
    return np.maximum(x, 0.0) + np.log1p(np.exp(-np.abs(x)))


def sigmoid(x):
    """1 / (1 + e^-x), written without overflow for either sign of x."""
    x = np.asarray(x, dtype=np.float64)
    e = np.exp(-np.abs(x))
    return np.where(x >= 0, 1.0 / (1.0 + e), e / (1.0 + e))


def _weights(logits, softmax):
    if not softmax:
        return logits.copy()
    z = logits - logits.max(axis=-1, keepdims=True)
    w = np.exp(z)
    return w / w.sum(axis=-1, keepdims=True)


def _f64(a):
    return None if a is None else np.asarray(a, dtype=np.float64)


def prep_fwd(dt_raw, alpha_raw, lam_raw, g_read, g_write, tau, dt_bias=None,
             cfg: PrepConfig = PrepConfig()):
    """Returns dict(dt, alpha, lam, w_read, w_write) in fp64."""
    dt_raw, alpha_raw, lam_raw, g_read, g_write, tau, dt_bias = map(
        _f64, (dt_raw, alpha_raw, lam_raw, g_read, g_write, tau, dt_bias))
    f = cfg.flags
    pre = dt_raw + (dt_bias if dt_bias is not None else 0.0)
    dt = np.clip(softplus(pre), cfg.dt_min, cfg.dt_max)
    alpha = np.ones_like(alpha_raw) if f & ALPHA_ONE else sigmoid(alpha_raw)
    lam = np.clip(softplus(lam_raw), cfg.lam_min, cfg.lam_max)
    prior = -alpha[..., None] * np.log(tau)              # -alpha_t ln tau_m, [..., H, K]
    zr = g_read + (0.0 if f & NO_READ_PRIOR else prior)
    zw = g_write + (0.0 if f & NO_WRITE_PRIOR else prior)
    w_read = _weights(zr, not f & NO_SOFTMAX)
    b = _weights(zw, not f & NO_SOFTMAX)
    w_write = b / lam[..., None] if f & ZOH_INJECTION else b
    return dict(dt=dt, alpha=alpha, lam=lam, w_read=w_read, w_write=w_write)


def _weights_bwd(w, dw, softmax):
    """Adjoint of w = softmax(z) (or w = z): dz_m = w_m (dw_m - sum_j w_j dw_j)."""
    if not softmax:
        return dw.copy()
    return w * (dw - (w * dw).sum(axis=-1, keepdims=True))


def prep_bwd(dt_raw, alpha_raw, lam_raw, g_read, g_write, tau, ddt, dalpha, dlam, dw_read,
             dw_write, dt_bias=None, cfg: PrepConfig = PrepConfig()):
    """Adjoint of prep_fwd.  Returns dict(ddt_raw, dalpha_raw, dlam_raw, dg_read, dg_write,
    ddt_bias [H], dtau [H, K]); dtau is the part that flows through the -alpha ln tau prior."""
    dt_raw, alpha_raw, lam_raw, g_read, g_write, tau, dt_bias = map(
        _f64, (dt_raw, alpha_raw, lam_raw, g_read, g_write, tau, dt_bias))
    ddt, dalpha, dlam, dw_read, dw_write = map(_f64, (ddt, dalpha, dlam, dw_read, dw_write))
    f = cfg.flags
    sm = not f & NO_SOFTMAX
    pre = dt_raw + (dt_bias if dt_bias is not None else 0.0)
    sp_dt = softplus(pre)
    alpha = np.ones_like(alpha_raw) if f & ALPHA_ONE else sigmoid(alpha_raw)
    sp_lam = softplus(lam_raw)
    lam = np.clip(sp_lam, cfg.lam_min, cfg.lam_max)
    ltau = np.log(tau)
    prior = -alpha[..., None] * ltau
    zr = g_read + (0.0 if f & NO_READ_PRIOR else prior)
    zw = g_write + (0.0 if f & NO_WRITE_PRIOR else prior)
    w_read = _weights(zr, sm)
    b = _weights(zw, sm)

    dlam_tot = dlam.copy()
    if f & ZOH_INJECTION:      # w_write = b / lambda
        db = dw_write / lam[..., None]
        dlam_tot = dlam_tot - (dw_write * b).sum(axis=-1) / (lam * lam)
    else:
        db = dw_write
    dzr = _weights_bwd(w_read, dw_read, sm)
    dzw = _weights_bwd(b, db, sm)
    # the prior -alpha ln tau feeds alpha and tau
    dprior = (0.0 if f & NO_READ_PRIOR else dzr) + (0.0 if f & NO_WRITE_PRIOR else dzw)
    dprior = np.broadcast_to(dprior, dzr.shape)
    dalpha_tot = dalpha - (dprior * ltau).sum(axis=-1)
    dtau_rows = dprior * (-alpha[..., None] / tau)        # d(-alpha ln tau)/dtau = -alpha / tau
    lead = tuple(range(dtau_rows.ndim - 2))
    dtau = dtau_rows.sum(axis=lead) if lead else dtau_rows.copy()

    dalpha_raw = np.zeros_like(alpha) if f & ALPHA_ONE else dalpha_tot * alpha * (1.0 - alpha)
    pass_dt = (sp_dt >= cfg.dt_min) & (sp_dt <= cfg.dt_max)
    ddt_raw = np.where(pass_dt, ddt * sigmoid(pre), 0.0)   # softplus' = sigmoid
    pass_lam = (sp_lam >= cfg.lam_min) & (sp_lam <= cfg.lam_max)
    dlam_raw = np.where(pass_lam, dlam_tot * sigmoid(lam_raw), 0.0)
    lead_h = tuple(range(ddt_raw.ndim - 1))
    ddt_bias = ddt_raw.sum(axis=lead_h) if lead_h else ddt_raw.copy()
    return dict(ddt_raw=ddt_raw, dalpha_raw=dalpha_raw, dlam_raw=dlam_raw, dg_read=dzr,
                dg_write=dzw, ddt_bias=ddt_bias, dtau=dtau)
