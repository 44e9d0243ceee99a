"""Mittag-Leffler functions and the finite sum-of-exponentials bank (test helpers).

* ``ml_series``: E_alpha(z) from its defining power series (Eq. Ea), summed in
  high precision with mpmath -- independent of everything else here.
* ``ml_quad``: E_alpha(-lambda t^alpha) from the diffusive (Laplace) representation
  of App. A, integral over r of exp(-r t) K_alpha(r; lambda), evaluated by a dense
  trapezoid rule in u = ln r plus the closed-form tail for r -> 0.
* ``soe_bank``: Theorem 2's midpoint grid tau_m = exp(A + (m - 1/2) h) and coefficients
  c_m = h tau_m R_{alpha,lambda}(tau_m) (Eq. cmdm-def), with R of Eq. r-density.
"""
from __future__ import annotations

import math

import mpmath
import numpy as np


def ml_series(alpha: float, z: float, dps: int | None = None) -> float:
    """E_alpha(z) = sum_k z^k / Gamma(alpha k + 1), summed until terms are negligible."""
    az = abs(z)
    if dps is None:
        # the largest term is ~exp(|z|^(1/alpha)); carry enough digits to absorb the cancellation
        dps = int(30 + az ** (1.0 / alpha) / 2.3) if az > 0 else 30
    with mpmath.workdps(dps):
        zz = mpmath.mpf(z)
        al = mpmath.mpf(alpha)       # exact value of the float alpha; alpha*k must not round
        total = mpmath.mpf(0)
        k = 0
        small = 0
        while True:
            term = zz ** k / mpmath.gamma(al * k + 1)
            total += term
            if abs(term) < mpmath.mpf(10) ** (-(dps - 5)) * max(1, abs(total)):
                small += 1
                if small > 5:
                    break
            else:
                small = 0
            k += 1
            if k > 200000:
                raise RuntimeError("series did not converge")
        return float(total)


def _kdensity_u(alpha, lam, u):
    """r K_alpha(r; lambda) with r = e^u (the integrand measure for du)."""
    s, c = math.sin(math.pi * alpha), math.cos(math.pi * alpha)
    ra = np.exp(alpha * u)
    return (lam * ra * s / math.pi) / (ra * ra + 2.0 * lam * ra * c + lam * lam)


def ml_quad(alpha: float, lam: float, t, u_lo: float = -60.0, du: float = 2e-3) -> np.ndarray:
    """E_alpha(-lambda t^alpha) for an array of t > 0 via the App. A Laplace representation."""
    t = np.atleast_1d(np.asarray(t, dtype=np.float64))
    out = np.empty_like(t)
    s, c = math.sin(math.pi * alpha), math.cos(math.pi * alpha)
    # closed-form part of the integral over (-inf, u_lo]: there exp(-r t) = 1 to 1e-20
    v0 = math.exp(alpha * u_lo) / lam ** 1.0  # substitution v = r^alpha / lambda
    tail = (math.atan((v0 + c) / s) - math.atan(c / s)) / (math.pi * alpha)
    for i, ti in enumerate(t):
        assert ti * math.exp(u_lo) < 1e-18
        u_hi = math.log(60.0 / ti)
        n = int(math.ceil((u_hi - u_lo) / du)) + 1
        u = np.linspace(u_lo, u_hi, n)
        f = _kdensity_u(alpha, lam, u) * np.exp(-np.exp(u) * ti)
        h = u[1] - u[0]
        out[i] = tail + h * (f.sum() - 0.5 * (f[0] + f[-1]))
    return out


def r_density(alpha: float, lam: float, tau):
    """R_{alpha,lambda}(tau) of Eq. r-density."""
    tau = np.asarray(tau, dtype=np.float64)
    s, c = math.sin(math.pi * alpha), math.cos(math.pi * alpha)
    ta = tau ** alpha
    return (lam * tau ** (alpha - 1.0) * s / math.pi) / (lam * lam * ta * ta + 2.0 * lam * ta * c + 1.0)


def h_density(alpha: float, lam: float, tau):
    """H_{alpha,lambda}(tau) of Eq. h-density."""
    tau = np.asarray(tau, dtype=np.float64)
    s, c = math.sin(math.pi * alpha), math.cos(math.pi * alpha)
    ta = tau ** alpha
    return (tau ** (alpha - 2.0) * s / math.pi) / (1.0 + 2.0 * lam * ta * c + lam * lam * ta * ta)


def soe_bank(alpha: float, lam: float, tau_lo: float, tau_hi: float, M: int):
    """Theorem 2 midpoint grid on [tau_lo, tau_hi] and coefficients c_m, d_m."""
    A, B = math.log(tau_lo), math.log(tau_hi)
    h = (B - A) / M
    x = A + (np.arange(1, M + 1) - 0.5) * h
    tau = np.exp(x)
    c = h * tau * r_density(alpha, lam, tau)
    d = h * tau * h_density(alpha, lam, tau)
    return tau, c, d


def ml_neg_power_many(alpha: float, s: np.ndarray, u_lo: float = -60.0, du: float = 3e-3):
    """E_alpha(-s^alpha) for many s at once (same Laplace representation as ``ml_quad``, lambda = 1)."""
    sn, cs = math.sin(math.pi * alpha), math.cos(math.pi * alpha)
    v0 = math.exp(alpha * u_lo)
    tail = (math.atan((v0 + cs) / sn) - math.atan(cs / sn)) / (math.pi * alpha)
    u = np.arange(u_lo, math.log(60.0 / float(np.min(s))) + du, du)
    ra = np.exp(alpha * u)
    f = (ra * sn / math.pi) / (ra * ra + 2 * ra * cs + 1)
    w = np.full(u.size, du)
    w[0] *= 0.5
    w[-1] *= 0.5
    return tail + np.exp(-np.exp(u)[None, :] * s[:, None]) @ (f * w)


def simplex_minimax_error(target: np.ndarray, s: np.ndarray, tau: np.ndarray) -> float:
    """min over c >= 0, sum c = 1 of max_s |target - sum_m c_m exp(-s/tau_m)| (an LP)."""
    from scipy.optimize import linprog
    M, n = tau.size, s.size
    Phi = np.exp(-s[:, None] / tau[None, :])
    cost = np.zeros(M + 1)
    cost[-1] = 1.0
    A_ub = np.vstack([np.hstack([-Phi, -np.ones((n, 1))]), np.hstack([Phi, -np.ones((n, 1))])])
    b_ub = np.concatenate([-target, target])
    A_eq = np.hstack([np.ones((1, M)), np.zeros((1, 1))])
    r = linprog(cost, A_ub=A_ub, b_ub=b_ub, A_eq=A_eq, b_eq=[1.0],
                bounds=[(0, None)] * (M + 1), method="highs")
    assert r.status == 0
    return float(r.x[-1])
