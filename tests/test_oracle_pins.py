"""Pins of the fp64 oracle against what the paper and the mathematics fix (CPU only).

Each test names the passage it follows.  Together they are chosen so that a
plausible slip anywhere in the oracle (lambda^alpha instead of lambda^(1/alpha),
1 - rho dropped or replaced by (1-rho)/lambda, rho^(t+1) vs rho^t, read/write weights
swapped, B and C swapped, outer-product orientation, a missing skip D) fails at least
one of them.
"""
import math

import numpy as np
import pytest
from scipy.integrate import solve_ivp
from scipy.special import erfcx

from oracle import oracle
from paper_2609_36314_gb300 import synth
from tests import mlf


def _call_fwd(d, h0=None):
    return oracle.fwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"],
                      d["w_read"], d["w_write"], d["D"], h0)


def _rand(Bz=2, L=24, H=4, P=3, G=2, N=5, K=3, seed=11, **kw):
    s = synth.Shape(Bz, L, H, P, G, N, K, 0, "f32")
    d = synth.make_scan_inputs(s, seed=seed, **kw)
    return {k: synth.to_f64(v) for k, v in d.items()}


def _const_controls(L, H, dt, alpha, lam):
    one = np.ones((1, L, H))
    return dt * one, alpha * one, lam * one


# ---------------------------------------------------------------- Mittag-Leffler reference
@pytest.mark.parametrize("x", [0.05, 0.4, 1.3, 3.0])
def test_ml_series_half_is_erfc(x):
    """E_{1/2}(-x) = exp(x^2) erfc(x): textbook closed form pins the series of Eq. Ea."""
    assert abs(mlf.ml_series(0.5, -x) - erfcx(x)) < 1e-13


@pytest.mark.parametrize("alpha", [0.3, 0.5, 0.7, 0.9])
@pytest.mark.parametrize("lam", [1.0, 2.5])
def test_ml_series_matches_diffusive_quadrature(alpha, lam):
    """Eq. Ea (series) == App. A Laplace representation with density K_alpha (pins R, H densities)."""
    t = np.array([0.1, 0.5, 1.0, 2.0, 4.0])
    q = mlf.ml_quad(alpha, lam, t)
    s = np.array([mlf.ml_series(alpha, -lam * ti ** alpha) for ti in t])
    assert np.max(np.abs(q - s)) < 1e-9


def test_densities_relation_and_self_similarity():
    """App. A remarks: H = R / (lambda tau); R_{a,l}(tau) = l^(1/a) R_{a,1}(l^(1/a) tau)."""
    tau = np.logspace(-3, 5, 50)
    for a in (0.2, 0.6, 0.95):
        for lam in (0.3, 1.0, 3.7):
            R, Hd = mlf.r_density(a, lam, tau), mlf.h_density(a, lam, tau)
            assert np.allclose(Hd, R / (lam * tau), rtol=1e-13, atol=0)
            s = lam ** (1 / a)
            assert np.allclose(R, s * mlf.r_density(a, 1.0, s * tau), rtol=1e-12, atol=0)


# ---------------------------------------------------------------- P1 impulse response
def test_impulse_response_is_the_log_spaced_soe_kernel():
    """Eq. frac-selective-update/readout with a unit impulse: y_t = D x_0 d_t0 + x_0 sum_m c_m kappa_m rho_m^t."""
    L, H, P, K = 40, 1, 2, 6
    dt, alpha, lam = _const_controls(L, H, 0.7, 0.45, 2.2)
    tau = (2.0 ** (17.0 * np.arange(K) / (K - 1)))[None, :]
    rng = np.random.default_rng(5)
    wr1 = rng.dirichlet(np.ones(K))
    ww1 = rng.dirichlet(np.ones(K))
    wr = np.broadcast_to(wr1, (1, L, H, K)).copy()
    ww = np.broadcast_to(ww1, (1, L, H, K)).copy()
    x = np.zeros((1, L, H, P))
    x[0, 0, 0] = [1.0, -0.5]
    Bm = np.ones((1, L, 1, 1))
    Cm = np.ones((1, L, 1, 1))
    D = np.array([0.8])
    y, _ = oracle.fwd(x, dt, alpha, lam, tau, Bm, Cm, wr, ww, D)
    rho = np.exp(-0.7 * 2.2 ** (1 / 0.45) / tau[0])
    kap = (1 - rho) * ww1
    t = np.arange(L)
    kern = (wr1 * kap * rho[None, :] ** t[:, None]).sum(-1)
    expect = kern[:, None] * np.array([1.0, -0.5])[None, :]
    expect[0] += D[0] * np.array([1.0, -0.5])
    assert np.max(np.abs(y[0, :, 0] - expect)) <= 1e-13 * np.max(np.abs(expect))


# ---------------------------------------------------------------- P3 bank vs fractional solution
def _fine_bank(alpha):
    # Theorem 2 midpoint grid; the mass below tau_lo is ~ sin(pi a) tau_lo^a / (pi a) and above
    # tau_hi ~ tau_hi^-a, both < 1e-7 for the alphas used here
    return mlf.soe_bank(alpha, 1.0, 1e-16, 1e22, 900)


@pytest.mark.parametrize("alpha,lam,dt", [(0.5, 1.0, 0.1), (0.7, 2.5, 0.05), (0.9, 0.4, 0.2),
                                          (0.6, 3.3, 0.02)])
def test_homogeneous_response_tracks_mittag_leffler(alpha, lam, dt):
    """h0 = 1 in every mode, no input, read weights c_m(alpha, 1) of Theorem 2 on the base grid:
    the layer's output after t+1 steps is sum_m c_m exp(-(t+1) dt lam^(1/alpha) / tau_m), which
    by Theorem 2 and the self-similarity remark equals E_alpha(-lam ((t+1) dt)^alpha)."""
    tau, c, _ = _fine_bank(alpha)
    K, L = tau.size, 60
    dts, als, lms = _const_controls(L, 1, dt, alpha, lam)
    wr = np.broadcast_to(c, (1, L, 1, K)).copy()
    ww = np.zeros((1, L, 1, K))
    x = np.zeros((1, L, 1, 1))
    y, _ = oracle.fwd(x, dts, als, lms, tau[None], np.ones((1, L, 1, 1)), np.ones((1, L, 1, 1)),
                      wr, ww, np.zeros(1), h0=np.ones((1, 1, K, 1, 1)))
    T = (np.arange(L) + 1) * dt
    ref = mlf.ml_quad(alpha, lam, T)
    assert np.max(np.abs(y[0, :, 0, 0] - ref)) < 2e-7


@pytest.mark.parametrize("alpha,lam,dt", [(0.5, 1.0, 0.1), (0.7, 2.5, 0.05), (0.8, 0.6, 0.25)])
def test_forced_response_with_exact_zoh_injection(alpha, lam, dt):
    """Write weight 1/lambda turns kappa = (1-rho) b into the exact ZOH injection (1-rho)/lambda of
    Eq. rho-beta-def-frac.  A unit input held on [0, dt) then produces, at time (t+1) dt, the
    fractional solution's integral of g over [t dt, (t+1) dt], which is
    (E_alpha(-lam (t dt)^alpha) - E_alpha(-lam ((t+1) dt)^alpha)) / lam."""
    tau, c, _ = _fine_bank(alpha)
    K, L = tau.size, 50
    dts, als, lms = _const_controls(L, 1, dt, alpha, lam)
    wr = np.broadcast_to(c, (1, L, 1, K)).copy()
    ww = np.full((1, L, 1, K), 1.0 / lam)
    x = np.zeros((1, L, 1, 1))
    x[0, 0, 0, 0] = 1.0
    y, _ = oracle.fwd(x, dts, als, lms, tau[None], np.ones((1, L, 1, 1)), np.ones((1, L, 1, 1)),
                      wr, ww, np.zeros(1))
    T = np.arange(L + 1) * dt
    E = np.concatenate([[1.0], mlf.ml_quad(alpha, lam, T[1:])])
    ref = (E[:-1] - E[1:]) / lam
    assert np.max(np.abs(y[0, :, 0, 0] - ref)) < 4e-7


# ---------------------------------------------------------------- P2 power-law tails
def _loglog_slope(t, y):
    A = np.vstack([np.log(t), np.ones_like(t)]).T
    return np.linalg.lstsq(A, np.log(y), rcond=None)[0][0]


@pytest.mark.parametrize("alpha", [0.3, 0.5, 0.7])
def test_power_law_tails_on_the_paper_bank(alpha):
    """K=16 geometric bank on [1, 2^17] (App. E.3).  With the log-timescale prior alone
    (weights proportional to tau^-alpha, Eq. read-softmax without content logits):
      * homogeneous decay ~ t^-alpha            (Eq. mittag-tail)
      * impulse response with write 1/lambda  ~ t^-(1+alpha)   (Eq. gal-tail)
      * impulse response with both priors     ~ t^-(1+2 alpha) (product of the two priors)."""
    K, L, dt, lam = 16, 6000, 1.0, 1.0
    tau = 2.0 ** (17.0 * np.arange(K) / (K - 1))
    prior = tau ** (-alpha) / np.sum(tau ** (-alpha))
    dts, als, lms = _const_controls(L, 1, dt, alpha, lam)
    ones = np.ones((1, L, 1, 1))
    wr = np.broadcast_to(prior, (1, L, 1, K)).copy()
    # fit where the bank covers the scale: between a few tau_2 and tau_{K-1}/4, in units of
    # the normalised time t * dt * lam^(1/alpha)
    t = np.arange(L) + 1.0
    sel = (t > 4 * tau[1]) & (t < tau[-2] / 4)
    y, _ = oracle.fwd(np.zeros((1, L, 1, 1)), dts, als, lms, tau[None], ones, ones, wr,
                      np.zeros((1, L, 1, K)), np.zeros(1), h0=np.ones((1, 1, K, 1, 1)))
    assert abs(_loglog_slope(t[sel], y[0, sel, 0, 0]) + alpha) < 0.1
    x = np.zeros((1, L, 1, 1))
    x[0, 0] = 1.0
    y, _ = oracle.fwd(x, dts, als, lms, tau[None], ones, ones, wr, np.full((1, L, 1, K), 1 / lam),
                      np.zeros(1))
    assert abs(_loglog_slope(t[sel], y[0, sel, 0, 0]) + 1 + alpha) < 0.1
    y, _ = oracle.fwd(x, dts, als, lms, tau[None], ones, ones, wr, wr, np.zeros(1))
    assert abs(_loglog_slope(t[sel], y[0, sel, 0, 0]) + 1 + 2 * alpha) < 0.1


# ---------------------------------------------------------------- P4 K = 1
def test_single_mode_is_the_textbook_selective_ssm():
    """K=1 (softmax over one mode is 1): h_t = a_t h_{t-1} + (1 - a_t) x_t B_t^T, y = h C + D x."""
    d = _rand(K=1, seed=4)
    d["w_read"][:] = 1.0
    d["w_write"][:] = 1.0
    y, hf = _call_fwd(d)
    Bz, L, H, P = d["x"].shape
    G, N = d["B"].shape[2:]
    ref = np.zeros_like(y)
    for b in range(Bz):
        for h in range(H):
            g = h // (H // G)
            state = np.zeros((P, N))
            for t in range(L):
                a = math.exp(-d["dt"][b, t, h] * d["lam"][b, t, h] ** (1 / d["alpha"][b, t, h])
                             / d["tau"][h, 0])
                state = a * state + (1 - a) * np.outer(d["x"][b, t, h], d["B"][b, t, g])
                ref[b, t, h] = state @ d["C"][b, t, g] + d["D"][h] * d["x"][b, t, h]
    assert np.max(np.abs(y - ref)) < 1e-14 * np.max(np.abs(ref)) * 10


# ---------------------------------------------------------------- P5 alpha = 1
def test_alpha_one_is_ode_relaxation():
    """alpha = 1: retention over one step equals the solution of ds/dt = -(lambda/tau) s over
    [0, Delta] (Eq. ode-relaxation with the ZOH of Eq. zoh-recurrence), integrated numerically."""
    L, K = 5, 3
    tau = np.array([[1.0, 7.0, 50.0]])
    dt, alpha, lam = _const_controls(L, 1, 0.37, 1.0, 2.9)
    y, hf = oracle.fwd(np.zeros((1, L, 1, 1)), dt, alpha, lam, tau, np.ones((1, L, 1, 1)),
                       np.ones((1, L, 1, 1)), np.ones((1, L, 1, K)), np.zeros((1, L, 1, K)),
                       np.zeros(1), h0=np.ones((1, 1, K, 1, 1)))
    for m in range(K):
        sol = solve_ivp(lambda t, s: -(2.9 / tau[0, m]) * s, (0, 0.37 * L), [1.0], rtol=1e-12,
                        atol=1e-14)
        assert abs(hf[0, 0, m, 0, 0] - sol.y[0, -1]) < 1e-9


# ---------------------------------------------------------------- P6 literal Algorithm 1
def test_literal_algorithm_one():
    """Algorithm 1 of App. D transcribed on an H x M x d_h state with N = 1 and B = C = 1: weights
    from logits by the softmax with the -alpha log tau prior, then the oracle with those weights."""
    rng = np.random.default_rng(9)
    L, H, dh, M = 30, 3, 4, 5
    tau = 2.0 ** (17.0 * np.arange(M) / (M - 1))
    u = rng.standard_normal((L, H, dh))
    dt = np.clip(np.log1p(np.exp(rng.standard_normal((L, H)) - 1)), 1e-4, 1)
    al = 1 / (1 + np.exp(-rng.standard_normal((L, H))))
    lam = np.clip(np.log1p(np.exp(rng.standard_normal((L, H)))), 0.25, 4)
    g_read = rng.standard_normal((L, H, M))
    g_write = rng.standard_normal((L, H, M))

    def softmax(v):
        v = v - v.max(-1, keepdims=True)
        return np.exp(v) / np.exp(v).sum(-1, keepdims=True)

    S = np.zeros((H, M, dh))
    hs = np.zeros((L, H, dh))
    cs = np.zeros((L, H, M))
    bs = np.zeros((L, H, M))
    for t in range(L):
        tau_t = tau[None, :] / (lam[t] ** (1 / al[t]))[:, None]          # line: tau~
        rho_t = np.exp(-dt[t][:, None] / tau_t)                           # line: rho~
        beta_t = 1 - rho_t                                                # line: beta~
        c_t = softmax(-al[t][:, None] * np.log(tau)[None] + g_read[t])    # read weights
        b_t = softmax(-al[t][:, None] * np.log(tau)[None] + g_write[t])   # write weights
        kap = beta_t * b_t
        S = rho_t[:, :, None] * S + kap[:, :, None] * u[t][:, None, :]
        hs[t] = np.einsum("hm,hmd->hd", c_t, S)
        cs[t], bs[t] = c_t, b_t
    y, hf = oracle.fwd(u[None], dt[None], al[None], lam[None], np.broadcast_to(tau, (H, M)),
                       np.ones((1, L, 1, 1)), np.ones((1, L, 1, 1)), cs[None], bs[None],
                       np.zeros(H))
    assert np.max(np.abs(y[0] - hs)) < 1e-12
    assert np.max(np.abs(hf[0, :, :, :, 0] - S)) < 1e-12


# ---------------------------------------------------------------- P7 brute force
def test_bruteforce_materialised_kernel():
    """y_t = sum_m c_{t,m} e^{L_t} S0 C_t + sum_{k<=t} (C_t.B_k) sum_m c_{t,m} kappa_{k,m}
    prod_{j=k+1..t} rho_{j,m} x_k + D x_t, evaluated pair by pair (O(L^2 K))."""
    d = _rand(L=20, seed=21, with_h0=True)
    y, _ = _call_fwd(d, d["h0"])
    Bz, L, H, P = d["x"].shape
    G, N = d["B"].shape[2:]
    K = d["tau"].shape[1]
    ref = np.zeros_like(y)
    for b in range(Bz):
        for h in range(H):
            g = h // (H // G)
            e = d["dt"][b, :, h] * d["lam"][b, :, h] ** (1 / d["alpha"][b, :, h])
            rho = np.exp(-e[:, None] / d["tau"][h][None, :])
            kap = (1 - rho) * d["w_write"][b, :, h]
            for t in range(L):
                acc = d["D"][h] * d["x"][b, t, h]
                decay0 = np.prod(rho[: t + 1], axis=0)
                for m in range(K):
                    acc = acc + d["w_read"][b, t, h, m] * decay0[m] * (d["h0"][b, h, m] @ d["C"][b, t, g])
                for k in range(t + 1):
                    prod = np.prod(rho[k + 1: t + 1], axis=0)
                    gam = np.sum(d["w_read"][b, t, h] * kap[k] * prod)
                    acc = acc + (d["C"][b, t, g] @ d["B"][b, k, g]) * gam * d["x"][b, k, h]
                ref[b, t, h] = acc
    assert np.max(np.abs(y - ref)) < 1e-13 * max(1.0, np.max(np.abs(ref)))


# ---------------------------------------------------------------- P9 hand-off
def test_state_handoff_and_decode_continuity():
    """scan(L1 + L2) == scan(L2; h0 = scan(L1).h_final) == scan(L1) then L2 single-token steps."""
    d = _rand(L=30, seed=8)
    y, hf = _call_fwd(d)
    L1 = 17
    first = {k: (v[:, :L1] if v.ndim >= 3 and k not in ("tau", "h0") else v) for k, v in d.items()}
    second = {k: (v[:, L1:] if v.ndim >= 3 and k not in ("tau", "h0") else v) for k, v in d.items()}
    y1, h1 = _call_fwd(first)
    y2, h2 = _call_fwd(second, h1)
    assert np.max(np.abs(np.concatenate([y1, y2], 1) - y)) < 1e-13
    assert np.max(np.abs(h2 - hf)) < 1e-13
    st = h1.copy()
    for t in range(L1, 30):
        yt, st = oracle.decode(d["x"][:, t], d["dt"][:, t], d["alpha"][:, t], d["lam"][:, t],
                               d["tau"], d["B"][:, t], d["C"][:, t], d["w_read"][:, t],
                               d["w_write"][:, t], d["D"], st)
        assert np.max(np.abs(yt - y[:, t])) < 1e-13
    assert np.max(np.abs(st - hf)) < 1e-13


# ---------------------------------------------------------------- P11 invariances
def test_invariances():
    d = _rand(seed=31, with_h0=True)
    y, hf = _call_fwd(d, d["h0"])
    # linear in (x, h0) jointly, with D x included
    d2 = dict(d, x=2.5 * d["x"])
    y2, hf2 = _call_fwd(d2, 2.5 * d["h0"])
    assert np.max(np.abs(y2 - 2.5 * y)) < 1e-12 * np.max(np.abs(y))
    # B -> sB, C -> C/s leaves y unchanged (state scales by s)
    d3 = dict(d, B=3.0 * d["B"], C=d["C"] / 3.0)
    y3, hf3 = _call_fwd(d3, 3.0 * d["h0"])
    assert np.max(np.abs(y3 - y)) < 1e-12 * np.max(np.abs(y))
    assert np.max(np.abs(hf3 - 3.0 * hf)) < 1e-12 * np.max(np.abs(hf))
    # permuting heads within a group permutes outputs
    perm = np.array([1, 0, 3, 2])
    d4 = {k: v for k, v in d.items()}
    for k in ("x", "dt", "alpha", "lam", "w_read", "w_write"):
        d4[k] = d[k][:, :, perm]
    d4["tau"] = d["tau"][perm]
    d4["D"] = d["D"][perm]
    y4, hf4 = _call_fwd(d4, d["h0"][:, perm])
    assert np.max(np.abs(y4 - y[:, :, perm])) < 1e-13
    assert np.max(np.abs(hf4 - hf[:, perm])) < 1e-13
