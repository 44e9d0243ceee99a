"""Pins of the scan-parameter oracle (oracle/param_prep.py), CPU only.

What fixes it, independently of its own code:
  * closed forms of softplus, sigmoid and the clips (Sec. 3.3, App. E.3);
  * Eq. read-softmax in closed form: with the prior alone the weights are tau^-alpha / sum, and
    any two weights stand in the ratio (tau_j / tau_m)^alpha e^(g_m - g_j); K = 1 gives 1;
  * Algorithm 1 of App. D transcribed literally with raw controls and logits in (the prep
    composed with the scan oracle must reproduce it);
  * the exact zero-order-hold injection of Eq. rho-beta-def-frac, written as its own
    recurrence, against the ZOH variant composed with the scan oracle;
  * the backward: central finite differences for every input (dt_bias and tau included), in
    every variant, and PyTorch float64 autograd of an independent implementation.
"""
import itertools

import numpy as np
import pytest
import torch

from oracle import oracle
from oracle import param_prep as pp


def _raw(seed=0, shape=(2, 5, 3), K=4, bias=True):
    rng = np.random.default_rng(seed)
    H = shape[-1]
    return dict(
        dt_raw=rng.standard_normal(shape), alpha_raw=rng.standard_normal(shape),
        lam_raw=rng.standard_normal(shape), g_read=0.5 * rng.standard_normal(shape + (K,)),
        g_write=0.5 * rng.standard_normal(shape + (K,)),
        tau=np.broadcast_to(2.0 ** (17.0 * np.arange(K) / max(K - 1, 1)), (H, K)).copy(),
        dt_bias=(-1.0 + 0.3 * rng.standard_normal(H)) if bias else None)


def _fwd(r, cfg=pp.PrepConfig()):
    return pp.prep_fwd(r["dt_raw"], r["alpha_raw"], r["lam_raw"], r["g_read"], r["g_write"],
                       r["tau"], r["dt_bias"], cfg)


# ------------------------------------------------------------------ closed forms
def test_softplus_sigmoid_closed_forms():
    assert pp.softplus(0.0) == pytest.approx(np.log(2.0), abs=1e-15)
    assert pp.softplus(np.log(np.e - 1.0)) == pytest.approx(1.0, abs=1e-15)
    assert pp.softplus(800.0) == 800.0 and pp.softplus(-800.0) == 0.0
    assert pp.sigmoid(0.0) == 0.5
    assert pp.sigmoid(np.log(3.0)) == pytest.approx(0.75, abs=1e-15)
    assert pp.sigmoid(-800.0) == 0.0 and pp.sigmoid(800.0) == 1.0


def test_clips_of_the_language_modelling_setting():
    r = _raw(1)
    r["dt_raw"][0, 0, 0] = -50.0   # softplus ~ 2e-22 -> clipped up to 1e-4
    r["dt_raw"][0, 1, 0] = 30.0    # ~30 -> clipped down to 1
    r["lam_raw"][0, 0, 1] = -20.0  # -> 0.25
    r["lam_raw"][0, 1, 1] = 9.0    # -> 4
    o = _fwd(r)
    assert o["dt"][0, 0, 0] == 1e-4 and o["dt"][0, 1, 0] == 1.0
    assert o["lam"][0, 0, 1] == 0.25 and o["lam"][0, 1, 1] == 4.0
    inside = (o["dt"] > 1e-4) & (o["dt"] < 1.0)
    pre = r["dt_raw"] + r["dt_bias"]
    np.testing.assert_allclose(o["dt"][inside], np.log1p(np.exp(pre))[inside], rtol=1e-14)
    np.testing.assert_allclose(o["alpha"], 1.0 / (1.0 + np.exp(-r["alpha_raw"])), rtol=1e-14)


def test_read_softmax_closed_form():
    r = _raw(2, K=6)
    r["g_read"][:] = 0.0
    o = _fwd(r)
    a = o["alpha"][..., None]
    prior = r["tau"] ** (-a)
    np.testing.assert_allclose(o["w_read"], prior / prior.sum(-1, keepdims=True), rtol=1e-13)
    # any two write weights: ratio (tau_j / tau_m)^alpha e^(g_m - g_j)
    w = o["w_write"]
    m, j = 1, 4
    ratio = (r["tau"][:, j] / r["tau"][:, m]) ** o["alpha"] * np.exp(
        r["g_write"][..., m] - r["g_write"][..., j])
    np.testing.assert_allclose(w[..., m] / w[..., j], ratio, rtol=1e-12)
    np.testing.assert_allclose(w.sum(-1), 1.0, rtol=1e-14)


def test_single_mode_weight_is_one():
    o = _fwd(_raw(3, K=1))
    assert np.all(o["w_read"] == 1.0) and np.all(o["w_write"] == 1.0)


def test_variants_closed_forms():
    r = _raw(4)
    base = _fwd(r)
    zoh = _fwd(r, pp.PrepConfig(flags=pp.ZOH_INJECTION))
    np.testing.assert_allclose(zoh["w_write"], base["w_write"] / base["lam"][..., None], rtol=1e-15)
    lin = _fwd(r, pp.PrepConfig(flags=pp.NO_SOFTMAX))
    np.testing.assert_allclose(lin["w_read"],
                               r["g_read"] - base["alpha"][..., None] * np.log(r["tau"]), rtol=1e-14)
    nwp = _fwd(r, pp.PrepConfig(flags=pp.NO_WRITE_PRIOR))
    e = np.exp(r["g_write"] - r["g_write"].max(-1, keepdims=True))
    np.testing.assert_allclose(nwp["w_write"], e / e.sum(-1, keepdims=True), rtol=1e-14)
    np.testing.assert_allclose(nwp["w_read"], base["w_read"], rtol=1e-15)
    a1 = _fwd(r, pp.PrepConfig(flags=pp.ALPHA_ONE))
    assert np.all(a1["alpha"] == 1.0)


# ------------------------------------------------------------------ Algorithm 1 with logits in
def test_literal_algorithm_one_from_raw_controls():
    """Algorithm 1 (App. D) with N = 1, B = C = 1, transcribed on an H x M x d_h state: the
    controls come from the raw projections by the Sec. 3.3 nonlinearities and the App. E.3
    clips, the weights from the logits by the softmax with the -alpha log tau prior.  The prep
    composed with the scan oracle must give the same outputs."""
    rng = np.random.default_rng(11)
    L, H, dh, M = 25, 3, 4, 6
    r = _raw(12, shape=(1, L, H), K=M)
    u = rng.standard_normal((L, H, dh))
    tau = r["tau"][0]
    S = np.zeros((H, M, dh))
    hs = np.zeros((L, H, dh))
    for t in range(L):
        dt = np.array([min(max(np.log1p(np.exp(r["dt_raw"][0, t, h] + r["dt_bias"][h])), 1e-4), 1.0)
                       for h in range(H)])
        al = np.array([1.0 / (1.0 + np.exp(-r["alpha_raw"][0, t, h])) for h in range(H)])
        lam = np.array([min(max(np.log1p(np.exp(r["lam_raw"][0, t, h])), 0.25), 4.0) for h in range(H)])
        tau_t = tau[None, :] / (lam ** (1.0 / al))[:, None]
        rho = np.exp(-dt[:, None] / tau_t)
        beta = 1.0 - rho
        lr = -al[:, None] * np.log(tau)[None] + r["g_read"][0, t]
        lw = -al[:, None] * np.log(tau)[None] + r["g_write"][0, t]
        c = np.exp(lr) / np.exp(lr).sum(-1, keepdims=True)
        b = np.exp(lw) / np.exp(lw).sum(-1, keepdims=True)
        S = rho[:, :, None] * S + (beta * b)[:, :, None] * u[t][:, None, :]
        hs[t] = np.einsum("hm,hmd->hd", c, S)
    o = _fwd(r)
    y, _ = oracle.fwd(u[None], o["dt"], o["alpha"], o["lam"], r["tau"], np.ones((1, L, 1, 1)),
                      np.ones((1, L, 1, 1)), o["w_read"], o["w_write"], np.zeros(H))
    assert np.max(np.abs(y[0] - hs)) < 1e-12


def test_zoh_injection_variant_is_the_exact_zoh_recurrence():
    """Eq. rho-beta-def-frac: beta~ = (1 - rho~) / lambda.  A recurrence written with that
    injection (N = 1, B = C = 1) equals the scan oracle fed by the ZOH variant of the prep."""
    L, H, dh, M = 20, 2, 3, 5
    r = _raw(13, shape=(1, L, H), K=M)
    u = np.random.default_rng(14).standard_normal((L, H, dh))
    o = _fwd(r, pp.PrepConfig(flags=pp.ZOH_INJECTION))
    base = _fwd(r)
    S = np.zeros((H, M, dh))
    hs = np.zeros((L, H, dh))
    for t in range(L):
        lam, al, dt = base["lam"][0, t], base["alpha"][0, t], base["dt"][0, t]
        rho = np.exp(-dt[:, None] * (lam ** (1.0 / al))[:, None] / r["tau"])
        beta = (1.0 - rho) / lam[:, None]
        S = rho[:, :, None] * S + (beta * base["w_write"][0, t])[:, :, None] * u[t][:, None, :]
        hs[t] = np.einsum("hm,hmd->hd", base["w_read"][0, t], S)
    y, _ = oracle.fwd(u[None], o["dt"], o["alpha"], o["lam"], r["tau"], np.ones((1, L, 1, 1)),
                      np.ones((1, L, 1, 1)), o["w_read"], o["w_write"], np.zeros(H))
    assert np.max(np.abs(y[0] - hs)) < 1e-12


# ------------------------------------------------------------------ backward
ALL_FLAGS = [0, pp.ZOH_INJECTION, pp.NO_SOFTMAX, pp.NO_READ_PRIOR | pp.NO_WRITE_PRIOR,
             pp.NO_WRITE_PRIOR | pp.ZOH_INJECTION, pp.ALPHA_ONE]


def _upstream(r, seed):
    rng = np.random.default_rng(seed)
    sh = r["dt_raw"].shape
    K = r["g_read"].shape[-1]
    return dict(ddt=rng.standard_normal(sh), dalpha=rng.standard_normal(sh),
                dlam=rng.standard_normal(sh), dw_read=rng.standard_normal(sh + (K,)),
                dw_write=rng.standard_normal(sh + (K,)))


def _loss(r, up, cfg):
    o = _fwd(r, cfg)
    return sum(float(np.sum(o[k] * up["d" + k])) for k in ("dt", "alpha", "lam", "w_read", "w_write"))


@pytest.mark.parametrize("flags", ALL_FLAGS)
def test_backward_finite_differences(flags):
    cfg = pp.PrepConfig(flags=flags)
    r = _raw(20 + flags, shape=(2, 4, 3), K=4)
    r["tau"] = r["tau"] * np.exp(0.2 * np.random.default_rng(5).standard_normal(r["tau"].shape))
    up = _upstream(r, 30 + flags)
    g = pp.prep_bwd(r["dt_raw"], r["alpha_raw"], r["lam_raw"], r["g_read"], r["g_write"],
                    r["tau"], up["ddt"], up["dalpha"], up["dlam"], up["dw_read"], up["dw_write"],
                    r["dt_bias"], cfg)
    names = dict(dt_raw="ddt_raw", alpha_raw="dalpha_raw", lam_raw="dlam_raw", g_read="dg_read",
                 g_write="dg_write", dt_bias="ddt_bias", tau="dtau")
    for name, gname in names.items():
        a = r[name]
        fd = np.zeros_like(a)
        for idx in itertools.product(*[range(n) for n in a.shape]):
            h = 1e-6 * max(1.0, abs(a[idx]))
            old = a[idx]
            a[idx] = old + h
            lp = _loss(r, up, cfg)
            a[idx] = old - h
            lm = _loss(r, up, cfg)
            a[idx] = old
            fd[idx] = (lp - lm) / (2 * h)
        err = np.linalg.norm(g[gname] - fd) / max(np.linalg.norm(fd), 1e-30)
        assert err < 1e-6, (name, err)


def test_backward_against_torch_autograd():
    """An independent torch implementation (softplus, sigmoid, clamp, softmax of torch) and its
    float64 autograd give the same gradients."""
    F = torch.nn.functional
    r = _raw(40, shape=(3, 6, 4), K=8)
    up = _upstream(r, 41)
    t = {k: torch.tensor(v, dtype=torch.float64, requires_grad=True) for k, v in r.items()}
    dt = torch.clamp(F.softplus(t["dt_raw"] + t["dt_bias"]), 1e-4, 1.0)
    al = torch.sigmoid(t["alpha_raw"])
    lam = torch.clamp(F.softplus(t["lam_raw"]), 0.25, 4.0)
    pri = -al[..., None] * torch.log(t["tau"])
    wr = torch.softmax(pri + t["g_read"], dim=-1)
    ww = torch.softmax(pri + t["g_write"], dim=-1)
    loss = sum((v * torch.tensor(up[k])).sum() for k, v in
               (("ddt", dt), ("dalpha", al), ("dlam", lam), ("dw_read", wr), ("dw_write", ww)))
    loss.backward()
    g = pp.prep_bwd(r["dt_raw"], r["alpha_raw"], r["lam_raw"], r["g_read"], r["g_write"],
                    r["tau"], up["ddt"], up["dalpha"], up["dlam"], up["dw_read"], up["dw_write"],
                    r["dt_bias"])
    for name, gname in (("dt_raw", "ddt_raw"), ("alpha_raw", "dalpha_raw"), ("lam_raw", "dlam_raw"),
                        ("g_read", "dg_read"), ("g_write", "dg_write"), ("dt_bias", "ddt_bias"),
                        ("tau", "dtau")):
        np.testing.assert_allclose(g[gname], t[name].grad.numpy(), rtol=1e-11, atol=1e-13)
