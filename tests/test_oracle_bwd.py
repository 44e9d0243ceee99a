"""Pins of the oracle's backward pass (CPU only).

The paper prints no gradient formulas; the backward is the adjoint of the
recurrence of Sec. 3.2 / Algorithm 1.  It is pinned two independent ways:
  * central finite differences of the oracle's own forward (fp64) for every input,
  * PyTorch float64 CPU autograd through a third, naive implementation of the
    layer written with torch tensor ops.
"""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2609_36314_gb300 import synth

NAMES = ["x", "dt", "alpha", "lam", "B", "C", "w_read", "w_write", "D", "h0", "tau"]
GRAD = dict(x="dx", dt="ddt", alpha="dalpha", lam="dlam", B="dB", C="dC", w_read="dw_read",
            w_write="dw_write", D="dD", h0="dh0", tau="dtau")


def _inputs(seed=2, L=9, shift=0.0):
    s = synth.Shape(2, L, 4, 3, 2, 2, 3, 0, "f32", dt_shift=shift)
    d = synth.make_scan_inputs(s, seed=seed, with_dy=True, with_h0=True, with_dh_final=True)
    d = {k: synth.to_f64(v) for k, v in d.items()}
    # keep lambda^(1/alpha) moderate so finite differences are well conditioned
    d["alpha"] = 0.3 + 0.6 * d["alpha"]
    # per-head timescales that differ between heads (learned-timescale variant), spanning the
    # range where the modes neither die within a step nor stay constant over the sequence
    d["tau"] = (2.0 ** np.linspace(-1.0, 5.0, d["tau"].size)).reshape(d["tau"].shape)
    return d


def _loss(d):
    y, hf = oracle.fwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"],
                       d["w_read"], d["w_write"], d["D"], d["h0"], nthreads=1)
    return float(np.sum(y * d["dy"]) + np.sum(hf * d["dh_final"]))


def _grads(d):
    return oracle.bwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"],
                      d["w_read"], d["w_write"], d["D"], d["dy"], h0=d["h0"],
                      dh_final=d["dh_final"], seg=4, nthreads=2)


@pytest.mark.parametrize("name", NAMES)
def test_backward_matches_central_differences(name):
    d = _inputs()
    g = _grads(d)[GRAD[name]]
    rng = np.random.default_rng(hash(name) % 2**32)
    flat = d[name].reshape(-1)
    idx = rng.choice(flat.size, size=min(12, flat.size), replace=False)
    for i in idx:
        v = flat[i]
        h = 1e-6 * max(1.0, abs(v))
        flat[i] = v + h
        lp = _loss(d)
        flat[i] = v - h
        lm = _loss(d)
        flat[i] = v
        fd = (lp - lm) / (2 * h)
        an = g.reshape(-1)[i]
        assert abs(fd - an) <= 1e-6 * max(1.0, abs(an)), (name, i, fd, an)


def _torch_layer(x, dt, alpha, lam, tau, Bm, Cm, wr, ww, D, h0):
    """Naive third implementation: per-token loop, all heads and modes at once, torch ops."""
    Bz, L, H, P = x.shape
    G, N = Bm.shape[2], Bm.shape[3]
    rep = H // G
    S = h0.clone()                                             # [B,H,K,P,N]
    ys = []
    for t in range(L):
        rate = torch.exp(torch.log(lam[:, t]) / alpha[:, t])   # lambda^(1/alpha)  [B,H]
        a = dt[:, t, :, None] * rate[..., None] / tau[None]    # [B,H,K]
        rho = torch.exp(-a)
        kap = (1 - rho) * ww[:, t]
        Bt = Bm[:, t].repeat_interleave(rep, dim=1)            # [B,H,N]
        Ct = Cm[:, t].repeat_interleave(rep, dim=1)
        outer = x[:, t, :, :, None] * Bt[:, :, None, :]        # [B,H,P,N]
        S = rho[..., None, None] * S + kap[..., None, None] * outer[:, :, None]
        read = torch.einsum("bhkpn,bhn->bhkp", S, Ct)
        ys.append(torch.einsum("bhk,bhkp->bhp", wr[:, t], read) + D[None, :, None] * x[:, t])
    return torch.stack(ys, 1), S


def test_backward_matches_torch_autograd_of_naive_layer():
    d = _inputs(seed=5, L=11, shift=1.0)
    d["alpha"] = synth.to_f64(synth.make_scan_inputs(
        synth.Shape(2, 11, 4, 3, 2, 2, 3, 0, "f32"), seed=5)["alpha"])
    g = _grads(d)
    T = {k: torch.tensor(d[k], dtype=torch.float64, requires_grad=(k in NAMES))
         for k in NAMES}
    y, hf = _torch_layer(T["x"], T["dt"], T["alpha"], T["lam"], T["tau"], T["B"], T["C"],
                         T["w_read"], T["w_write"], T["D"], T["h0"])
    yo, hfo = oracle.fwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"],
                         d["w_read"], d["w_write"], d["D"], d["h0"])
    assert np.max(np.abs(y.detach().numpy() - yo)) < 1e-12
    assert np.max(np.abs(hf.detach().numpy() - hfo)) < 1e-12
    loss = (y * torch.tensor(d["dy"])).sum() + (hf * torch.tensor(d["dh_final"])).sum()
    loss.backward()
    for k in NAMES:
        ref = T[k].grad.numpy()
        assert synth.rel_l2(g[GRAD[k]], ref) < 1e-11, k


def test_backward_without_final_state_gradient_and_h0():
    """dh_final = None and h0 = None are the defaults of a training step (zeros)."""
    d = _inputs(seed=7)
    g0 = oracle.bwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"],
                    d["w_read"], d["w_write"], d["D"], d["dy"])
    z = np.zeros_like(d["h0"])
    g1 = oracle.bwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"],
                    d["w_read"], d["w_write"], d["D"], d["dy"], h0=z, dh_final=z)
    for k in g0:
        assert np.array_equal(g0[k], g1[k]), k


def test_backward_is_finite_when_lambda_pow_overflows():
    """lambda^(1/alpha) = +inf (alpha -> 0): rho = 0, kappa = b; gradients through rho vanish."""
    d = _inputs(seed=3)
    d["alpha"][0, 2, 1] = 1e-4
    d["lam"][0, 2, 1] = 3.0
    g = _grads(d)
    for k, v in g.items():
        assert np.all(np.isfinite(v)), k
    assert g["ddt"][0, 2, 1] == 0.0 and g["dalpha"][0, 2, 1] == 0.0 and g["dlam"][0, 2, 1] == 0.0
