"""Pins of the mixer-glue oracle (oracle/mixer_glue.py), CPU only.

Causal depthwise convolution (Sec. 3.3): equals numpy's full convolution truncated to the first
L outputs, channel by channel; the impulse response is the reversed filter; an output never
depends on a later input; carrying the state across a split (and decoding step by step)
reproduces the unsplit sequence.  Gated RMS normalisation: with unit weight and no epsilon each
group of the output has mean square 1 and is invariant to scaling y; a constant group maps to
its sign times the weight; without a gate it is plain RMSNorm.  Backwards: central finite
differences, and float64 autograd of independent torch implementations (torch's grouped
conv1d, torch's silu and rsqrt).
"""
import numpy as np
import pytest
import torch

from oracle import mixer_glue as mg


def _conv_inputs(seed=0, B=2, L=23, C=5, W=4):
    rng = np.random.default_rng(seed)
    return dict(x=rng.standard_normal((B, L, C)), w=rng.standard_normal((C, W)),
                bias=rng.standard_normal(C), state=rng.standard_normal((B, C, W - 1)))


def test_silu_closed_forms():
    assert mg.silu(0.0) == 0.0
    assert mg.silu_grad(0.0) == 0.5
    assert mg.silu(np.log(3.0)) == pytest.approx(0.75 * np.log(3.0), abs=1e-15)


def test_conv_equals_truncated_full_convolution():
    d = _conv_inputs(1)
    u, _ = mg.conv1d_fwd(d["x"], d["w"], d["bias"])
    B, L, C = d["x"].shape
    for b in range(B):
        for c in range(C):
            ref = np.convolve(d["x"][b, :, c], d["w"][c, ::-1])[:L] + d["bias"][c]
            np.testing.assert_allclose(u[b, :, c], ref, rtol=1e-13, atol=1e-13)


def test_conv_impulse_response_and_causality():
    W, L, C = 4, 12, 3
    w = np.random.default_rng(2).standard_normal((C, W))
    x = np.zeros((1, L, C))
    x[0, 5, :] = 1.0
    u, _ = mg.conv1d_fwd(x, w)
    for c in range(C):
        np.testing.assert_array_equal(u[0, :5, c], 0.0)          # nothing before the impulse
        np.testing.assert_allclose(u[0, 5:5 + W, c], w[c, ::-1], rtol=1e-15)
        np.testing.assert_array_equal(u[0, 5 + W:, c], 0.0)
    d = _conv_inputs(3)
    u0, _ = mg.conv1d_fwd(d["x"], d["w"], d["bias"], d["state"], activation=True)
    x2 = d["x"].copy()
    x2[:, 10:, :] += 1.0
    u1, _ = mg.conv1d_fwd(x2, d["w"], d["bias"], d["state"], activation=True)
    np.testing.assert_array_equal(u0[:, :10], u1[:, :10])


def test_conv_state_handoff_and_decode_steps():
    d = _conv_inputs(4, L=30)
    full, fin = mg.conv1d_fwd(d["x"], d["w"], d["bias"], d["state"], activation=True)
    a, st = mg.conv1d_fwd(d["x"][:, :11], d["w"], d["bias"], d["state"], activation=True)
    b, fin2 = mg.conv1d_fwd(d["x"][:, 11:], d["w"], d["bias"], st, activation=True)
    np.testing.assert_allclose(np.concatenate([a, b], 1), full, rtol=1e-14, atol=1e-14)
    np.testing.assert_array_equal(fin, fin2)
    st = d["state"]
    for t in range(30):
        ut, st = mg.conv1d_step(d["x"][:, t], d["w"], st, d["bias"], activation=True)
        np.testing.assert_allclose(ut, full[:, t], rtol=1e-14, atol=1e-14)
    np.testing.assert_array_equal(st, fin)


def test_rmsnorm_invariants():
    rng = np.random.default_rng(5)
    R, D, gs = 4, 12, 4
    y, z = rng.standard_normal((R, D)), rng.standard_normal((R, D))
    one = np.ones(D)
    out = mg.gated_rmsnorm_fwd(y, z, one, gs, eps=0.0)
    np.testing.assert_allclose(np.mean(out.reshape(R, D // gs, gs) ** 2, -1), 1.0, rtol=1e-14)
    np.testing.assert_allclose(mg.gated_rmsnorm_fwd(7.5 * y, z, one, gs, eps=0.0), out, rtol=1e-13)
    wgt = rng.standard_normal(D)
    c = np.full((1, D), -3.0)
    np.testing.assert_allclose(mg.gated_rmsnorm_fwd(c, None, wgt, gs, eps=0.0), -wgt[None], rtol=1e-15)
    plain = y / np.sqrt(np.mean(y ** 2, axis=-1, keepdims=True) + 1e-5) * wgt
    np.testing.assert_allclose(mg.gated_rmsnorm_fwd(y, None, wgt, D), plain, rtol=1e-14)


def _fd(f, arrays, name, h=1e-6):
    a = arrays[name]
    g = np.zeros_like(a)
    it = np.nditer(a, flags=["multi_index"])
    for _ in it:
        i = it.multi_index
        old = a[i]
        a[i] = old + h
        lp = f()
        a[i] = old - h
        lm = f()
        a[i] = old
        g[i] = (lp - lm) / (2 * h)
    return g


@pytest.mark.parametrize("activation", [False, True])
def test_conv_backward_finite_differences(activation):
    d = _conv_inputs(6, B=2, L=9, C=3, W=4)
    du = np.random.default_rng(7).standard_normal(d["x"].shape)

    def loss():
        return float(np.sum(mg.conv1d_fwd(d["x"], d["w"], d["bias"], d["state"], activation)[0] * du))

    g = mg.conv1d_bwd(d["x"], d["w"], du, d["bias"], d["state"], activation)
    for name, gname in (("x", "dx"), ("w", "dw"), ("bias", "dbias"), ("state", "dstate")):
        fd = _fd(loss, d, name)
        assert np.max(np.abs(g[gname] - fd)) < 1e-7 * max(1.0, np.max(np.abs(fd))), name


def test_conv_backward_against_torch_grouped_conv1d():
    F = torch.nn.functional
    d = _conv_inputs(8, B=3, L=17, C=6, W=4)
    du = np.random.default_rng(9).standard_normal(d["x"].shape)
    t = {k: torch.tensor(v, requires_grad=True) for k, v in d.items()}
    xin = torch.cat([t["state"], t["x"].transpose(1, 2)], dim=2)          # [B, C, W-1+L]
    pre = F.conv1d(xin, t["w"][:, None, :], t["bias"], groups=6)          # valid: L outputs
    u = F.silu(pre).transpose(1, 2)
    (u * torch.tensor(du)).sum().backward()
    ref, _ = mg.conv1d_fwd(d["x"], d["w"], d["bias"], d["state"], activation=True)
    np.testing.assert_allclose(u.detach().numpy(), ref, rtol=1e-13, atol=1e-13)
    g = mg.conv1d_bwd(d["x"], d["w"], du, d["bias"], d["state"], activation=True)
    for name, gname in (("x", "dx"), ("w", "dw"), ("bias", "dbias"), ("state", "dstate")):
        np.testing.assert_allclose(g[gname], t[name].grad.numpy(), rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("gated", [False, True])
def test_rmsnorm_backward(gated):
    rng = np.random.default_rng(10)
    R, D, gs = 3, 8, 4
    arr = dict(y=rng.standard_normal((R, D)), z=rng.standard_normal((R, D)),
               w=rng.standard_normal(D))
    dout = rng.standard_normal((R, D))

    def loss():
        return float(np.sum(mg.gated_rmsnorm_fwd(arr["y"], arr["z"] if gated else None, arr["w"],
                                                 gs) * dout))

    g = mg.gated_rmsnorm_bwd(arr["y"], arr["z"] if gated else None, arr["w"], dout, gs)
    names = [("y", "dy"), ("w", "dweight")] + ([("z", "dz")] if gated else [])
    for name, gname in names:
        fd = _fd(loss, arr, name)
        assert np.max(np.abs(g[gname] - fd)) < 1e-7 * max(1.0, np.max(np.abs(fd))), name
    # float64 autograd of an independent torch implementation
    t = {k: torch.tensor(v, requires_grad=True) for k, v in arr.items()}
    v = t["y"] * torch.nn.functional.silu(t["z"]) if gated else t["y"]
    vg = v.reshape(R, D // gs, gs)
    out = (vg * torch.rsqrt(vg.pow(2).mean(-1, keepdim=True) + 1e-5)).reshape(R, D) * t["w"]
    (out * torch.tensor(dout)).sum().backward()
    for name, gname in names:
        np.testing.assert_allclose(g[gname], t[name].grad.numpy(), rtol=1e-12, atol=1e-13)
