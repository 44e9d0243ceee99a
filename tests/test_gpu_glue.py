"""GPU parity of the mixer glue (causal depthwise conv1d with its decode step, gated RMSNorm)
against the fp64 oracle (oracle/mixer_glue.py), through the C ABI.

Tolerances as for the scan: relative L2 per output <= 1e-5 float32, <= 1e-2 bf16.  The conv
cases cover lengths inside, at and across the 32-position runs of a thread (1, 31, 33, 300),
widths 1 to 8, channel counts that take the shared-memory tiles (bf16, a multiple of 8), four or
two channels per thread or the scalar path, the
carried state and SiLU on and off; the norm cases cover gated and ungated rows, several group
sizes, and rows held in registers (dim <= 8192 forward, <= 4096 backward) or streamed.
"""
import numpy as np
import pytest
import torch

from oracle import mixer_glue as mg
from paper_2609_36314_gb300 import (conv1d_bwd, conv1d_fwd, conv1d_step, gated_rmsnorm_bwd,
                                    gated_rmsnorm_fwd, synth)
from tests.gpu_util import assert_close, dev_inputs, f64_inputs, to_host64, tol

pytestmark = pytest.mark.gpu


def _conv_case(B, L, C, W, dtype, silu, with_state, seed=0):
    host = synth.make_conv_inputs(B, L, C, W, dtype, seed=seed, with_state=with_state and W > 1)
    d = dev_inputs(host)
    o = f64_inputs(host)
    st, st64 = d.get("state"), o.get("state")
    u, fin = conv1d_fwd(d["x"], d["w"], d["bias"], st, silu=silu, want_state=True)
    g = conv1d_bwd(d["x"], d["w"], d["du"], d["bias"], st, silu=silu, want_dstate=True)
    torch.cuda.synchronize()
    ur, finr = mg.conv1d_fwd(o["x"], o["w"], o["bias"], st64, silu)
    gr = mg.conv1d_bwd(o["x"], o["w"], o["du"], o["bias"], st64, silu)
    t = tol(dtype)
    if L > 0:
        assert_close("u", to_host64(u), ur, t)
        assert_close("dx", to_host64(g["dx"]), gr["dx"], t)
        assert_close("dw", to_host64(g["dw"]), gr["dw"], t)
        assert_close("dbias", to_host64(g["dbias"]), gr["dbias"], t)
    if W > 1:
        np.testing.assert_array_equal(to_host64(fin), synth.to_f64(synth.cast(finr, dtype))
                                      if dtype == "bf16" else finr)
        if L > 0:
            assert_close("dstate", to_host64(g["dstate"]), gr["dstate"], t)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("L", [1, 31, 33, 300])
@pytest.mark.parametrize("C", [68, 70, 72])  # four / two channels per thread / shared-memory tiles (bf16)
def test_conv_lengths(dtype, L, C):
    _conv_case(2, L, C, 4, dtype, silu=True, with_state=True, seed=L)


@pytest.mark.parametrize("W", [1, 2, 3, 5, 8])
def test_conv_widths(W):
    _conv_case(2, 97, 64, W, "f32", silu=False, with_state=True, seed=W)


@pytest.mark.parametrize("W", [1, 2, 3, 5, 8])
def test_conv_widths_bf16_tiles(W):
    """bf16 with 8-divisible channels takes the shared-memory tile kernels (forward and backward):
    every width, a sequence across two 64-position tiles and the carried state."""
    _conv_case(2, 150, 72, W, "bf16", silu=True, with_state=True, seed=40 + W)
    _conv_case(1, W // 2 + 1, 16, W, "bf16", silu=False, with_state=True, seed=50 + W)  # L < W possible


@pytest.mark.parametrize("C", [1, 33, 129])
def test_conv_odd_channels(C):
    _conv_case(3, 70, C, 4, "bf16", silu=True, with_state=True, seed=C)


def test_conv_without_state_and_short_sequence():
    _conv_case(2, 50, 40, 4, "f32", silu=True, with_state=False)
    _conv_case(2, 2, 40, 6, "f32", silu=True, with_state=True, seed=3)   # L < W - 1


def test_conv_decode_steps_continue_the_prefill():
    """prefill conv over 40 positions with the state kept, then 10 decode steps == the conv
    over all 50 positions (the oracle's full sequence)."""
    host = synth.make_conv_inputs(3, 50, 96, 4, "bf16", seed=5)
    d = dev_inputs(host)
    o = f64_inputs(host)
    _, st = conv1d_fwd(d["x"][:, :40].contiguous(), d["w"], d["bias"], d["state"], silu=True,
                       want_state=True)
    ys = [conv1d_step(d["x"][:, t].contiguous(), d["w"], st, d["bias"], silu=True)
          for t in range(40, 50)]
    torch.cuda.synchronize()
    ur, finr = mg.conv1d_fwd(o["x"], o["w"], o["bias"], o["state"], True)
    assert_close("decode u", to_host64(torch.stack(ys, 1)), ur[:, 40:], 1e-2)
    np.testing.assert_array_equal(to_host64(st), synth.to_f64(synth.cast(finr, "bf16")))


def test_conv_training_shape():
    """The conv of the 1.3B-scale layer (d_inner 4096 plus B and C of 128 each: 4352 channels,
    width 4, SiLU) at L4096, batch 2 of the training batch."""
    _conv_case(2, 4096, 4352, 4, "bf16", silu=True, with_state=False, seed=9)


def _norm_case(R, D, gs, dtype, gated, seed=0):
    host = synth.make_norm_inputs(R, D, dtype, seed=seed)
    d = dev_inputs(host)
    o = f64_inputs(host)
    z, z64 = (d["z"], o["z"]) if gated else (None, None)
    out = gated_rmsnorm_fwd(d["y"], z, d["weight"], gs)
    g = gated_rmsnorm_bwd(d["y"], z, d["weight"], d["dout"], gs)
    torch.cuda.synchronize()
    ref = mg.gated_rmsnorm_fwd(o["y"], z64, o["weight"], gs)
    gr = mg.gated_rmsnorm_bwd(o["y"], z64, o["weight"], o["dout"], gs)
    t = tol(dtype)
    assert_close("out", to_host64(out), ref, t)
    assert_close("dy", to_host64(g["dy"]), gr["dy"], t)
    assert_close("dweight", to_host64(g["dweight"]), gr["dweight"], t)
    if gated:
        assert_close("dz", to_host64(g["dz"]), gr["dz"], t)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("gated", [False, True])
@pytest.mark.parametrize("D,gs", [(64, 64), (256, 32), (1032, 8), (4096, 512), (6000, 600), (8200, 1640)])
def test_rmsnorm_shapes(dtype, gated, D, gs):
    _norm_case(37, D, gs, dtype, gated, seed=D + gs)


def test_rmsnorm_training_shape():
    """Gated RMSNorm of the 1.3B-scale layer's scan output: 8192 rows (2 x 4096 tokens) of
    d_inner 4096, one group."""
    _norm_case(8192, 4096, 4096, "bf16", True, seed=11)


def test_glue_empty_sequence():
    host = synth.make_conv_inputs(2, 0, 16, 4, "f32", seed=1)
    d = dev_inputs(host)
    u, fin = conv1d_fwd(d["x"], d["w"], d["bias"], d["state"], want_state=True)
    g = conv1d_bwd(d["x"], d["w"], d["du"], d["bias"], d["state"], want_dstate=True)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(to_host64(fin), to_host64(d["state"]))
    assert np.all(to_host64(g["dw"]) == 0) and np.all(to_host64(g["dstate"]) == 0)
    out = gated_rmsnorm_fwd(torch.empty((0, 64), device="cuda"), None,
                            torch.ones(64, device="cuda"))
    assert out.shape == (0, 64)
