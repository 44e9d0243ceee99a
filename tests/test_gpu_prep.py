"""GPU parity of the scan-parameter construction (frac_param_prep_fwd / _bwd) against the fp64
oracle (oracle/param_prep.py), through the C ABI, on the seeded synthetic recipe.

Tolerances as for the scan: relative L2 per output <= 1e-5 on the float32 path, <= 1e-2 with
bf16 logits (float32 arithmetic).  Shapes cover the vectorised rows (K * element size a
multiple of 16 bytes), the scalar rows (K = 5, 4 in bf16), every variant flag, more heads than
a block has threads (the direct-atomic reduction), an empty sequence and the training shape.
"""
import numpy as np
import pytest
import torch

from oracle import oracle
from oracle import param_prep as pp
from paper_2609_36314_gb300 import param_prep_bwd, param_prep_fwd, prep_config, scan_fwd, synth
from tests.gpu_util import assert_close, dev_inputs, f64_inputs, to_host64, tol

pytestmark = pytest.mark.gpu

FLAGS = dict(zoh=pp.ZOH_INJECTION, no_softmax=pp.NO_SOFTMAX, no_read_prior=pp.NO_READ_PRIOR,
             no_write_prior=pp.NO_WRITE_PRIOR, alpha_one=pp.ALPHA_ONE)


def _cfgs(flags):
    kw = {k: bool(flags & v) for k, v in FLAGS.items()}
    return (prep_config(zoh_injection=kw["zoh"], no_softmax=kw["no_softmax"],
                        no_read_prior=kw["no_read_prior"], no_write_prior=kw["no_write_prior"],
                        alpha_one=kw["alpha_one"]),
            pp.PrepConfig(flags=flags))


def _check(s, flags=0, bias=True, seed=0):
    host = synth.make_prep_inputs(s, seed=seed, with_grads=True)
    if not bias:
        host["dt_bias"] = None
    d = {k: (v if v is None else dev_inputs({k: v})[k]) for k, v in host.items()}
    o64 = {k: (None if v is None else synth.to_f64(v)) for k, v in host.items()}
    cfg, cfg64 = _cfgs(flags)
    out = param_prep_fwd(d["dt_raw"], d["alpha_raw"], d["lam_raw"], d["g_read"], d["g_write"],
                         d["tau"], d["dt_bias"], cfg)
    g = param_prep_bwd(d["dt_raw"], d["alpha_raw"], d["lam_raw"], d["g_read"], d["g_write"],
                       d["tau"], d["ddt"], d["dalpha"], d["dlam"], d["dw_read"], d["dw_write"],
                       d["dt_bias"], cfg, want_dt_bias=bias)
    torch.cuda.synchronize()
    ref = pp.prep_fwd(o64["dt_raw"], o64["alpha_raw"], o64["lam_raw"], o64["g_read"],
                      o64["g_write"], o64["tau"], o64["dt_bias"], cfg64)
    gr = pp.prep_bwd(o64["dt_raw"], o64["alpha_raw"], o64["lam_raw"], o64["g_read"],
                     o64["g_write"], o64["tau"], o64["ddt"], o64["dalpha"], o64["dlam"],
                     o64["dw_read"], o64["dw_write"], o64["dt_bias"], cfg64)
    t = tol(s.dtype)
    if s.batch * s.seqlen == 0:
        assert np.all(to_host64(g["dtau"]) == 0.0)
        return
    for k in ("dt", "alpha", "lam", "w_read", "w_write"):
        assert_close(k, to_host64(out[k]), ref[k], t)
    keys = ["ddt_raw", "dlam_raw", "dg_read", "dg_write", "dtau"] + (["ddt_bias"] if bias else [])
    if not flags & pp.ALPHA_ONE:
        keys.append("dalpha_raw")
    for k in keys:
        assert_close(k, to_host64(g[k]), gr[k], t)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("K", [4, 5, 8, 16])
def test_prep_shapes(dtype, K):
    _check(synth.Shape(2, 77, 6, 1, 1, 1, K, 0, dtype), seed=K)


@pytest.mark.parametrize("flags", [pp.ZOH_INJECTION, pp.NO_SOFTMAX,
                                   pp.NO_READ_PRIOR | pp.NO_WRITE_PRIOR,
                                   pp.NO_WRITE_PRIOR | pp.ZOH_INJECTION, pp.ALPHA_ONE])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_prep_variants(flags, dtype):
    _check(synth.Shape(1, 150, 4, 1, 1, 1, 8, 0, dtype), flags=flags, seed=flags)


def test_prep_many_heads_and_no_bias():
    _check(synth.Shape(1, 9, 300, 1, 1, 1, 8, 0, "f32"), bias=False, seed=3)


@pytest.mark.parametrize("K", [8, 16])
def test_prep_more_heads_than_one_wave_of_threads(K):
    """More heads than the backward's resident threads (its row stride must still hold whole
    head cycles), and per-head sums across only a couple of positions."""
    _check(synth.Shape(1, 2, 45000, 1, 1, 1, K, 0, "f32"), seed=11 + K)


def test_prep_empty_sequence():
    _check(synth.Shape(2, 0, 4, 1, 1, 1, 8, 0, "bf16"))


def test_prep_training_shape():
    """B8 L4096 H64 K8 bf16, every output compared in full."""
    _check(synth.Shape(8, 4096, 64, 1, 1, 1, 8, 0, "bf16"), seed=7)


def test_prep_paper_shape():
    """The paper's layer: 16 heads, 16 modes."""
    _check(synth.Shape(1, 2048, 16, 1, 1, 1, 16, 0, "bf16"), seed=8)


def test_prep_zoh_variant_through_the_scan():
    """The ZOH variant of the prep feeding the GPU scan equals the oracle scan fed by the
    oracle prep (the pinned exact-ZOH injection (1 - rho)/lambda)."""
    s = synth.Shape(1, 200, 4, 64, 1, 64, 8, 0, "bf16")
    host = synth.make_prep_inputs(s, seed=9)
    x = synth.cast(synth.normal(9, "x", (1, 200, 4, 64)), "bf16")
    Bm = synth.cast(synth.normal(9, "B", (1, 200, 1, 64)), "bf16")
    Cm = synth.cast(synth.normal(9, "C", (1, 200, 1, 64)), "bf16")
    D = synth.normal(9, "D", (4,))
    d = dev_inputs(dict(host, x=x, B=Bm, C=Cm, D=D))
    cfg, cfg64 = _cfgs(pp.ZOH_INJECTION)
    o = param_prep_fwd(d["dt_raw"], d["alpha_raw"], d["lam_raw"], d["g_read"], d["g_write"],
                       d["tau"], d["dt_bias"], cfg)
    y, hf = scan_fwd(d["x"], o["dt"], o["alpha"], o["lam"], d["tau"], d["B"], d["C"],
                     o["w_read"], o["w_write"], d["D"])
    torch.cuda.synchronize()
    h64 = f64_inputs(dict(host, x=x, B=Bm, C=Cm, D=D))
    r = pp.prep_fwd(h64["dt_raw"], h64["alpha_raw"], h64["lam_raw"], h64["g_read"],
                    h64["g_write"], h64["tau"], h64["dt_bias"], cfg64)
    yr, hr = oracle.fwd(h64["x"], r["dt"], r["alpha"], r["lam"], h64["tau"], h64["B"], h64["C"],
                        r["w_read"], r["w_write"], h64["D"])
    assert_close("y", to_host64(y), yr, 1e-2)
    assert_close("h_final", to_host64(hf), hr, 1e-2)
