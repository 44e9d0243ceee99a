"""GPU parity of the chunked scan (forward and backward) against the fp64 oracle.

Inputs are the seeded synthetic workloads; the CUDA path runs through the C ABI
(libfrac.so via the thin binding) and is compared element by element with the
oracle on the same bytes.  Tolerances (relative L2 per output tensor): 1e-5 on the
float32 path, 1e-2 for bf16 inputs with float32 accumulation.
"""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2609_36314_gb300 import scan_bwd, scan_fwd, synth
from tests.gpu_util import assert_close, dev_inputs, f64_inputs, to_host64, tol

pytestmark = pytest.mark.gpu

GRADS = ["dx", "ddt", "dalpha", "dlam", "dB", "dC", "dw_read", "dw_write", "dD", "dh0"]


def _gpu_fwd(dv, **kw):
    return scan_fwd(dv["x"], dv["dt"], dv["alpha"], dv["lam"], dv["tau"], dv["B"], dv["C"],
                    dv["w_read"], dv["w_write"], dv["D"], dv.get("h0"), **kw)


def _gpu_bwd(dv, **kw):
    return scan_bwd(dv["x"], dv["dt"], dv["alpha"], dv["lam"], dv["tau"], dv["B"], dv["C"],
                    dv["w_read"], dv["w_write"], dv["D"], dv["dy"], dv.get("h0"),
                    dv.get("dh_final"), **kw)


def _ora_fwd(d):
    return oracle.fwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"],
                      d["w_read"], d["w_write"], d["D"], d.get("h0"))


def _ora_bwd(d):
    return oracle.bwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"],
                      d["w_read"], d["w_write"], d["D"], d["dy"], h0=d.get("h0"),
                      dh_final=d.get("dh_final"))


def _check_fwd(shape, seed=0, h0=False, **kw):
    host = synth.make_scan_inputs(shape, seed=seed, with_h0=h0)
    dv = dev_inputs(host)
    y, hf = _gpu_fwd(dv, **kw)
    torch.cuda.synchronize()
    yr, hfr = _ora_fwd(f64_inputs(host))
    t = tol(shape.dtype)
    assert_close("y", to_host64(y), yr, t)
    assert_close("h_final", to_host64(hf), hfr, t)


def _check_bwd(shape, seed=0, h0=False, dhf=False, **kw):
    host = synth.make_scan_inputs(shape, seed=seed, with_dy=True, with_h0=h0, with_dh_final=dhf)
    dv = dev_inputs(host)
    g = _gpu_bwd(dv, **kw)
    torch.cuda.synchronize()
    gr = _ora_bwd(f64_inputs(host))
    t = tol(shape.dtype)
    for k in GRADS:
        assert_close(k, to_host64(g[k]), gr[k], t)


# ------------------------------------------------------------------ float32 path (1e-5)
def test_fwd_f32_small_workload():
    """B1 L256 H2 P32 N16 K4, chunk 64, float32."""
    _check_fwd(synth.WORKLOADS["fwd_f32_small"], chunk=64)


@pytest.mark.parametrize("chunk", [16, 32, 64])
@pytest.mark.parametrize("L", [1, 37, 100, 128])
def test_fwd_f32_chunks_and_ragged_lengths(chunk, L):
    s = synth.Shape(2, L, 4, 24, 2, 12, 3, chunk, "f32")
    _check_fwd(s, seed=L, h0=True, chunk=chunk)


@pytest.mark.parametrize("chunk", [16, 64])
def test_bwd_f32(chunk):
    s = synth.Shape(2, 150, 4, 16, 2, 12, 3, chunk, "f32")
    _check_bwd(s, seed=3, h0=True, dhf=True, chunk=chunk)


def test_bwd_f32_small_workload_shape():
    s = synth.WORKLOADS["fwd_f32_small"]
    _check_bwd(s, seed=1, chunk=64)


def test_odd_sizes_f32():
    """N not a multiple of 4, P not a multiple of 8, one head, K = 1."""
    _check_fwd(synth.Shape(1, 45, 1, 5, 1, 5, 1, 0, "f32"), seed=9, h0=True)
    _check_bwd(synth.Shape(1, 45, 1, 5, 1, 5, 1, 0, "f32"), seed=9, h0=True, dhf=True)


def test_empty_sequence():
    s = synth.Shape(2, 0, 3, 8, 1, 4, 2, 0, "f32")
    host = synth.make_scan_inputs(s, with_h0=True, with_dy=True, with_dh_final=True)
    dv = dev_inputs(host)
    y, hf = _gpu_fwd(dv)
    assert y.numel() == 0
    assert torch.equal(hf, dv["h0"])
    g = _gpu_bwd(dv)
    assert torch.equal(g["dh0"], dv["dh_final"])
    assert torch.count_nonzero(g["dD"]) == 0


# ------------------------------------------------------------------ bf16 path (1e-2)
def test_fwd_bf16_b4_l2048_workload():
    """B4 L2048 H16 P64 N64 K8, chunk 128 requested by the workload: full-size parity."""
    s = synth.WORKLOADS["fwd_bf16_b4_l2048"]
    _check_fwd(s)


@pytest.mark.parametrize("L", [1, 63, 200])
def test_fwd_bf16_ragged(L):
    _check_fwd(synth.Shape(2, L, 4, 64, 1, 64, 8, 0, "bf16"), seed=L, h0=True)


def test_bwd_bf16_medium():
    _check_bwd(synth.Shape(2, 300, 4, 64, 1, 64, 8, 0, "bf16"), seed=5, h0=True, dhf=True)


def test_bwd_bf16_groups():
    _check_bwd(synth.Shape(1, 130, 4, 32, 2, 32, 4, 0, "bf16"), seed=6)


@pytest.mark.parametrize("N,K,G", [(128, 4, 1), (64, 4, 2), (128, 8, 2)])
def test_tensor_path_modes_and_groups(N, K, G):
    """bf16, headdim 64: every (N, K) the tensor-core kernels take, with B/C groups; the trace
    shows that the tensor-core kernels ran."""
    from paper_2609_36314_gb300 import _lib
    s = synth.Shape(2, 200, 4, 64, G, N, K, 0, "bf16")
    _lib.trace_reset()
    _lib.trace_enable(True)
    try:
        _check_fwd(s, seed=20 + N + K, h0=True)
        _check_bwd(s, seed=30 + N + K, h0=True, dhf=True)
        names = set(_lib.trace_collect())
    finally:
        _lib.trace_enable(False)
    assert {"state_pass_fwd_tc", "chunk_fwd_tc", "state_pass_rev_tc", "bwd_intra_tc"} <= names


def test_tensor_path_sixteen_heads_per_group():
    """bf16, sixteen heads sharing B/C: the state-term backward takes all sixteen heads of the
    group in one CTA (fifteen head switches with staged inputs), on a ragged sequence."""
    s = synth.Shape(1, 200, 16, 64, 1, 128, 8, 0, "bf16")
    _check_fwd(s, seed=41, h0=True)
    _check_bwd(s, seed=42, h0=True, dhf=True)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_paper_layer_shape(dtype):
    """The paper's own layer shape, cut to two heads and 300 tokens: head dim 256, N = 1, K = 16
    modes on the geometric 1 .. 2^17 bank (the CUDA-core path)."""
    s = synth.Shape(1, 300, 2, 256, 1, 1, 16, 0, dtype)
    _check_fwd(s, seed=50, h0=True)
    _check_bwd(s, seed=51, h0=True, dhf=True)


@pytest.mark.parametrize("shape", [
    synth.Shape(2, 77, 3, 200, 1, 1, 5, 16, "f32"),   # K = 5 (per-mode loop), two p blocks, ragged
    synth.Shape(1, 130, 2, 64, 2, 1, 8, 32, "bf16"),  # one head per B/C group, chunk 32
    synth.Shape(1, 0, 2, 32, 1, 1, 4, 0, "f32"),      # empty sequence: h_final = h0
])
def test_n1_forward_shapes(shape):
    """N = 1 forward (the direct per-mode recurrence): mode counts off a multiple of 4, p blocks
    past the head dimension, groups, chunk sizes, ragged and empty sequences."""
    _check_fwd(shape, seed=60 + shape.nmodes, h0=True)


def test_force_simt_matches_default_path():
    s = synth.Shape(2, 260, 4, 64, 1, 128, 8, 0, "bf16")
    host = synth.make_scan_inputs(s, seed=12, with_dy=True)
    dv = dev_inputs(host)
    y0, h0 = _gpu_fwd(dv)
    y1, h1 = _gpu_fwd(dv, force_simt=True)
    torch.cuda.synchronize()
    yr, hr = _ora_fwd(f64_inputs(host))
    assert_close("y default", to_host64(y0), yr, 1e-2)
    assert_close("y simt", to_host64(y1), yr, 1e-2)
    assert_close("h default", to_host64(h0), hr, 1e-2)
    assert_close("h simt", to_host64(h1), hr, 1e-2)


# ------------------------------------------------------------------ full-size workloads, sampled
def _slice_streams(host, b, heads):
    """Oracle inputs for batch row b and a subset of heads (B/C groups kept whole; G = 1)."""
    out = {}
    for k, v in host.items():
        a = synth.to_f64(v)
        if k in ("x", "dy", "w_read", "w_write", "dt", "alpha", "lam"):
            out[k] = a[b:b + 1][:, :, heads]
        elif k in ("B", "C"):
            out[k] = a[b:b + 1]
        elif k in ("tau",):
            out[k] = a[heads]
        elif k == "D":
            out[k] = a[heads]
        else:
            out[k] = a
    return out


@pytest.mark.slow
def test_train_workload_fwd_bwd_sampled():
    """B8 L4096 H64 P64 N128 K8 bf16 at full size, in the configuration the benchmark times: one
    workspace for both calls, the backward reusing the forward's per-chunk states.  y, h_final and
    every per-stream gradient are compared on four (batch, head) streams in two batch rows; dy is
    zero outside those streams so that dB, dC (sums over a row's heads) and dD are exactly the
    sampled streams' contributions, which the oracle computes."""
    from paper_2609_36314_gb300.api import bwd_workspace_size, fwd_workspace_size, make_dims
    s = synth.WORKLOADS["train_bf16_b8_l4096"]
    host = synth.make_scan_inputs(s, seed=0, with_dy=True)
    sample = {3: [5, 37], 6: [12, 60]}
    mask = np.zeros((s.batch, 1, s.nheads, 1), dtype=bool)
    for b, heads in sample.items():
        mask[b, 0, heads] = True
    dy = synth.bf16_bits_to_f32(host["dy"]) * mask
    host["dy"] = synth.f32_to_bf16_bits(dy)
    dv = dev_inputs(host)
    dims = make_dims(s.batch, s.seqlen, s.nheads, s.headdim, s.ngroups, s.dstate, s.nmodes,
                     torch.bfloat16)
    ws = torch.empty(max(bwd_workspace_size(dims), fwd_workspace_size(dims)), dtype=torch.uint8,
                     device="cuda")
    y, hf = _gpu_fwd(dv, workspace=ws)
    g = _gpu_bwd(dv, workspace=ws, reuse_fwd_states=True)
    torch.cuda.synchronize()
    dD = np.zeros(s.nheads)
    for b, heads in sample.items():
        sub = _slice_streams(host, b, heads)
        yr, hfr = _ora_fwd(sub)
        gr = _ora_bwd(sub)
        assert_close("y", to_host64(y[b:b + 1][:, :, heads]), yr, 1e-2)
        assert_close("h_final", to_host64(hf[b:b + 1][:, heads]), hfr, 1e-2)
        for k in ("dx", "dw_read", "dw_write", "ddt", "dalpha", "dlam"):
            assert_close(k, to_host64(g[k][b:b + 1][:, :, heads]), gr[k], 1e-2)
        assert_close("dh0", to_host64(g["dh0"][b:b + 1][:, heads]), gr["dh0"], 1e-2)
        assert_close("dB", to_host64(g["dB"][b:b + 1]), gr["dB"], 1e-2)
        assert_close("dC", to_host64(g["dC"][b:b + 1]), gr["dC"], 1e-2)
        dD[heads] += gr["dD"]
    hs = sorted({h for heads in sample.values() for h in heads})
    assert_close("dD", to_host64(g["dD"][hs]), dD[hs], 1e-2)
    # rows outside the sample got no upstream gradient
    other = torch.ones(s.batch, dtype=torch.bool)
    other[list(sample)] = False
    assert torch.count_nonzero(g["dB"][other]) == 0


def test_nonfinite_input_stays_in_its_stream():
    """A NaN in one element of x (batch 1, head 2, channel 5, position 300 of a ragged 3-chunk
    sequence) on the tensor-core path: y of every other (batch, head) stream and of every other
    channel of the stream stays finite, and so do the positions of the chunks before the NaN's
    chunk; y of that channel is NaN from the NaN's position on.  Inside its chunk the NaN may also
    reach the positions before it (the chunk's intra-chunk product multiplies the masked-out
    coefficients by it), which the sequential recurrence would not do."""
    s = synth.Shape(2, 330, 4, 64, 1, 128, 8, 0, "bf16")
    host = synth.make_scan_inputs(s, seed=13)
    x = synth.bf16_bits_to_f32(host["x"]).copy()
    b, h, p, t = 1, 2, 5, 300
    x[b, t, h, p] = np.nan
    host["x"] = synth.f32_to_bf16_bits(x)
    dv = dev_inputs(host)
    y, hf = _gpu_fwd(dv)
    torch.cuda.synchronize()
    yy = to_host64(y)
    bad = np.isnan(yy)
    keep = np.ones_like(bad)
    keep[b, :, h, p] = False
    assert not bad[keep].any()
    assert bad[b, t:, h, p].all()
    c0 = (t // 128) * 128
    assert not bad[b, :c0, h, p].any()


def _heads_per_bwd_state_cta(B, L, H, G, sms, chunk=128):
    """The host's choice of heads per CTA for the state-term backward: the largest divisor (at
    most 16) of a group's heads that still leaves two waves of CTAs, else the largest divisor."""
    hpg, nc = H // G, (L + chunk - 1) // chunk
    divisors = [hg for hg in range(1, 17) if hpg % hg == 0]
    fits = [hg for hg in divisors if (H // hg) * nc * B >= 2 * sms]
    return (fits or divisors)[-1], divisors[-1]


def test_bwd_state_fewer_heads_per_cta_sampled():
    """B4 L2048 H16 P64 N64 K8 bf16 (the forward workload's shape) through the backward: here the
    state-term backward takes fewer heads per CTA than the largest divisor of the group (two
    instead of sixteen, so that at least two waves of CTAs remain).  Two (batch, head) streams are
    compared with the oracle, dy zero elsewhere as in the training-shape test."""
    s = synth.WORKLOADS["fwd_bf16_b4_l2048"]
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    hg, largest = _heads_per_bwd_state_cta(s.batch, s.seqlen, s.nheads, s.ngroups, sms)
    assert hg < largest, (hg, largest)
    host = synth.make_scan_inputs(s, seed=4, with_dy=True)
    b, heads = 2, [3, 12]
    mask = np.zeros((s.batch, 1, s.nheads, 1), dtype=bool)
    mask[b, 0, heads] = True
    host["dy"] = synth.f32_to_bf16_bits(synth.bf16_bits_to_f32(host["dy"]) * mask)
    dv = dev_inputs(host)
    g = _gpu_bwd(dv)
    torch.cuda.synchronize()
    sub = _slice_streams(host, b, heads)
    gr = _ora_bwd(sub)
    for k in ("dx", "dw_read", "dw_write", "ddt", "dalpha", "dlam"):
        assert_close(k, to_host64(g[k][b:b + 1][:, :, heads]), gr[k], 1e-2)
    assert_close("dh0", to_host64(g["dh0"][b:b + 1][:, heads]), gr["dh0"], 1e-2)
    assert_close("dB", to_host64(g["dB"][b:b + 1]), gr["dB"], 1e-2)
    assert_close("dC", to_host64(g["dC"][b:b + 1]), gr["dC"], 1e-2)
    assert_close("dD", to_host64(g["dD"][heads]), gr["dD"], 1e-2)


@pytest.mark.slow
def test_long_prefill_workload_sampled():
    """B1 L65536 H64 P64 N128 K8 bf16, Delta skewed small: y and h_final of two heads."""
    s = synth.WORKLOADS["prefill_bf16_l65536"]
    host = synth.make_scan_inputs(s, seed=0)
    dv = dev_inputs(host)
    y, hf = _gpu_fwd(dv)
    torch.cuda.synchronize()
    heads = [0, 50]
    sub = _slice_streams(host, 0, heads)
    yr, hfr = _ora_fwd(sub)
    assert_close("y", to_host64(y[:, :, heads]), yr, 1e-2)
    assert_close("h_final", to_host64(hf[:, heads]), hfr, 1e-2)


def test_bwd_tensor_core_path_matches_cuda_core_path():
    """bf16, P = 64: the default (tensor-core) backward and the CUDA-core backward against the
    oracle, with h0 and dh_final, a ragged last chunk and several chunks."""
    s = synth.Shape(2, 300, 4, 64, 1, 128, 8, 0, "bf16")
    host = synth.make_scan_inputs(s, seed=21, with_dy=True, with_h0=True, with_dh_final=True)
    dv = dev_inputs(host)
    g_tc = _gpu_bwd(dv)
    g_simt = _gpu_bwd(dv, force_simt=True)
    torch.cuda.synchronize()
    gr = _ora_bwd(f64_inputs(host))
    for k in GRADS:
        assert_close(k + " (tensor cores)", to_host64(g_tc[k]), gr[k], 1e-2)
        assert_close(k + " (CUDA cores)", to_host64(g_simt[k]), gr[k], 1e-2)


def test_bwd_bf16_paper_like_lambda_alpha_extremes():
    """Small alpha and large lambda make e = Delta lambda^(1/alpha) huge (clamped) on some
    positions; the decay gradient must stay accurate there (per-position decayed terms)."""
    s = synth.Shape(1, 256, 4, 64, 1, 64, 8, 0, "bf16")
    host = synth.make_scan_inputs(s, seed=33, with_dy=True)
    host["alpha"] = (host["alpha"] * 0.25).astype(np.float32)   # alpha in (0, 0.25)
    host["lam"] = np.full_like(host["lam"], 3.5)
    host["w_read"] = synth.cast(synth.mode_weights(host["alpha"], host["tau"], synth.normal(33, "w_read", (1, 256, 4, 8))), "bf16")
    host["w_write"] = synth.cast(synth.mode_weights(host["alpha"], host["tau"], synth.normal(33, "w_write", (1, 256, 4, 8))), "bf16")
    dv = dev_inputs(host)
    g = _gpu_bwd(dv)
    torch.cuda.synchronize()
    gr = _ora_bwd(f64_inputs(host))
    for k in GRADS:
        assert_close(k, to_host64(g[k]), gr[k], 1e-2)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_bwd_reusing_forward_states(dtype):
    """The backward may take the per-chunk states the forward left in a shared workspace."""
    from paper_2609_36314_gb300 import bwd_workspace_size, fwd_workspace_size, make_dims
    s = synth.Shape(2, 260, 4, 64, 1, 64, 8, 0, dtype)
    host = synth.make_scan_inputs(s, seed=44, with_dy=True, with_h0=True)
    dv = dev_inputs(host)
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    dims = make_dims(2, 260, 4, 64, 1, 64, 8, tdt)
    ws = torch.empty(max(bwd_workspace_size(dims), fwd_workspace_size(dims)), dtype=torch.uint8,
                     device="cuda")
    _gpu_fwd(dv, workspace=ws)
    g = _gpu_bwd(dv, workspace=ws, reuse_fwd_states=True)
    g_ref = _gpu_bwd(dv)
    torch.cuda.synchronize()
    for k in GRADS:
        assert torch.equal(g[k], g_ref[k]) or synth.rel_l2(to_host64(g[k]), to_host64(g_ref[k])) < 1e-6, k


# ------------------------------------------------------------------ learned timescales (dtau)
def _learned_tau(d64, dv, seed):
    """Per-head timescales off the geometric grid (the learned-timescale variant, App. G)."""
    rng = np.random.default_rng(seed)
    tau = (d64["tau"] * np.exp(0.3 * rng.standard_normal(d64["tau"].shape))).astype(np.float32)
    d64["tau"] = tau.astype(np.float64)
    dv["tau"] = torch.from_numpy(tau).cuda()


@pytest.mark.parametrize("dtype,shape", [
    ("f32", synth.Shape(2, 150, 3, 16, 1, 8, 4, 32, "f32")),          # CUDA-core path
    ("bf16", synth.Shape(2, 260, 4, 64, 1, 64, 8, 0, "bf16")),        # tensor-core path
    ("bf16", synth.Shape(1, 300, 4, 64, 2, 128, 4, 0, "bf16")),       # tensor-core, K = 4, G = 2
    ("f32", synth.Shape(1, 200, 2, 256, 1, 1, 16, 0, "f32")),         # the paper's N = 1 shape
    ("bf16", synth.Shape(2, 200, 2, 256, 1, 1, 16, 0, "bf16")),       # N = 1, tensor-core gradients
])
def test_bwd_timescale_gradient(dtype, shape):
    host = synth.make_scan_inputs(shape, seed=31, with_dy=True, with_h0=True, with_dh_final=True)
    d64 = f64_inputs(host)
    dv = dev_inputs(host)
    _learned_tau(d64, dv, 32)
    g = _gpu_bwd(dv, chunk=shape.chunk, want_dtau=True)
    torch.cuda.synchronize()
    ref = _ora_bwd(d64)
    assert_close("dtau", to_host64(g["dtau"]), ref["dtau"], tol(dtype))
    assert_close("ddt", to_host64(g["ddt"]), ref["ddt"], tol(dtype))


def test_bwd_timescale_gradient_reusing_forward_states():
    """The benchmarked mode (one workspace, the backward reusing the forward's states) with
    the timescale gradient, on the tensor-core path."""
    s = synth.Shape(2, 384, 4, 64, 1, 128, 8, 0, "bf16")
    host = synth.make_scan_inputs(s, seed=33, with_dy=True)
    d64 = f64_inputs(host)
    dv = dev_inputs(host)
    _learned_tau(d64, dv, 34)
    from paper_2609_36314_gb300.api import bwd_workspace_size, fwd_workspace_size, make_dims
    dims = make_dims(s.batch, s.seqlen, s.nheads, s.headdim, s.ngroups, s.dstate, s.nmodes,
                     torch.bfloat16)
    ws = torch.empty(max(bwd_workspace_size(dims), fwd_workspace_size(dims)), dtype=torch.uint8,
                     device="cuda")
    _gpu_fwd(dv, workspace=ws, want_final_state=False)
    g = _gpu_bwd(dv, workspace=ws, reuse_fwd_states=True, want_dtau=True)
    torch.cuda.synchronize()
    ref = _ora_bwd(d64)
    for k in GRADS + ["dtau"]:
        assert_close(k, to_host64(g[k]), ref[k], 1e-2)


def test_paper_layer_shape_all_heads_long():
    """All 16 heads of the paper's layer at 4096 tokens (64 chunks through the chunk-parallel
    N = 1 forward's local pass, serial combine and output pass), every output compared."""
    s = synth.Shape(1, 4096, 16, 256, 1, 1, 16, 0, "bf16")
    _check_fwd(s, seed=52, h0=True)


def test_paper_layer_shape_backward_reusing_forward_states():
    """One buffer of frac_scan_bwd_workspace_size serves the N = 1 forward (whose scratch holds
    the chunk-local states) and the backward that reuses its per-chunk states."""
    from paper_2609_36314_gb300.api import bwd_workspace_size, make_dims
    s = synth.Shape(1, 700, 4, 256, 1, 1, 16, 0, "bf16")
    host = synth.make_scan_inputs(s, seed=53, with_dy=True)
    dv = dev_inputs(host)
    dims = make_dims(s.batch, s.seqlen, s.nheads, s.headdim, s.ngroups, s.dstate, s.nmodes,
                     torch.bfloat16)
    ws = torch.empty(bwd_workspace_size(dims), dtype=torch.uint8, device="cuda")
    y, _ = _gpu_fwd(dv, workspace=ws, want_final_state=False)
    g = _gpu_bwd(dv, workspace=ws, reuse_fwd_states=True)
    torch.cuda.synchronize()
    d64 = f64_inputs(host)
    yr, _ = _ora_fwd(d64)
    assert_close("y", to_host64(y), yr, 1e-2)
    ref = _ora_bwd(d64)
    for k in GRADS:
        assert_close(k, to_host64(g[k]), ref[k], 1e-2)


@pytest.mark.parametrize("shape", [
    synth.Shape(2, 77, 3, 200, 1, 1, 5, 16, "f32"),   # K = 5, P off a multiple of 256, chunk 16, ragged
    synth.Shape(1, 130, 2, 64, 2, 1, 8, 32, "bf16"),  # one head per B/C group
    synth.Shape(1, 96, 4, 256, 2, 1, 16, 0, "f32"),   # two heads per group, whole chunks
    synth.Shape(1, 0, 2, 32, 1, 1, 4, 0, "f32"),      # empty sequence: dh0 = dh_final
])
def test_n1_backward_shapes(shape):
    """N = 1 backward (reverse chunk carries and the per-chunk gradient kernel): mode counts off a
    multiple of 4, p blocks past the head dimension, groups (dB, dC summed over their heads),
    chunk sizes, ragged and empty sequences."""
    _check_bwd(shape, seed=70 + shape.nmodes, h0=True, dhf=True, chunk=shape.chunk)


@pytest.mark.parametrize("shape", [
    synth.Shape(2, 75, 4, 128, 2, 1, 4, 0, "bf16"),    # K = 4, P = 128, two sequences with ragged ends, groups
    synth.Shape(1, 150, 2, 256, 1, 1, 5, 0, "bf16"),   # K = 5 (eight lanes per row), ragged
    synth.Shape(1, 96, 2, 384, 1, 1, 16, 0, "bf16"),   # P = 384: three 128-wide dx tiles, whole chunks
    synth.Shape(1, 70, 2, 128, 1, 1, 20, 0, "bf16"),   # K = 20 (32-row mode slots, 32 lanes per row)
    synth.Shape(1, 20, 3, 256, 1, 1, 16, 0, "bf16"),   # one chunk, shorter than 32
])
def test_n1_backward_tensor_core_variant(shape):
    """bf16 N = 1 backward with the head dimension a multiple of 128: the per-chunk gradient kernel
    whose contractions over p and over positions run on tcgen05 (the trace shows it ran), for each
    mode-slot layout, tile count and ragged or short sequence."""
    from paper_2609_36314_gb300 import _lib
    _lib.trace_reset()
    _lib.trace_enable(True)
    try:
        _check_bwd(shape, seed=90 + shape.nmodes, h0=True, dhf=True)
        names = set(_lib.trace_collect())
    finally:
        _lib.trace_enable(False)
    assert "chunk_bwd_n1_tc" in names and "chunk_bwd_n1" not in names
