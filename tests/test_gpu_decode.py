"""GPU parity of the decode step (Algorithm 1, one token with the cached state)."""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2609_36314_gb300 import decode_step, scan_fwd, synth
from tests.gpu_util import assert_close, dev_inputs, f64_inputs, to_dev, to_host64, tol

pytestmark = pytest.mark.gpu


def _step_inputs(dv, t):
    return {k: (v[t] if k not in ("tau", "D") else v) for k, v in dv.items()}


def _run_decode(shape, steps, seed, state_host):
    dec = synth.make_decode_inputs(shape, steps, seed=seed)
    dv = dev_inputs(dec)
    state = to_dev(state_host.astype(np.float32)).clone()
    ys = []
    for t in range(steps):
        s = _step_inputs(dv, t)
        ys.append(decode_step(s["x"], s["dt"], s["alpha"], s["lam"], s["tau"], s["B"], s["C"],
                              s["w_read"], s["w_write"], s["D"], state))
    torch.cuda.synchronize()
    return dec, torch.stack(ys), state


def _oracle_decode(dec, state0, steps, bsel=None, hsel=None):
    d = f64_inputs(dec)
    st = state0.astype(np.float64)
    ys = []
    for t in range(steps):
        x, dt, al, lm = d["x"][t], d["dt"][t], d["alpha"][t], d["lam"][t]
        Bt, Ct, wr, ww = d["B"][t], d["C"][t], d["w_read"][t], d["w_write"][t]
        tau, D = d["tau"], d["D"]
        if bsel is not None:
            x, dt, al, lm, wr, ww = (a[bsel][:, hsel] for a in (x, dt, al, lm, wr, ww))
            Bt, Ct = Bt[bsel], Ct[bsel]
            tau, D = tau[hsel], D[hsel]
        y, st = oracle.decode(x, dt, al, lm, tau, Bt, Ct, wr, ww, D, st)
        ys.append(y)
    return np.stack(ys), st


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("N", [128, 20])
def test_decode_steps_match_oracle(dtype, N):
    s = synth.Shape(3, 0, 4, 16, 2, N, 5, 0, dtype)
    rng = np.random.default_rng(1)
    st0 = (0.3 * rng.standard_normal((3, 4, 5, 16, N))).astype(np.float32)
    dec, y, st = _run_decode(s, 12, 2, st0)
    yr, str_ = _oracle_decode(dec, st0, 12)
    t = tol(dtype)
    assert_close("y", to_host64(y), yr, t)
    assert_close("state", to_host64(st), str_, 1e-5)


def test_prefill_then_decode_equals_longer_prefill():
    """scan(L1) + (L2 single-token steps) == scan(L1 + L2) on the GPU (decode hand-off)."""
    s = synth.Shape(2, 40, 4, 32, 1, 64, 8, 0, "f32")
    host = synth.make_scan_inputs(s, seed=4)
    dv = dev_inputs(host)
    y_all, h_all = scan_fwd(dv["x"], dv["dt"], dv["alpha"], dv["lam"], dv["tau"], dv["B"],
                            dv["C"], dv["w_read"], dv["w_write"], dv["D"])
    L1 = 29
    sl = lambda v: v[:, :L1].contiguous()
    y1, h1 = scan_fwd(sl(dv["x"]), sl(dv["dt"]), sl(dv["alpha"]), sl(dv["lam"]), dv["tau"],
                      sl(dv["B"]), sl(dv["C"]), sl(dv["w_read"]), sl(dv["w_write"]), dv["D"])
    state = h1.clone()
    for t in range(L1, s.seqlen):
        yt = decode_step(dv["x"][:, t].contiguous(), dv["dt"][:, t].contiguous(),
                         dv["alpha"][:, t].contiguous(), dv["lam"][:, t].contiguous(), dv["tau"],
                         dv["B"][:, t].contiguous(), dv["C"][:, t].contiguous(),
                         dv["w_read"][:, t].contiguous(), dv["w_write"][:, t].contiguous(),
                         dv["D"], state)
        assert_close(f"y[{t}]", to_host64(yt), to_host64(y_all[:, t]), 1e-5)
    assert_close("state", to_host64(state), to_host64(h_all), 1e-5)


@pytest.mark.slow
def test_decode_workload_sampled():
    """B128 H64 P64 N128 K8: 512-token prefill then 1024 decode steps at full size; 16 (b, h)
    streams are replayed by the oracle from the GPU prefill's input bytes."""
    s = synth.WORKLOADS["decode_b128"]
    host = synth.make_scan_inputs(s, seed=0)
    dv = dev_inputs(host)
    _, hf = scan_fwd(dv["x"], dv["dt"], dv["alpha"], dv["lam"], dv["tau"], dv["B"], dv["C"],
                     dv["w_read"], dv["w_write"], dv["D"])
    del dv
    steps = synth.DECODE_STEPS
    dec = synth.make_decode_inputs(s, steps, seed=0)
    ddev = dev_inputs(dec)
    state = hf
    bsel = np.array([0, 17, 64, 127])
    hsel = np.array([0, 9, 33, 63])
    bt, ht = torch.tensor(bsel, device="cuda"), torch.tensor(hsel, device="cuda")
    ys = []
    for t in range(steps):
        st = _step_inputs(ddev, t)
        y = decode_step(st["x"], st["dt"], st["alpha"], st["lam"], st["tau"], st["B"], st["C"],
                        st["w_read"], st["w_write"], st["D"], state)
        ys.append(y[bt][:, ht])
    torch.cuda.synchronize()
    # oracle: its own prefill of the sampled streams, then the same steps
    pre = {k: synth.to_f64(v) for k, v in host.items()}
    sub = dict(x=pre["x"][bsel][:, :, hsel], dt=pre["dt"][bsel][:, :, hsel],
               alpha=pre["alpha"][bsel][:, :, hsel], lam=pre["lam"][bsel][:, :, hsel],
               w_read=pre["w_read"][bsel][:, :, hsel], w_write=pre["w_write"][bsel][:, :, hsel],
               B=pre["B"][bsel], C=pre["C"][bsel], tau=pre["tau"][hsel], D=pre["D"][hsel])
    _, h_or = oracle.fwd(sub["x"], sub["dt"], sub["alpha"], sub["lam"], sub["tau"], sub["B"],
                         sub["C"], sub["w_read"], sub["w_write"], sub["D"])
    yr, st_r = _oracle_decode(dec, h_or, steps, bsel, hsel)
    got = torch.stack(ys)
    assert_close("y", to_host64(got), yr, 1e-2)
    assert_close("state", to_host64(state[bt][:, ht]), st_r, 1e-2)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_decode_paper_layer_shape(dtype):
    """The paper's layer (H16, head dim 256, N = 1, K = 16 on the 1 .. 2^17 bank): a 300-token
    prefill through the chunk-parallel N = 1 forward, then 16 decode steps (Algorithm 1's
    one-step form), against the oracle's prefill and steps on the same bytes."""
    s = synth.Shape(2, 300, 16, 256, 1, 1, 16, 0, dtype)
    host = synth.make_scan_inputs(s, seed=12)
    dv = dev_inputs(host)
    _, hf = scan_fwd(dv["x"], dv["dt"], dv["alpha"], dv["lam"], dv["tau"], dv["B"], dv["C"],
                     dv["w_read"], dv["w_write"], dv["D"])
    dec, y, st = _run_decode(s, 16, 13, to_host64(hf))
    o = f64_inputs(host)
    _, h_or = oracle.fwd(o["x"], o["dt"], o["alpha"], o["lam"], o["tau"], o["B"], o["C"],
                         o["w_read"], o["w_write"], o["D"])
    assert_close("prefill state", to_host64(hf), h_or, tol(dtype))
    yr, str_ = _oracle_decode(dec, h_or, 16)
    assert_close("y", to_host64(y), yr, tol(dtype))
    assert_close("state", to_host64(st), str_, tol(dtype))


@pytest.mark.parametrize("K,P,G", [(5, 40, 1), (1, 33, 1), (4, 64, 2)])
def test_decode_n1_shapes(K, P, G):
    """N = 1 decode (one thread per (b, h, p)) off the paper's shape: odd mode counts, a single
    mode, head dims that are not a multiple of 32, B/C groups; float32 and 8 steps."""
    s = synth.Shape(3, 40, 4, P, G, 1, K, 0, "f32")
    host = synth.make_scan_inputs(s, seed=60 + K)
    dv = dev_inputs(host)
    _, hf = scan_fwd(dv["x"], dv["dt"], dv["alpha"], dv["lam"], dv["tau"], dv["B"], dv["C"],
                     dv["w_read"], dv["w_write"], dv["D"])
    dec, y, st = _run_decode(s, 8, 61 + K, to_host64(hf))
    o = f64_inputs(host)
    _, h_or = oracle.fwd(o["x"], o["dt"], o["alpha"], o["lam"], o["tau"], o["B"], o["C"],
                         o["w_read"], o["w_write"], o["D"])
    yr, str_ = _oracle_decode(dec, h_or, 8)
    assert_close("y", to_host64(y), yr, tol("f32"))
    assert_close("state", to_host64(st), str_, tol("f32"))
