"""The bounded device waits give up cleanly and the caller sees it.

Every mbarrier wait in the tensor-core kernels has a time limit; a kernel whose wait runs out
records FRAC_ERR_TIMEOUT in the call's status word, frees its tensor memory and returns, so the
CUDA context stays usable.  FRAC_FLAG_TEST_EXPIRE_WAIT makes the forward state pass wait about a
millisecond on a barrier that nothing signals (before it has issued any copy or MMA), which
takes exactly that path without faulting anything.  The test reads the status back through
frac_workspace_status and then checks that a normal call on the same workspace succeeds and
still matches the oracle.
"""
import ctypes

import pytest
import torch

from oracle import oracle
from paper_2609_36314_gb300 import _lib, synth
from paper_2609_36314_gb300.api import _ptr, _stream, fwd_workspace_size, make_dims
from tests.gpu_util import assert_close, dev_inputs, f64_inputs, to_host64

pytestmark = pytest.mark.gpu

FRAC_ERR_UNSUPPORTED = 2
FRAC_ERR_TIMEOUT = 4


def _fwd(dims, d, y, hf, ws):
    return _lib.load().frac_scan_fwd(
        ctypes.byref(dims), _ptr(d["x"]), _ptr(d["dt"]), _ptr(d["alpha"]), _ptr(d["lam"]),
        _ptr(d["tau"]), _ptr(d["B"]), _ptr(d["C"]), _ptr(d["w_read"]), _ptr(d["w_write"]),
        _ptr(d["D"]), None, _ptr(y), _ptr(hf), _ptr(ws), ws.numel(), _stream(None))


def test_expired_wait_is_reported_and_the_next_call_succeeds():
    s = synth.Shape(1, 300, 2, 64, 1, 64, 8, 0, "bf16")
    host = synth.make_scan_inputs(s, seed=5)
    d = dev_inputs(host)
    y = torch.empty_like(d["x"])
    hf = torch.empty((s.batch, s.nheads, s.nmodes, s.headdim, s.dstate), dtype=torch.float32,
                     device="cuda")
    args = (s.batch, s.seqlen, s.nheads, s.headdim, s.ngroups, s.dstate, s.nmodes, torch.bfloat16)
    dims_expire = make_dims(*args, extra_flags=_lib.FRAC_FLAG_TEST_EXPIRE_WAIT)
    dims = make_dims(*args)
    ws = torch.empty(fwd_workspace_size(dims), dtype=torch.uint8, device="cuda")
    lib = _lib.load()

    assert _fwd(dims_expire, d, y, hf, ws) == 0, lib.frac_last_error()
    assert lib.frac_workspace_status(_ptr(ws), _stream(None)) == FRAC_ERR_TIMEOUT
    assert b"gave up" in lib.frac_last_error()

    # the context is still usable: a normal call on the same workspace succeeds and is correct
    assert _fwd(dims, d, y, hf, ws) == 0, lib.frac_last_error()
    assert lib.frac_workspace_status(_ptr(ws), _stream(None)) == 0
    torch.cuda.synchronize()
    o = f64_inputs(host)
    yr, hr = oracle.fwd(o["x"], o["dt"], o["alpha"], o["lam"], o["tau"], o["B"], o["C"],
                        o["w_read"], o["w_write"], o["D"])
    assert_close("y", to_host64(y), yr, 1e-2)
    assert_close("h_final", to_host64(hf), hr, 1e-2)


def test_expire_hook_is_refused_off_the_tensor_core_forward():
    s = synth.Shape(1, 64, 2, 32, 1, 16, 4, 0, "f32")
    d = dev_inputs(synth.make_scan_inputs(s, seed=0))
    y = torch.empty_like(d["x"])
    dims = make_dims(s.batch, s.seqlen, s.nheads, s.headdim, s.ngroups, s.dstate, s.nmodes,
                     torch.float32, extra_flags=_lib.FRAC_FLAG_TEST_EXPIRE_WAIT)
    ws = torch.empty(1 << 20, dtype=torch.uint8, device="cuda")
    assert _fwd(dims, d, y, None, ws) == FRAC_ERR_UNSUPPORTED
