"""The allocation-free forward scan (frac_scan_fwd_static).

It is meant for callers that cannot hand the library scratch memory -- for instance code
living inside a host application that owns all device memory and gives its plug-ins no
allocator.  Instead of a caller workspace it uses one fixed device array owned by the
library.  These checks call it through the C ABI and compare it with frac_scan_fwd (which is
given a normal workspace) on two calls in a row, the second with different inputs, so that
leftovers of the first call in the shared array would show up.  The file is named so that
pytest collects it last.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2609_36314_gb300 import _lib, scan_fwd, synth
from paper_2609_36314_gb300.api import _ptr, _stream, fwd_workspace_size, make_dims
from tests.gpu_util import assert_close, dev_inputs, to_host64, tol

pytestmark = pytest.mark.gpu


def _static_call(dims, d, y, hf):
    lib = _lib.load()
    return lib.frac_scan_fwd_static(
        ctypes.byref(dims), _ptr(d["x"]), _ptr(d["dt"]), _ptr(d["alpha"]), _ptr(d["lam"]),
        _ptr(d["tau"]), _ptr(d["B"]), _ptr(d["C"]), _ptr(d["w_read"]), _ptr(d["w_write"]),
        _ptr(d["D"]), _ptr(d.get("h0")), _ptr(y), _ptr(hf), _stream(None))


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_static_scratch_forward_matches_workspace_forward(dtype):
    s = synth.Shape(2, 300, 8, 64, 1, 64, 8, 0, dtype)
    dims = make_dims(s.batch, s.seqlen, s.nheads, s.headdim, s.ngroups, s.dstate, s.nmodes,
                     torch.bfloat16 if dtype == "bf16" else torch.float32)
    assert fwd_workspace_size(dims) <= _lib.FRAC_SCAN_FWD_STATIC_SCRATCH_BYTES
    for seed in (0, 1):  # two calls in a row through the shared array
        d = dev_inputs(synth.make_scan_inputs(s, seed=seed, with_h0=(seed == 1)))
        y = torch.empty_like(d["x"])
        hf = torch.empty((s.batch, s.nheads, s.nmodes, s.headdim, s.dstate), dtype=torch.float32,
                         device="cuda")
        st = _static_call(dims, d, y, hf)
        assert st == 0, _lib.load().frac_last_error()
        assert _lib.load().frac_scan_fwd_static_status(_stream(None)) == 0
        y_ref, hf_ref = scan_fwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"],
                                 d["C"], d["w_read"], d["w_write"], d["D"], d.get("h0"))
        torch.cuda.synchronize()
        assert_close(f"y (call {seed})", to_host64(y), to_host64(y_ref), tol(dtype))
        assert_close(f"h_final (call {seed})", to_host64(hf), to_host64(hf_ref), tol(dtype))


def test_static_scratch_smaller_problem_after_a_larger_one():
    """A larger problem first, then a smaller one with another length and mode count on the
    same (tensor-core) path: the second result must not depend on what the first left in the
    shared array, so it is compared with frac_scan_fwd given a fresh workspace."""
    big = synth.Shape(2, 517, 8, 64, 1, 128, 8, 0, "bf16")
    small = synth.Shape(1, 131, 4, 64, 1, 128, 4, 0, "bf16")
    for s, seed in ((big, 3), (small, 4)):
        dims = make_dims(s.batch, s.seqlen, s.nheads, s.headdim, s.ngroups, s.dstate, s.nmodes,
                         torch.bfloat16)
        assert fwd_workspace_size(dims) <= _lib.FRAC_SCAN_FWD_STATIC_SCRATCH_BYTES
        d = dev_inputs(synth.make_scan_inputs(s, seed=seed))
        y = torch.empty_like(d["x"])
        hf = torch.empty((s.batch, s.nheads, s.nmodes, s.headdim, s.dstate), dtype=torch.float32,
                         device="cuda")
        assert _static_call(dims, d, y, hf) == 0, _lib.load().frac_last_error()
        assert _lib.load().frac_scan_fwd_static_status(_stream(None)) == 0
        ws = torch.zeros(fwd_workspace_size(dims), dtype=torch.uint8, device="cuda")
        y_ref, hf_ref = scan_fwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"],
                                 d["C"], d["w_read"], d["w_write"], d["D"], workspace=ws)
        torch.cuda.synchronize()
        assert_close(f"y (L={s.seqlen})", to_host64(y), to_host64(y_ref), tol("bf16"))
        assert_close(f"h_final (L={s.seqlen})", to_host64(hf), to_host64(hf_ref), tol("bf16"))


def test_static_scratch_status_reports_an_expired_wait():
    """A bounded device wait that runs out inside the allocation-free forward is visible to
    the caller through frac_scan_fwd_static_status (the test hook makes the forward state
    pass's waits run out), and the next call resets the word."""
    s = synth.Shape(1, 200, 2, 64, 1, 64, 8, 0, "bf16")
    args = (s.batch, s.seqlen, s.nheads, s.headdim, s.ngroups, s.dstate, s.nmodes, torch.bfloat16)
    d = dev_inputs(synth.make_scan_inputs(s, seed=6))
    y = torch.empty_like(d["x"])
    lib = _lib.load()
    dims = make_dims(*args, extra_flags=_lib.FRAC_FLAG_TEST_EXPIRE_WAIT)
    assert _static_call(dims, d, y, None) == 0, lib.frac_last_error()
    assert lib.frac_scan_fwd_static_status(_stream(None)) == 4  # FRAC_ERR_TIMEOUT
    assert _static_call(make_dims(*args), d, y, None) == 0, lib.frac_last_error()
    assert lib.frac_scan_fwd_static_status(_stream(None)) == 0


def test_static_scratch_rejects_problems_that_do_not_fit():
    s = synth.Shape(4, 4096, 16, 64, 1, 64, 8, 0, "bf16")
    dims = make_dims(s.batch, s.seqlen, s.nheads, s.headdim, s.ngroups, s.dstate, s.nmodes,
                     torch.bfloat16)
    assert fwd_workspace_size(dims) > _lib.FRAC_SCAN_FWD_STATIC_SCRATCH_BYTES
    d = dev_inputs(synth.make_scan_inputs(s.replace(seqlen=1), seed=0))  # pointers only
    y = torch.empty(1, device="cuda")
    st = _static_call(dims, d, y, None)
    assert st == 2
    assert b"scratch" in _lib.load().frac_last_error()
