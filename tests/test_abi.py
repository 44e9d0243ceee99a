"""The C-ABI library loads, exports every symbol include/frac.h declares, and rejects bad
arguments before anything is enqueued (CPU only: none of these calls reaches the GPU)."""
import ctypes
import os
import re

import pytest

from paper_2609_36314_gb300 import _lib
from paper_2609_36314_gb300.api import make_dims

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "frac.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(frac_[a-z0-9_]+)\s*\(", src)))


def test_header_declares_the_boundary():
    fns = declared_functions()
    for f in ("frac_scan_fwd", "frac_scan_bwd", "frac_decode_step", "frac_scan_fwd_workspace_size",
              "frac_scan_bwd_workspace_size", "frac_status_string", "frac_last_error"):
        assert f in fns
    assert set(fns) == set(_lib.EXPORTS)


def test_library_exports_every_declared_symbol():
    lib = _lib.load()
    for f in declared_functions():
        assert hasattr(lib, f), f


def _fwd_call(lib, dims, ptr=ctypes.c_void_p(0x1000), **over):
    args = dict(x=ptr, dt=ptr, alpha=ptr, lam=ptr, tau=ptr, Bm=ptr, Cm=ptr, wr=ptr, ww=ptr,
                D=ptr, h0=None, y=ptr, hf=None, ws=ptr, wsb=1 << 40, stream=None)
    args.update(over)
    return lib.frac_scan_fwd(ctypes.byref(dims), args["x"], args["dt"], args["alpha"],
                             args["lam"], args["tau"], args["Bm"], args["Cm"], args["wr"],
                             args["ww"], args["D"], args["h0"], args["y"], args["hf"],
                             args["ws"], args["wsb"], args["stream"])


@pytest.mark.parametrize("bad", [
    dict(nheads=6, ngroups=4),
    dict(nmodes=0),
    dict(nmodes=33),
    dict(headdim=0),
    dict(seqlen=-1),
    dict(chunk=-2),
])
def test_invalid_dims_are_rejected(bad):
    import torch
    kw = dict(batch=2, seqlen=64, nheads=4, headdim=32, ngroups=1, dstate=16, nmodes=4,
              dtype=torch.bfloat16)
    kw.update(bad)
    dims = make_dims(**kw)
    lib = _lib.load()
    st = _fwd_call(lib, dims)
    assert st == 1, lib.frac_last_error()
    assert lib.frac_last_error().decode()


def test_unknown_dtype_and_null_pointers():
    import torch
    lib = _lib.load()
    dims = make_dims(2, 64, 4, 32, 1, 16, 4, torch.float32)
    dims.dtype = 7
    assert _fwd_call(lib, dims) == 1
    dims = make_dims(2, 64, 4, 32, 1, 16, 4, torch.float32)
    assert _fwd_call(lib, dims, tau=None) == 1
    assert b"tau" in lib.frac_last_error()
    assert _fwd_call(lib, dims, x=ctypes.c_void_p(0x1002)) == 1
    assert b"aligned" in lib.frac_last_error()
    assert _fwd_call(lib, dims, ws=ctypes.c_void_p(0x1010)) == 1
    assert b"workspace" in lib.frac_last_error()
    assert _fwd_call(lib, dims, wsb=16) == 1
    assert b"too small" in lib.frac_last_error()


def test_unsupported_chunk_is_reported():
    import torch
    lib = _lib.load()
    dims = make_dims(1, 64, 2, 32, 1, 16, 4, torch.float32, chunk=48)
    assert _fwd_call(lib, dims) == 2
    assert lib.frac_status_string(2) == b"unsupported"


def test_workspace_queries():
    import torch
    from paper_2609_36314_gb300 import bwd_workspace_size, fwd_workspace_size
    d = make_dims(2, 100, 4, 32, 1, 16, 4, torch.float32, chunk=32)
    # per-chunk mode states: B * H * ceil(L / Q) * K * P * N float32
    states = 2 * 4 * 4 * 4 * 32 * 16 * 4
    assert fwd_workspace_size(d) >= states
    assert bwd_workspace_size(d) >= 2 * states
    with pytest.raises(_lib.FracError):
        fwd_workspace_size(make_dims(2, 100, 4, 32, 3, 16, 4, torch.float32))


def test_decode_rejects_null_state():
    import torch
    lib = _lib.load()
    dims = make_dims(2, 1, 4, 32, 1, 16, 4, torch.bfloat16)
    p = ctypes.c_void_p(0x1000)
    st = lib.frac_decode_step(ctypes.byref(dims), p, p, p, p, p, p, p, p, p, p, None, p, None)
    assert st == 1
    assert b"state" in lib.frac_last_error()


@pytest.mark.parametrize("bad", ["flags", "order", "modes", "null_cfg"])
def test_param_prep_rejects_bad_arguments(bad):
    """The scan-parameter calls check dims and the config before touching the device."""
    import torch
    from paper_2609_36314_gb300.api import prep_config
    lib = _lib.load()
    dims = make_dims(batch=1, seqlen=8, nheads=2, headdim=1, ngroups=1, dstate=1,
                     nmodes=33 if bad == "modes" else 4, dtype=torch.float32)
    cfg = prep_config(dt_min=2.0 if bad == "order" else 1e-4)
    if bad == "flags":
        cfg.flags = 1 << 10
    p = ctypes.c_void_p(0x1000)
    cfg_ref = None if bad == "null_cfg" else ctypes.byref(cfg)
    st = lib.frac_param_prep_fwd(ctypes.byref(dims), cfg_ref, *([p] * 12), None)
    assert st == 1
    st = lib.frac_param_prep_bwd(ctypes.byref(dims), cfg_ref, *([p] * 19), None)
    assert st == 1


def test_plain_c_caller(tmp_path):
    """tests/abi_check.c includes the header as C99, links libfrac.so and checks the calls that
    need no GPU (status strings, workspace queries, rejection before anything is enqueued)."""
    import shutil
    import subprocess
    from paper_2609_36314_gb300 import build
    if shutil.which("gcc") is None:
        pytest.skip("gcc not found")
    lib = _lib.load()  # builds the library if needed
    del lib
    libdir = os.path.dirname(build.LIB_PATH)
    exe = str(tmp_path / "abi_check")
    subprocess.run(["gcc", "-std=c99", "-Wall", "-Wextra", "-Werror", "-I", os.path.join(ROOT, "include"),
                    os.path.join(ROOT, "tests", "abi_check.c"), "-L", libdir, "-lfrac",
                    "-Wl,-rpath," + libdir, "-o", exe], check=True, capture_output=True, text=True)
    out = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert out.returncode == 0, out.stderr
    assert out.stdout.strip() == "ok"


@pytest.mark.parametrize("case", ["conv_wide", "conv_zero_width", "conv_flag", "conv_null_x",
                                  "conv_alias", "conv_bwd_null_dims", "step_null_state",
                                  "norm_group", "norm_split", "norm_big", "norm_null_weight",
                                  "norm_bwd_null_dz"])
def test_glue_rejects_bad_arguments(case):
    """The conv1d and gated RMSNorm calls check dims, flags, pointers and aliasing before
    touching the device (each case fails validation, so nothing is launched)."""
    lib = _lib.load()
    p, q = ctypes.c_void_p(0x1000), ctypes.c_void_p(0x2000)
    cd = _lib.FracConvDims(2, 16, 64, 4, 1, 0)
    nd = _lib.FracNormDims(4, 64, 64, 1e-5, 1, 0)
    if case == "conv_wide":
        cd.width = 9
        st, want = lib.frac_conv1d_fwd(ctypes.byref(cd), p, p, None, None, q, None, None), 2
    elif case == "conv_zero_width":
        cd.width = 0
        st, want = lib.frac_conv1d_fwd(ctypes.byref(cd), p, p, None, None, q, None, None), 1
    elif case == "conv_flag":
        cd.flags = 2
        st, want = lib.frac_conv1d_fwd(ctypes.byref(cd), p, p, None, None, q, None, None), 1
    elif case == "conv_null_x":
        st, want = lib.frac_conv1d_fwd(ctypes.byref(cd), None, p, None, None, q, None, None), 1
    elif case == "conv_alias":
        st, want = lib.frac_conv1d_fwd(ctypes.byref(cd), p, p, None, q, p, q, None), 1
    elif case == "conv_bwd_null_dims":
        st, want = lib.frac_conv1d_bwd(None, p, p, None, None, p, q, p, None, None, None), 1
    elif case == "step_null_state":
        st, want = lib.frac_conv1d_step(ctypes.byref(cd), p, p, None, None, q, None), 1
    elif case == "norm_group":
        nd.group_size = 12
        st, want = lib.frac_gated_rmsnorm_fwd(ctypes.byref(nd), p, None, p, q, None), 1
    elif case == "norm_split":
        nd.dim, nd.group_size = 40, 16
        st, want = lib.frac_gated_rmsnorm_fwd(ctypes.byref(nd), p, None, p, q, None), 1
    elif case == "norm_big":
        nd.dim, nd.group_size = 40000, 40000
        st, want = lib.frac_gated_rmsnorm_fwd(ctypes.byref(nd), p, None, p, q, None), 2
    elif case == "norm_null_weight":
        st, want = lib.frac_gated_rmsnorm_fwd(ctypes.byref(nd), p, None, None, q, None), 1
    else:  # a gate without its gradient
        st, want = lib.frac_gated_rmsnorm_bwd(ctypes.byref(nd), p, p, p, p, q, None, p, None), 1
    assert st == want
    assert lib.frac_last_error()
