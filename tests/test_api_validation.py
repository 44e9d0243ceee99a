"""Host-side checks of the Python binding (CPU only): every tensor the kernels read or write,
inputs and caller-supplied outputs alike, must have the shape, dtype and layout the call's
dims imply, so that a mismatched tensor is refused before anything is enqueued instead of
being read or written out of bounds.  Stand-in tensor objects carry only the attributes the
checks look at (no GPU needed)."""
import pytest
import torch

from paper_2609_36314_gb300 import api


class Fake:
    """The attributes of a CUDA tensor that the binding's checks read."""

    def __init__(self, shape, dtype, cuda=True, contiguous=True):
        self.shape = tuple(shape)
        self.dtype = dtype
        self.is_cuda = cuda
        self._contig = contiguous

    def is_contiguous(self):
        return self._contig

    def dim(self):
        return len(self.shape)

    def numel(self):
        n = 1
        for v in self.shape:
            n *= v
        return n


BZ, L, H, P, G, N, K = 2, 40, 4, 64, 1, 128, 8
BF, F32 = torch.bfloat16, torch.float32


def scan_inputs(**over):
    t = dict(x=Fake((BZ, L, H, P), BF), dt=Fake((BZ, L, H), F32), alpha=Fake((BZ, L, H), F32),
             lam=Fake((BZ, L, H), F32), tau=Fake((H, K), F32), B=Fake((BZ, L, G, N), BF),
             C=Fake((BZ, L, G, N), BF), w_read=Fake((BZ, L, H, K), BF),
             w_write=Fake((BZ, L, H, K), BF), D=Fake((H,), F32))
    t.update(over)
    return t


def good_grads():
    return dict(dx=Fake((BZ, L, H, P), BF), ddt=Fake((BZ, L, H), F32),
                dalpha=Fake((BZ, L, H), F32), dlam=Fake((BZ, L, H), F32),
                dB=Fake((BZ, L, G, N), BF), dC=Fake((BZ, L, G, N), BF),
                dw_read=Fake((BZ, L, H, K), BF), dw_write=Fake((BZ, L, H, K), BF),
                dD=Fake((H,), F32), dh0=None)


def call_fwd(t, **kw):
    return api.scan_fwd(t["x"], t["dt"], t["alpha"], t["lam"], t["tau"], t["B"], t["C"],
                        t["w_read"], t["w_write"], t["D"], **kw)


def call_bwd(t, dy, **kw):
    return api.scan_bwd(t["x"], t["dt"], t["alpha"], t["lam"], t["tau"], t["B"], t["C"],
                        t["w_read"], t["w_write"], t["D"], dy, **kw)


@pytest.mark.parametrize("name,bad", [
    ("dt", Fake((BZ, L - 1, H), F32)),
    ("alpha", Fake((BZ, L, H), BF)),
    ("C", Fake((BZ, L, G, N // 2), BF)),
    ("w_write", Fake((BZ, L, H, K - 1), BF)),
    ("D", Fake((H + 1,), F32)),
    ("lam", Fake((BZ, L, H), F32, cuda=False)),
    ("B", Fake((BZ, L, G, N), BF, contiguous=False)),
])
def test_scan_inputs_are_checked(name, bad):
    t = scan_inputs(**{name: bad})
    with pytest.raises(ValueError, match=name):
        call_fwd(t)
    with pytest.raises(ValueError, match=name):
        call_bwd(t, Fake((BZ, L, H, P), BF))
    with pytest.raises(ValueError, match=name):
        api.scan_fwd_static(t["x"], t["dt"], t["alpha"], t["lam"], t["tau"], t["B"], t["C"],
                            t["w_read"], t["w_write"], t["D"])


def test_forward_outputs_are_checked():
    t = scan_inputs()
    with pytest.raises(ValueError, match="y"):
        call_fwd(t, y=Fake((BZ, L, H, P - 1), BF))
    with pytest.raises(ValueError, match="y"):
        call_fwd(t, y=Fake((BZ, L, H, P), F32))
    with pytest.raises(ValueError, match="h_final"):
        call_fwd(t, y=Fake((BZ, L, H, P), BF), h_final=Fake((BZ, H, K, P, N // 2), F32))
    with pytest.raises(ValueError, match="h0"):
        call_fwd(t, h0=Fake((BZ, H, K, P, N), BF))


@pytest.mark.parametrize("name,bad", [
    ("dx", Fake((BZ, L, H, P + 1), BF)),
    ("ddt", Fake((BZ, L, H), BF)),
    ("dB", Fake((BZ, L, G + 1, N), BF)),
    ("dw_read", Fake((BZ, L, H, K // 2), BF)),
    ("dD", Fake((H, 1), F32)),
    ("dh0", Fake((BZ, H, K, P, N - 1), F32)),
    ("dtau", Fake((H, K + 1), F32)),
])
def test_backward_outputs_are_checked(name, bad):
    g = good_grads()
    g[name] = bad
    with pytest.raises(ValueError, match=name):
        call_bwd(scan_inputs(), Fake((BZ, L, H, P), BF), out=g)


def test_backward_needs_every_gradient_it_writes():
    g = good_grads()
    del g["dC"]
    with pytest.raises(ValueError, match="dC"):
        call_bwd(scan_inputs(), Fake((BZ, L, H, P), BF), out=g)


def test_backward_upstream_gradient_is_checked():
    with pytest.raises(ValueError, match="dy"):
        call_bwd(scan_inputs(), Fake((BZ, L, H, P - 2), BF))


def test_decode_output_is_checked():
    x_t = Fake((BZ, H, P), BF)
    args = (x_t, Fake((BZ, H), F32), Fake((BZ, H), F32), Fake((BZ, H), F32), Fake((H, K), F32),
            Fake((BZ, G, N), BF), Fake((BZ, G, N), BF), Fake((BZ, H, K), BF), Fake((BZ, H, K), BF),
            Fake((H,), F32), Fake((BZ, H, K, P, N), F32))
    with pytest.raises(ValueError, match="y_t"):
        api.decode_step(*args, y_t=Fake((BZ, H, P + 1), BF))


def test_glue_arguments_are_checked():
    Bz, Lc, C, W = 2, 30, 72, 4
    x = Fake((Bz, Lc, C), BF)
    w = Fake((C, W), F32)
    with pytest.raises(ValueError, match="w"):
        api.conv1d_fwd(x, Fake((C, W), BF))
    with pytest.raises(ValueError, match="bias"):
        api.conv1d_fwd(x, w, Fake((C + 1,), F32))
    with pytest.raises(ValueError, match="state"):
        api.conv1d_bwd(x, w, Fake((Bz, Lc, C), BF), state=Fake((Bz, C, W), BF))
    with pytest.raises(ValueError, match="du"):
        api.conv1d_bwd(x, w, Fake((Bz, Lc - 1, C), BF))
    with pytest.raises(ValueError, match="u_t"):
        api.conv1d_step(Fake((Bz, C), BF), w, Fake((Bz, C, W - 1), BF), u_t=Fake((Bz, C + 8), BF))
    with pytest.raises(ValueError, match="w"):
        api.conv1d_step(Fake((Bz, C), BF), Fake((C - 8, W), F32), Fake((Bz, C, W - 1), BF))
    y = Fake((16, 256), BF)
    with pytest.raises(ValueError, match="weight"):
        api.gated_rmsnorm_bwd(y, None, Fake((255,), F32), Fake((16, 256), BF))
    with pytest.raises(ValueError, match="z"):
        api.gated_rmsnorm_bwd(y, Fake((16, 256), F32), Fake((256,), F32), Fake((16, 256), BF))


def test_prep_arguments_are_checked():
    Bz, Lp, Hp, Kp = 2, 9, 4, 8
    dt_raw = Fake((Bz, Lp, Hp), F32)
    g = Fake((Bz, Lp, Hp, Kp), BF)
    tau = Fake((Hp, Kp), F32)
    ok = dict(dt_raw=dt_raw, alpha_raw=Fake((Bz, Lp, Hp), F32), lam_raw=Fake((Bz, Lp, Hp), F32),
              g_read=g, g_write=Fake((Bz, Lp, Hp, Kp), BF), tau=tau)
    up = (Fake((Bz, Lp, Hp), F32), Fake((Bz, Lp, Hp), F32), Fake((Bz, Lp, Hp), F32),
          Fake((Bz, Lp, Hp, Kp), BF), Fake((Bz, Lp, Hp, Kp), BF))
    for name, bad in (("lam_raw", Fake((Bz, Lp + 1, Hp), F32)), ("g_write", Fake((Bz, Lp, Hp, Kp), F32)),
                      ("g_read", Fake((Bz, Lp - 1, Hp, Kp), BF)), ("alpha_raw", Fake((Bz, Lp, Hp), BF))):
        a = dict(ok, **{name: bad})
        args = (a["dt_raw"], a["alpha_raw"], a["lam_raw"], a["g_read"], a["g_write"], a["tau"])
        with pytest.raises(ValueError, match=name):
            api.param_prep_fwd(*args)
        with pytest.raises(ValueError, match=name):
            api.param_prep_bwd(*args, *up)
    args = (ok["dt_raw"], ok["alpha_raw"], ok["lam_raw"], ok["g_read"], ok["g_write"], ok["tau"])
    with pytest.raises(ValueError, match="dt_bias"):
        api.param_prep_bwd(*args, *up, dt_bias=Fake((Hp + 1,), F32))
    with pytest.raises(ValueError, match="w_read"):
        api.param_prep_fwd(*args, out=dict(dt=Fake((Bz, Lp, Hp), F32), alpha=Fake((Bz, Lp, Hp), F32),
                                            lam=Fake((Bz, Lp, Hp), F32), w_read=Fake((Bz, Lp, Hp, 4), BF),
                                            w_write=Fake((Bz, Lp, Hp, Kp), BF)))
