"""Chunked evaluation == sequential recurrence (fp64, CPU).

Pins the decomposition every GPU kernel uses (App. F: chunk-local cumulative
log-decays, the stable intra-chunk coefficient Gamma, cross-chunk state
passing) against the sequential oracle, for many chunk sizes including ragged
last chunks and chunks larger than the sequence.

Tolerance: 1e-10 relative L2.  With alpha small and lambda large, e_t = Delta lambda^(1/alpha)
reaches 1e5-1e7, so in-chunk cumulative sums E carry that magnitude and fp64 differences
E_t - E_k keep only ~1e-16 * E / (E_t - E_k) relative accuracy; the observed gap is ~2e-12.
"""
import numpy as np
import pytest

from oracle import oracle
from paper_2609_36314_gb300 import synth
from tests import chunked_model as cm


def _inputs(Bz=2, L=37, H=4, P=5, G=2, N=3, K=4, seed=3, h0=False, dhf=False, shift=1.0):
    s = synth.Shape(Bz, L, H, P, G, N, K, 0, "f32", dt_shift=shift)
    d = synth.make_scan_inputs(s, seed=seed, with_dy=True, with_h0=h0, with_dh_final=dhf)
    return {k: synth.to_f64(v) for k, v in d.items()}


@pytest.mark.parametrize("Q", [1, 2, 3, 7, 16, 37, 64])
def test_chunked_forward_equals_sequential(Q):
    d = _inputs(h0=True)
    y0, h0f = oracle.fwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"],
                         d["w_read"], d["w_write"], d["D"], d["h0"])
    y1, h1f = cm.fwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"],
                     d["w_read"], d["w_write"], d["D"], d["h0"], Q=Q)
    assert synth.rel_l2(y1, y0) < 1e-10
    assert synth.rel_l2(h1f, h0f) < 1e-10


@pytest.mark.parametrize("Q,sb", [(16, 4), (17, 4), (32, 8), (64, 16), (37, 5)])
def test_subblock_factorisation_of_gamma(Q, sb):
    d = _inputs(L=Q, shift=0.0)
    y0, _ = cm.fwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"],
                   d["w_read"], d["w_write"], d["D"], Q=Q)
    y1, _ = cm.fwd(d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"],
                   d["w_read"], d["w_write"], d["D"], Q=Q, sb=sb)
    assert synth.rel_l2(y1, y0) < 1e-13


def _chunk_terms(Q, seed, shift=0.0):
    rng = np.random.default_rng(seed)
    K = 4
    tau = np.array([1.0, 7.0, 80.0, 2000.0])
    e = np.exp(rng.normal(0.0, 1.5, Q) + shift)          # wide spread of decay rates
    E = np.cumsum(e)
    wr = rng.random((Q, K))
    kap = rng.random((Q, K)) - 0.3
    return E, wr, kap, tau, rng


@pytest.mark.parametrize("Q,sb,shift", [(128, 32, 0.0), (128, 32, 3.0), (100, 32, 0.0), (37, 8, 1.0)])
def test_column_anchored_gamma(Q, sb, shift):
    """The kernels' factorisation (one anchor at the end of each column block) equals Gamma."""
    E, wr, kap, tau, _ = _chunk_terms(Q, seed=Q + sb, shift=shift)
    g0, _ = cm.gamma_direct(E, wr, kap, tau)
    g1 = cm.gamma_col_anchor(E, wr, kap, tau, sb)
    assert np.max(np.abs(g1 - g0)) <= 1e-13 * max(1.0, np.max(np.abs(g0)))


@pytest.mark.parametrize("Q,sb,shift", [(128, 32, 0.0), (128, 32, 2.0), (77, 32, 0.0)])
def test_column_anchored_intra_mode_sums(Q, sb, shift):
    """dw_read and dkappa pair sums of the intra backward through the same factorisation."""
    E, wr, kap, tau, rng = _chunk_terms(Q, seed=3 * Q + sb, shift=shift)
    GH = np.tril(rng.normal(size=(Q, Q)))
    _, W = cm.gamma_direct(E, wr, kap, tau)
    dwr0 = np.einsum("km,tkm,tk->tm", kap, W, GH)
    dk0 = np.einsum("tm,tkm,tk->km", wr, W, GH)
    dwr1, dk1 = cm.intra_mode_sums_col_anchor(E, wr, kap, tau, GH, sb)
    assert synth.rel_l2(dwr1, dwr0) < 1e-12
    assert synth.rel_l2(dk1, dk0) < 1e-12


@pytest.mark.parametrize("Q", [1, 5, 16, 64])
def test_chunked_backward_equals_sequential_adjoint(Q):
    d = _inputs(h0=True, dhf=True)
    args = (d["x"], d["dt"], d["alpha"], d["lam"], d["tau"], d["B"], d["C"], d["w_read"],
            d["w_write"], d["D"])
    g0 = oracle.bwd(*args, d["dy"], h0=d["h0"], dh_final=d["dh_final"], seg=5)
    g1 = cm.bwd(*args, d["dy"], h0=d["h0"], dh_final=d["dh_final"], Q=Q)
    for k in g0:
        assert synth.rel_l2(g1[k], g0[k]) < 1e-10, k
