"""fp64 numpy model of the chunked evaluation order the GPU kernels use.

Test helper only (never imported by the product path).  It restates, chunk by
chunk, the same recurrence the sequential oracle runs step by step, so that
``tests/test_chunked_model.py`` can check the decomposition on the CPU:

forward, per chunk of Q positions with E_t the in-chunk inclusive cumulative sum of
e_j = Delta_j lambda_j^(1/alpha_j) (so log rho_{t,m} summed over the chunk prefix is
-E_t / tau_m, the stable log-space form of App. F):
    y_t     = sum_m f_{t,m} S_in,m C_t + sum_{k<=t} Gamma_{t,k} (C_t . B_k) x_k + D x_t
    S_out,m = d_m S_in,m + sum_k s_{k,m} x_k B_k^T
with f = w_read exp(-E_t/tau), s = kappa exp(-(E_end - E_k)/tau), d = exp(-E_end/tau) and
Gamma_{t,k} = sum_m w_read_{t,m} kappa_{k,m} exp(-(E_t - E_k)/tau_m) (App. F).

Gamma can also be evaluated through the sub-block factorisation
exp(-(E_t-E_k)/tau) = exp(-(E_t-E_a)/tau) exp(-(E_a-E_b)/tau) exp(-(E_b-E_k)/tau)
(a = first position of t's block, b = last position of k's block, every factor <= 1),
which is what lets the kernels replace most exponentials by multiply-adds.

backward: the chunked adjoint (reverse walk over chunks carrying dS).  The gradient
through the decay, rho_t <dS_t, S_{t-1}>, is evaluated per position from chunk-local
terms that each carry their own decay factor (pairs k < t <= t' inside the chunk, plus
the S_in / dS_out terms), not as a difference of suffix sums: the latter cancels
catastrophically once e_t is large, because the true value is then ~0 while the summands
are O(1) and get multiplied by e_t in dDelta.

The timescale gradient needs the same quantity per mode, weighted by e_t:
dtau_m = tau_m^-2 sum_t e_t (rho_t <dS_t, S_{t-1}>_m - dkappa_{t,m} rho_{t,m} w_write_{t,m}).
Each term of the chunked decomposition covers a span of positions whose e_t sum in closed form
(sum over t in (k, t'] of e_t = E_t' - E_k), so per chunk and mode
  sum_t e_t rho_t <dS_t, S_{t-1}>_m = E_end d_m <dS_out, S_in>_m
      + sum_t E_t w_read_t dw_read^inter_t + sum_k (E_end - E_k) kappa_k dkappa^inter_k
      + sum_{k<t} (E_t - E_k) w_read_t kappa_k W_{t,k} G_{t,k} H_{t,k}
with the inter parts those that come from S_in and dS_out.  The pair sum is kept with its
(E_t - E_k) weight: rewritten as sum_t E_t w dw_read^intra - sum_k E_k kappa dkappa^intra it
cancels (condition number ~1e4 at the test shapes), so float32 inputs would lose three digits.
"""
from __future__ import annotations

import numpy as np


def mode_params(dt, alpha, lam, tau, w_write):
    """e [B,L,H], rho/kappa [B,L,H,K] in fp64 (no clamp)."""
    e = dt * np.power(lam, 1.0 / alpha)
    z = e[..., None] / tau[None, None]
    rho = np.exp(-z)
    kappa = -np.expm1(-z) * w_write
    return e, rho, kappa


def gamma_direct(E, wr, kap, tau):
    """Gamma[t,k] for one (b,h,chunk): E [Q], wr/kap [Q,K], tau [K]."""
    Q = E.shape[0]
    diff = E[:, None] - E[None, :]                        # E_t - E_k
    mask = np.tril(np.ones((Q, Q), dtype=bool))
    W = np.exp(-np.where(mask, diff, 0.0)[..., None] / tau)  # [Q,Q,K]
    G = np.einsum("tm,km,tkm->tk", wr, kap, W)
    return np.where(mask, G, 0.0), np.where(mask[..., None], W, 0.0)


def gamma_factorised(E, wr, kap, tau, sb):
    """Same Gamma via sub-blocks of size sb (direct exponentials only on diagonal blocks)."""
    Q = E.shape[0]
    G = np.zeros((Q, Q))
    nb = (Q + sb - 1) // sb
    for i in range(nb):
        a0, a1 = i * sb, min(Q, (i + 1) * sb)
        Pm = wr[a0:a1] * np.exp(-(E[a0:a1, None] - E[a0]) / tau)       # rows of block i
        for j in range(i + 1):
            b0, b1 = j * sb, min(Q, (j + 1) * sb)
            if j == i:
                d, _ = gamma_direct(E[a0:a1], wr[a0:a1], kap[a0:a1], tau)
                G[a0:a1, a0:a1] = d
            else:
                Qm = kap[b0:b1] * np.exp(-(E[b1 - 1] - E[b0:b1, None]) / tau)   # cols of block j
                Dm = np.exp(-(E[a0] - E[b1 - 1]) / tau)                          # block-to-block
                G[a0:a1, b0:b1] = (Pm * Dm) @ Qm.T
    return G


def gamma_col_anchor(E, wr, kap, tau, sb):
    """Gamma with one anchor per column block, the form the tensor-core kernels use: below the
    diagonal blocks exp(-(E_t - E_k)/tau) = exp(-(E_t - E_a)/tau) exp(-(E_a - E_k)/tau) with
    E_a = E at the last position of k's block (both factors <= 1), so
    Gamma[t, k] = sum_m U_J[t, m] V[k, m]; diagonal blocks are summed directly."""
    Q = E.shape[0]
    G = np.zeros((Q, Q))
    for j0 in range(0, Q, sb):
        j1 = min(Q, j0 + sb)
        G[j0:j1, j0:j1] = gamma_direct(E[j0:j1], wr[j0:j1], kap[j0:j1], tau)[0]
        Ea = E[j1 - 1]
        V = kap[j0:j1] * np.exp(-(Ea - E[j0:j1, None]) / tau)   # [sb, K]
        U = wr[j1:] * np.exp(-(E[j1:, None] - Ea) / tau)         # [rows after the block, K]
        G[j1:, j0:j1] = U @ V.T
    return G


def intra_mode_sums_col_anchor(E, wr, kap, tau, GH, sb):
    """The per-mode pair sums of the intra backward with the same factorisation:
    dwr[t, m] = sum_{k<=t} kappa_{k,m} W_{t,k,m} GH[t,k] and
    dk[k, m]  = sum_{t>=k} w_read_{t,m} W_{t,k,m} GH[t,k];
    below the diagonal blocks dwr = exp(-(E_t - E_a)/tau) sum_k V[k] GH[t,k] and
    dk = exp(-(E_a - E_k)/tau) sum_t U_J[t] GH[t,k]."""
    Q, K = wr.shape
    dwr = np.zeros((Q, K))
    dk = np.zeros((Q, K))
    for j0 in range(0, Q, sb):
        j1 = min(Q, j0 + sb)
        _, W = gamma_direct(E[j0:j1], wr[j0:j1], kap[j0:j1], tau)   # diagonal block, [q,q,K]
        g = GH[j0:j1, j0:j1]
        dwr[j0:j1] += np.einsum("km,tkm,tk->tm", kap[j0:j1], W, g)
        dk[j0:j1] += np.einsum("tm,tkm,tk->km", wr[j0:j1], W, g)
        Ea = E[j1 - 1]
        b = np.exp(-(Ea - E[j0:j1, None]) / tau)                    # [sb, K]
        a = np.exp(-(E[j1:, None] - Ea) / tau)                      # [rows after, K]
        V = kap[j0:j1] * b
        U = wr[j1:] * a
        dwr[j1:] += a * (GH[j1:, j0:j1] @ V)
        dk[j0:j1] += b * (GH[j1:, j0:j1].T @ U)
    return dwr, dk


def fwd(x, dt, alpha, lam, tau, Bm, Cm, wr, ww, D, h0=None, Q=64, sb=None, keep=False):
    Bz, L, H, P = x.shape
    G, N, K = Bm.shape[2], Bm.shape[3], tau.shape[1]
    hpg = H // G
    e, rho, kap = mode_params(dt, alpha, lam, tau, ww)
    y = np.zeros_like(x)
    hf = np.zeros((Bz, H, K, P, N))
    states = {}
    for b in range(Bz):
        for h in range(H):
            g = h // hpg
            S = np.zeros((K, P, N)) if h0 is None else h0[b, h].copy()
            for c0 in range(0, L, Q):
                c1 = min(L, c0 + Q)
                if keep:
                    states[(b, h, c0)] = S.copy()
                E = np.cumsum(e[b, c0:c1, h])
                t_ = tau[h]
                w_r, k_ = wr[b, c0:c1, h], kap[b, c0:c1, h]
                f = w_r * np.exp(-E[:, None] / t_)
                s = k_ * np.exp(-(E[-1] - E[:, None]) / t_)
                dm = np.exp(-E[-1] / t_)
                Gam = gamma_factorised(E, w_r, k_, t_, sb) if sb else gamma_direct(E, w_r, k_, t_)[0]
                Bc, Cc, xc = Bm[b, c0:c1, g], Cm[b, c0:c1, g], x[b, c0:c1, h]
                Z = np.einsum("mpn,tn->tmp", S, Cc)
                yc = np.einsum("tm,tmp->tp", f, Z) + (Gam * (Cc @ Bc.T)) @ xc + D[h] * xc
                y[b, c0:c1, h] = yc
                S = dm[:, None, None] * S + np.einsum("km,kp,kn->mpn", s, xc, Bc)
            hf[b, h] = S
    if keep:
        return y, hf, states
    return y, hf


def bwd(x, dt, alpha, lam, tau, Bm, Cm, wr, ww, D, dy, h0=None, dh_final=None, Q=64):
    Bz, L, H, P = x.shape
    G, N, K = Bm.shape[2], Bm.shape[3], tau.shape[1]
    hpg = H // G
    e, rho, kap = mode_params(dt, alpha, lam, tau, ww)
    _, hf, states = fwd(x, dt, alpha, lam, tau, Bm, Cm, wr, ww, D, h0, Q=Q, keep=True)
    dx = np.zeros_like(x)
    dB = np.zeros_like(Bm)
    dC = np.zeros_like(Cm)
    dwr = np.zeros_like(wr)
    dkap = np.zeros_like(wr)
    dD = np.zeros(H)
    dh0 = np.zeros((Bz, H, K, P, N))
    Rp = np.zeros_like(dt)          # sum_m rho_t <dS_t, S_{t-1}>_m / tau_m
    Te = np.zeros((H, K))           # sum over b, t of e_t rho_t <dS_t, S_{t-1}>_m
    for b in range(Bz):
        for h in range(H):
            g = h // hpg
            t_ = tau[h]
            dS = np.zeros((K, P, N)) if dh_final is None else dh_final[b, h].copy()
            starts = list(range(0, L, Q))
            for c0 in reversed(starts):
                c1 = min(L, c0 + Q)
                S_in = states[(b, h, c0)]
                E = np.cumsum(e[b, c0:c1, h])
                w_r, k_ = wr[b, c0:c1, h], kap[b, c0:c1, h]
                fdec = np.exp(-E[:, None] / t_)            # exp(-E_t/tau)
                f = w_r * fdec
                u = np.exp(-(E[-1] - E[:, None]) / t_)     # exp(-(E_end-E_k)/tau)
                s = k_ * u
                dm = np.exp(-E[-1] / t_)
                Gam, W = gamma_direct(E, w_r, k_, t_)
                Gam_t, _ = gamma_direct(E, w_r, k_ / t_, t_)   # same with kappa / tau
                Bc, Cc = Bm[b, c0:c1, g], Cm[b, c0:c1, g]
                xc, dyc = x[b, c0:c1, h], dy[b, c0:c1, h]
                Gm = Cc @ Bc.T                    # G[t,k] = C_t . B_k
                Hm = dyc @ xc.T                   # H[t,k] = dy_t . x_k
                U = np.einsum("mpn,kn->kmp", dS, Bc)
                Z = np.einsum("mpn,tn->tmp", S_in, Cc)
                dx[b, c0:c1, h] = (np.einsum("km,kmp->kp", s, U) + (Gam * Gm).T @ dyc
                                   + D[h] * dyc)
                GH = Gm * Hm
                xU = np.einsum("kp,kmp->km", xc, U)
                dyZ = np.einsum("tp,tmp->tm", dyc, Z)
                dk_inter = u * xU
                dk_intra = np.einsum("tm,tkm,tk->km", w_r, W, GH)
                dkap[b, c0:c1, h] = dk_inter + dk_intra
                dwr[b, c0:c1, h] = fdec * dyZ + np.einsum("km,tkm,tk->tm", k_, W, GH)
                cdot = np.einsum("mpn,mpn->m", dS, S_in)
                dEp = np.tril(E[:, None] - E[None, :], -1)               # E_t - E_k, k < t
                pairs = np.einsum("tk,tkm,tm,km,tk->m", dEp, W, w_r, k_, GH)
                Te[h] += (E[-1] * dm * cdot + np.sum(E[:, None] * w_r * fdec * dyZ, axis=0)
                          + np.sum((E[-1] - E)[:, None] * k_ * dk_inter, axis=0) + pairs)
                dC[b, c0:c1, g] += (np.einsum("tm,tp,mpn->tn", f, dyc, S_in)
                                    + (Gam * Hm) @ Bc)
                dB[b, c0:c1, g] += (np.einsum("km,kp,mpn->kn", s, xc, dS)
                                    + (Gam * Hm).T @ Cc)
                dD[h] += float(np.sum(dyc * xc))
                # rho_t <dS_t, S_{t-1}> per position, every term written with its own decay:
                a = np.sum(f * dyZ / t_, axis=-1)                 # t' >= t   (dS from y, S_in)
                bb = np.sum(s * xU / t_, axis=-1)                 # k < t     (dS_out, S from x)
                cc = float(np.sum(dm * np.einsum("mpn,mpn->m", dS, S_in) / t_))
                X = Gam_t * GH                                    # pairs k < t <= t'
                n = c1 - c0
                rect = np.array([X[t:, :t].sum() for t in range(n)])
                Rp[b, c0:c1, h] = (np.cumsum(a[::-1])[::-1] + np.concatenate([[0.0], np.cumsum(bb)[:-1]])
                                   + cc + rect)
                dS = dm[:, None, None] * dS + np.einsum("tm,tp,tn->mpn", f, dyc, Cc)
            dh0[b, h] = dS
    de = -Rp + np.sum(dkap * rho * ww / tau[None, None], axis=-1)
    ddt = de * e / dt
    dlam = de * e / (alpha * lam)
    dalpha = -de * e * np.log(lam) / alpha ** 2
    dww = dkap * (-np.expm1(-e[..., None] / tau[None, None]))
    dtau = (Te - np.einsum("blh,blhm->hm", e, dkap * rho * ww)) / tau ** 2
    return dict(dx=dx, ddt=ddt, dalpha=dalpha, dlam=dlam, dB=dB, dC=dC, dw_read=dwr,
                dw_write=dww, dD=dD, dh0=dh0, dtau=dtau)
