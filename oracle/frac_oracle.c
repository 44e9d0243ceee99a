/*
 * frac_oracle.c -- plain fp64 CPU oracle for the Frac selective fractional
 * state-space scan (arXiv 2609.36314).
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference leg of bench.py may load this library.  It shares
 * no code, header or constant with the CUDA path.
 *
 * What it computes (the paper's layer, lifted to an N-dimensional outer
 * product state exactly like a Mamba2 SSD head; with N=1 and B=C=1 it is
 * Algorithm 1 of Appendix D verbatim):
 *
 *   effective timescale   tau~_{t,m} = tau_m / lambda_t^(1/alpha_t)      (Eq. tau-eff, Sec. 3.2)
 *   retention             rho_{t,m}  = exp(-Delta_t / tau~_{t,m})         (Eq. rho-beta-def-frac)
 *   injection             beta_{t,m} = 1 - rho_{t,m}                      (Algorithm 1 step 3 and the
 *                                                                           remark after it: all of the
 *                                                                           paper's runs use 1 - rho)
 *   write coefficient     kappa_{t,m} = beta_{t,m} * b_{t,m}              (Eq. frac-selective-update)
 *   update                S_{t,m} = rho_{t,m} S_{t-1,m} + kappa_{t,m} x_t B_t^T   (P x N per mode)
 *   readout               y_t = sum_m c_{t,m} S_{t,m} C_t + D x_t          (Eq. frac-readout, skip D u_t of Sec. 3.3)
 *
 * b (write weights, "w_write") and c (read weights, "w_read") are the
 * already-normalised softmax mode weights of Eq. read-softmax; they are inputs.
 * beta is evaluated as -expm1(-Delta/tau~), which is 1 - rho written without
 * cancellation.
 *
 * The backward pass is the adjoint of the same sequential recurrence, run
 * backwards in t.  States needed by the adjoint are recomputed from
 * checkpoints taken every `seg` steps of the forward pass (plain
 * recomputation; no reordering of any arithmetic).
 *
 * Layouts (row-major, contiguous):
 *   x, y, dy, dx   [B, L, H, P]      dt, alpha, lam (+ grads) [B, L, H]
 *   Bm, Cm (+grad) [B, L, G, N]      w_read, w_write (+grads) [B, L, H, K]
 *   tau            [H, K]            D, dD  [H]
 *   h0, h_final, dh_final, dh0        [B, H, K, P, N]
 * Head h reads group g = h / (H / G).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef struct {
    int64_t B, L, H, P, G, N, K;
} dims_t;

/* Mode parameters of one (t, h): rho, kappa and z = Delta * lambda^(1/alpha) / tau_m. */
static void mode_params(double dt, double alpha, double lam, const double *tau_h,
                        const double *ww, int64_t K, double *rho, double *kappa, double *z) {
    const double lam_pow = pow(lam, 1.0 / alpha);         /* lambda^(1/alpha) */
    for (int64_t m = 0; m < K; ++m) {
        const double tau_eff = tau_h[m] / lam_pow;          /* tau~ = tau / lambda^(1/alpha) */
        const double zm = dt / tau_eff;                     /* Delta / tau~ (may be +inf) */
        z[m] = zm;
        rho[m] = exp(-zm);
        kappa[m] = -expm1(-zm) * ww[m];                     /* (1 - rho) * b */
    }
}

/* One recurrence step for one (b, h): S <- rho S + kappa x B^T, then y = sum_m c_m S_m C + D x. */
static void step_fwd(const dims_t *d, double *S, const double *rho, const double *kappa,
                     const double *x, const double *Bv, const double *Cv, const double *wr,
                     double Dh, double *y) {
    const int64_t P = d->P, N = d->N, K = d->K;
    for (int64_t m = 0; m < K; ++m) {
        double *Sm = S + m * P * N;
        for (int64_t p = 0; p < P; ++p) {
            const double kx = kappa[m] * x[p];
            for (int64_t n = 0; n < N; ++n)
                Sm[p * N + n] = rho[m] * Sm[p * N + n] + kx * Bv[n];
        }
    }
    for (int64_t p = 0; p < P; ++p) {
        double acc = 0.0;
        for (int64_t m = 0; m < K; ++m) {
            const double *Sm = S + m * P * N;
            double dot = 0.0;
            for (int64_t n = 0; n < N; ++n) dot += Sm[p * N + n] * Cv[n];
            acc += wr[m] * dot;
        }
        y[p] = acc + Dh * x[p];
    }
}

static int valid(const dims_t *d) {
    if (d->B < 0 || d->L < 0 || d->H <= 0 || d->P <= 0 || d->G <= 0 || d->N <= 0 || d->K <= 0) return 0;
    if (d->H % d->G) return 0;
    return 1;
}

#define IDX_BLH(b, t, h) (((b) * d.L + (t)) * d.H + (h))

int frac_oracle_fwd(int64_t Bsz, int64_t L, int64_t H, int64_t P, int64_t G, int64_t N, int64_t K,
                    const double *x, const double *dt, const double *alpha, const double *lam,
                    const double *tau, const double *Bm, const double *Cm, const double *wr,
                    const double *ww, const double *D, const double *h0, double *y,
                    double *h_final, int nthreads) {
    dims_t d = {Bsz, L, H, P, G, N, K};
    if (!valid(&d)) return 2;
    const int64_t SZ = K * P * N, hpg = H / G;
    int err = 0;
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads > 0 ? nthreads : 1)
    for (int64_t bh = 0; bh < Bsz * H; ++bh) {
        const int64_t b = bh / H, h = bh % H, g = h / hpg;
        double *S = (double *)malloc(sizeof(double) * SZ);
        double *rho = (double *)malloc(sizeof(double) * K * 3);
        if (!S || !rho) { err = 1; free(S); free(rho); continue; }
        double *kappa = rho + K, *z = rho + 2 * K;
        if (h0) memcpy(S, h0 + bh * SZ, sizeof(double) * SZ);
        else memset(S, 0, sizeof(double) * SZ);
        for (int64_t t = 0; t < L; ++t) {
            const int64_t i = IDX_BLH(b, t, h);
            mode_params(dt[i], alpha[i], lam[i], tau + h * K, ww + i * K, K, rho, kappa, z);
            step_fwd(&d, S, rho, kappa, x + i * P, Bm + ((b * L + t) * G + g) * N,
                     Cm + ((b * L + t) * G + g) * N, wr + i * K, D[h], y + i * P);
        }
        if (h_final) memcpy(h_final + bh * SZ, S, sizeof(double) * SZ);
        free(S);
        free(rho);
    }
    return err;
}

/* Decode: exactly one step of the recurrence on a cached state (Algorithm 1, one token). */
int frac_oracle_decode(int64_t Bsz, int64_t H, int64_t P, int64_t G, int64_t N, int64_t K,
                       const double *x_t, const double *dt, const double *alpha, const double *lam,
                       const double *tau, const double *B_t, const double *C_t, const double *wr,
                       const double *ww, const double *D, double *state, double *y_t) {
    dims_t d = {Bsz, 1, H, P, G, N, K};
    if (!valid(&d)) return 2;
    const int64_t SZ = K * P * N, hpg = H / G;
    double *rho = (double *)malloc(sizeof(double) * K * 3);
    if (!rho) return 1;
    double *kappa = rho + K, *z = rho + 2 * K;
    for (int64_t b = 0; b < Bsz; ++b)
        for (int64_t h = 0; h < H; ++h) {
            const int64_t i = b * H + h, g = h / hpg;
            mode_params(dt[i], alpha[i], lam[i], tau + h * K, ww + i * K, K, rho, kappa, z);
            step_fwd(&d, state + i * SZ, rho, kappa, x_t + i * P, B_t + (b * G + g) * N,
                     C_t + (b * G + g) * N, wr + i * K, D[h], y_t + i * P);
        }
    free(rho);
    return 0;
}

/*
 * Backward: adjoint of the forward recurrence.  With dS the adjoint of S_t
 * (initialised from dh_final), going from t = L-1 down to 0:
 *   dS_m      += c_{t,m} dy_t C_t^T
 *   dc_{t,m}   = dy_t^T S_{t,m} C_t
 *   dC_t      += sum_m c_{t,m} S_{t,m}^T dy_t
 *   dkappa_m   = x_t^T dS_m B_t
 *   dx_t       = sum_m kappa_m dS_m B_t + D dy_t
 *   dB_t      += sum_m kappa_m dS_m^T x_t
 *   drho_m     = <dS_m, S_{t-1,m}>
 *   dS_m      *= rho_m
 *   dD        += <dy_t, x_t>
 * and the chain rule through kappa = -expm1(-z) b, rho = exp(-z),
 * z = Delta lambda^(1/alpha) / tau_m:
 *   db_{t,m}   = dkappa_m (1 - rho_m)
 *   dz_m       = -(drho_m - dkappa_m b_m) rho_m
 *   dDelta     = sum_m dz_m z_m / Delta
 *   dlambda    = sum_m dz_m z_m / (alpha lambda)
 *   dalpha     = sum_m dz_m z_m (-ln lambda / alpha^2)
 *   dtau_m     = sum over b, t of dz_m z_m (-1 / tau_m)   (z = Delta lambda^(1/alpha) / tau: the
 *                timescale gradient of the App. G "learned timescales" variant)
 * (rho_m z_m is taken as its limit 0 when z_m = +inf.)  dh0 = final dS.  dtau may be NULL.
 */
int frac_oracle_bwd(int64_t Bsz, int64_t L, int64_t H, int64_t P, int64_t G, int64_t N, int64_t K,
                    const double *x, const double *dt, const double *alpha, const double *lam,
                    const double *tau, const double *Bm, const double *Cm, const double *wr,
                    const double *ww, const double *D, const double *h0, const double *dy,
                    const double *dh_final, double *dx, double *ddt, double *dalpha, double *dlam,
                    double *dB, double *dC, double *dwr, double *dww, double *dD, double *dh0,
                    double *dtau, int64_t seg, int nthreads) {
    dims_t d = {Bsz, L, H, P, G, N, K};
    if (!valid(&d)) return 2;
    if (seg <= 0) seg = 32;
    const int64_t SZ = K * P * N, hpg = H / G;
    const int64_t nseg = (L + seg - 1) / seg;
    /* per-(b,h) partial sums of dB, dC, dD; reduced over the heads of a group afterwards */
    double *pB = (double *)calloc((size_t)(Bsz * H * L * N > 0 ? Bsz * H * L * N : 1), sizeof(double));
    double *pC = (double *)calloc((size_t)(Bsz * H * L * N > 0 ? Bsz * H * L * N : 1), sizeof(double));
    double *pD = (double *)calloc((size_t)(Bsz * H > 0 ? Bsz * H : 1), sizeof(double));
    double *pT = (double *)calloc((size_t)(Bsz * H * K > 0 ? Bsz * H * K : 1), sizeof(double));
    if (!pB || !pC || !pD || !pT) { free(pB); free(pC); free(pD); free(pT); return 1; }
    int err = 0;
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads > 0 ? nthreads : 1)
    for (int64_t bh = 0; bh < Bsz * H; ++bh) {
        const int64_t b = bh / H, h = bh % H, g = h / hpg;
        /* checkpoints: state before step s*seg, s = 0..nseg-1 */
        double *ck = (double *)malloc(sizeof(double) * SZ * (nseg > 0 ? nseg : 1));
        double *St = (double *)malloc(sizeof(double) * SZ * (seg + 1)); /* S_{t0-1} .. S_{t0+seg-1} */
        double *dS = (double *)malloc(sizeof(double) * SZ);
        double *tmp = (double *)malloc(sizeof(double) * (K * 6 + P));
        if (!ck || !St || !dS || !tmp) { err = 1; free(ck); free(St); free(dS); free(tmp); continue; }
        double *rho = tmp, *kappa = tmp + K, *z = tmp + 2 * K, *dkap = tmp + 3 * K,
               *drho = tmp + 4 * K, *ydummy = tmp + 6 * K;
        /* forward pass for checkpoints */
        double *S = St;
        if (h0) memcpy(S, h0 + bh * SZ, sizeof(double) * SZ);
        else memset(S, 0, sizeof(double) * SZ);
        for (int64_t t = 0; t < L; ++t) {
            if (t % seg == 0) memcpy(ck + (t / seg) * SZ, S, sizeof(double) * SZ);
            const int64_t i = IDX_BLH(b, t, h);
            mode_params(dt[i], alpha[i], lam[i], tau + h * K, ww + i * K, K, rho, kappa, z);
            step_fwd(&d, S, rho, kappa, x + i * P, Bm + ((b * L + t) * G + g) * N,
                     Cm + ((b * L + t) * G + g) * N, wr + i * K, D[h], ydummy);
        }
        if (dh_final) memcpy(dS, dh_final + bh * SZ, sizeof(double) * SZ);
        else memset(dS, 0, sizeof(double) * SZ);
        double dDacc = 0.0;
        for (int64_t s = nseg - 1; s >= 0; --s) {
            const int64_t t0 = s * seg, t1 = (t0 + seg < L) ? t0 + seg : L;
            /* recompute S_{t0-1} .. S_{t1-1}: St[j] = S_{t0-1+j} */
            memcpy(St, ck + s * SZ, sizeof(double) * SZ);
            for (int64_t t = t0; t < t1; ++t) {
                const int64_t i = IDX_BLH(b, t, h), j = t - t0;
                memcpy(St + (j + 1) * SZ, St + j * SZ, sizeof(double) * SZ);
                mode_params(dt[i], alpha[i], lam[i], tau + h * K, ww + i * K, K, rho, kappa, z);
                step_fwd(&d, St + (j + 1) * SZ, rho, kappa, x + i * P,
                         Bm + ((b * L + t) * G + g) * N, Cm + ((b * L + t) * G + g) * N,
                         wr + i * K, D[h], ydummy);
            }
            for (int64_t t = t1 - 1; t >= t0; --t) {
                const int64_t i = IDX_BLH(b, t, h), j = t - t0;
                const double *Scur = St + (j + 1) * SZ, *Sprev = St + j * SZ;
                const double *xt = x + i * P, *dyt = dy + i * P;
                const double *Bt = Bm + ((b * L + t) * G + g) * N, *Ct = Cm + ((b * L + t) * G + g) * N;
                const double *wrt = wr + i * K, *wwt = ww + i * K;
                double *pBt = pB + (bh * L + t) * N, *pCt = pC + (bh * L + t) * N;
                mode_params(dt[i], alpha[i], lam[i], tau + h * K, wwt, K, rho, kappa, z);
                for (int64_t m = 0; m < K; ++m) {
                    const double *Sm = Scur + m * SZ / K;
                    double *dSm = dS + m * SZ / K;
                    double dw = 0.0;
                    for (int64_t p = 0; p < P; ++p) {
                        double dot = 0.0;
                        for (int64_t n = 0; n < N; ++n) {
                            dSm[p * N + n] += wrt[m] * dyt[p] * Ct[n];
                            dot += Sm[p * N + n] * Ct[n];
                            pCt[n] += wrt[m] * Sm[p * N + n] * dyt[p];
                        }
                        dw += dyt[p] * dot;
                    }
                    dwr[i * K + m] = dw;
                }
                for (int64_t p = 0; p < P; ++p) dx[i * P + p] = D[h] * dyt[p];
                for (int64_t m = 0; m < K; ++m) {
                    const double *Spm = Sprev + m * SZ / K;
                    double *dSm = dS + m * SZ / K;
                    double dk = 0.0, dr = 0.0;
                    for (int64_t p = 0; p < P; ++p) {
                        double dsb = 0.0;
                        for (int64_t n = 0; n < N; ++n) {
                            dsb += dSm[p * N + n] * Bt[n];
                            pBt[n] += kappa[m] * dSm[p * N + n] * xt[p];
                            dr += dSm[p * N + n] * Spm[p * N + n];
                        }
                        dk += xt[p] * dsb;
                        dx[i * P + p] += kappa[m] * dsb;
                    }
                    dkap[m] = dk;
                    drho[m] = dr;
                    for (int64_t q = 0; q < P * N; ++q) dSm[q] *= rho[m];
                }
                double dd = 0.0;
                for (int64_t p = 0; p < P; ++p) dd += dyt[p] * xt[p];
                dDacc += dd;
                const double lnl = log(lam[i]), al = alpha[i];
                double gdt = 0.0, gal = 0.0, glm = 0.0;
                for (int64_t m = 0; m < K; ++m) {
                    dww[i * K + m] = dkap[m] * (-expm1(-z[m]));
                    const double rz = isinf(z[m]) ? 0.0 : rho[m] * z[m];
                    const double dzr = -(drho[m] - dkap[m] * wwt[m]); /* d loss / d z, times 1/rho */
                    const double dz_z = dzr * rz;                       /* (d loss / d z) * z */
                    gdt += dz_z / dt[i];
                    glm += dz_z / (al * lam[i]);
                    gal += dz_z * (-lnl / (al * al));
                    pT[bh * K + m] += dz_z * (-1.0 / tau[h * K + m]);
                }
                ddt[i] = gdt;
                dlam[i] = glm;
                dalpha[i] = gal;
            }
        }
        if (dh0) memcpy(dh0 + bh * SZ, dS, sizeof(double) * SZ);
        pD[bh] = dDacc;
        free(ck); free(St); free(dS); free(tmp);
    }
    if (!err) {
        for (int64_t b = 0; b < Bsz; ++b)
            for (int64_t t = 0; t < L; ++t)
                for (int64_t g = 0; g < G; ++g) {
                    double *oB = dB + ((b * L + t) * G + g) * N, *oC = dC + ((b * L + t) * G + g) * N;
                    for (int64_t n = 0; n < N; ++n) { oB[n] = 0.0; oC[n] = 0.0; }
                    for (int64_t h = g * hpg; h < (g + 1) * hpg; ++h) {
                        const double *sB = pB + ((b * H + h) * L + t) * N, *sC = pC + ((b * H + h) * L + t) * N;
                        for (int64_t n = 0; n < N; ++n) { oB[n] += sB[n]; oC[n] += sC[n]; }
                    }
                }
        for (int64_t h = 0; h < H; ++h) {
            double s = 0.0;
            for (int64_t b = 0; b < Bsz; ++b) s += pD[b * H + h];
            dD[h] = s;
        }
        if (dtau)
            for (int64_t h = 0; h < H; ++h)
                for (int64_t m = 0; m < K; ++m) {
                    double s = 0.0;
                    for (int64_t b = 0; b < Bsz; ++b) s += pT[(b * H + h) * K + m];
                    dtau[h * K + m] = s;
                }
    }
    free(pB); free(pC); free(pD); free(pT);
    return err;
}

int frac_oracle_max_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
