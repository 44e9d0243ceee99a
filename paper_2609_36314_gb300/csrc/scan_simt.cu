// CUDA-core (SIMT) chunked Frac scan: forward and backward, float32 arithmetic.
//
// The chunked evaluation order (App. F of the paper; the Remark after Eq. read-softmax):
// per chunk of Q positions, E_t = sum of e_j = Delta_j lambda_j^(1/alpha_j) from the chunk
// start through t (kept in double so that differences E_t - E_k are exact to float
// precision even when e_j is huge), so that the log of the product of retentions from k+1
// to t in mode m is -(E_t - E_k) / tau_m.
//
//   state pass (chunk-serial per (b, h, p-slice)):  S_out,m = d_m S_in,m + sum_k s_{k,m} x_k B_k^T
//        d_m = exp(-E_end / tau_m),  s_{k,m} = kappa_{k,m} exp(-(E_end - E_k) / tau_m)
//        emits S_in of every chunk into the workspace; the same kernel run over the chunks in
//        reverse with (dy, C, f_{t,m} = w_read_{t,m} exp(-E_t / tau_m)) carries dS backwards.
//   chunk output (chunk-parallel per (b, h, c)):
//        y_t = sum_m f_{t,m} S_in,m C_t + sum_{k<=t} Gamma_{t,k} (C_t . B_k) x_k + D x_t
//        Gamma_{t,k} = sum_m w_read_{t,m} kappa_{k,m} exp(-(E_t - E_k) / tau_m)   (App. F)
//   chunk backward (chunk-parallel per (b, h, c)): every gradient from x, dy, B, C, the mode
//        weights, S_in and dS_out of the chunk (see the comments in simt_chunk_bwd).
//
// Threads own register tiles of the small per-chunk contractions; shared-memory rows are
// padded by one float so that both row and column walks are free of bank conflicts.
#include <algorithm>
#include <type_traits>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace frac {
namespace {

constexpr int kQMax = 64;
constexpr int kThreads = 256;

template <typename TS> __device__ __forceinline__ TS cvt_state(float v);
template <> __device__ __forceinline__ float cvt_state<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 cvt_state<__nv_bfloat16>(float v) {
    return __float2bfloat16_rn(v);
}

__device__ __forceinline__ size_t blh(const ScanDims &d, int b, int t, int h) {
    return (size_t(b) * d.L + t) * d.H + h;
}

// e_t of positions [c0, c0 + n) of head h and their in-chunk inclusive prefix sums (double).
// Executed by warp 0.
__device__ void chunk_rates(const ScanDims &d, int b, int h, int c0, int n, float log_cap,
                            const float *__restrict__ dt, const float *__restrict__ alpha,
                            const float *__restrict__ lam, float *e_s, double *E_s,
                            float *clamp_s) {
    if (threadIdx.x >= 32) return;
    const int lane = threadIdx.x;
    double carry = 0.0;
    for (int base = 0; base < n; base += 32) {
        const int t = base + lane;
        float e = 0.f;
        bool cl = false;
        if (t < n) {
            const size_t i = blh(d, b, c0 + t, h);
            e = token_rate(dt[i], alpha[i], lam[i], log_cap, &cl);
        }
        double v = warp_inclusive_scan_d(double(e)) + carry;
        if (t < n) {
            e_s[t] = e;
            E_s[t] = v;
            if (clamp_s) clamp_s[t] = cl ? 1.f : 0.f;
        }
        carry = __shfl_sync(0xffffffffu, v, 31);
    }
}

__device__ __forceinline__ float head_log_cap(const float *__restrict__ tau, int h, int K) {
    float tmax = 0.f;
    for (int j = 0; j < K; ++j) tmax = fmaxf(tmax, tau[h * K + j]);
    return logf(64.f * tmax);
}

__device__ float block_sum(float v, float *red) {
    v = warp_sum(v);
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    __syncthreads();
    if (lane == 0) red[w] = v;
    __syncthreads();
    float s = 0.f;
    if (threadIdx.x < 32) {
        s = (lane < int(blockDim.x >> 5)) ? red[lane] : 0.f;
        s = warp_sum(s);
        if (lane == 0) red[0] = s;
    }
    __syncthreads();
    s = red[0];
    __syncthreads();
    return s;
}

// ---------------------------------------------------------------------------------------------
// State pass.  REV = false: forward (U = x, V = B, W = w_write, coefficient s).
//              REV = true : backward (U = dy, V = C, W = w_read, coefficient f), chunks reversed.
// Thread tile: one mode m, 8 consecutive p, 4 consecutive n of the CTA's p-slice.
template <typename T, typename TS, bool REV>
__global__ void __launch_bounds__(512) simt_state_pass(
    ScanDims d, int Ps, const T *__restrict__ U, const T *__restrict__ V,
    const T *__restrict__ W, const float *__restrict__ dt, const float *__restrict__ alpha,
    const float *__restrict__ lam, const float *__restrict__ tau, const float *__restrict__ init,
    TS *__restrict__ emit, float *__restrict__ fin) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int b = blockIdx.z, h = blockIdx.y, pbase = blockIdx.x * Ps;
    const int g = h / (d.H / d.G);
    const int K = d.K, N = d.N, P = d.P;
    const int nnt = (N + 3) >> 2, npt = Ps >> 3, Npad = nnt * 4;
    const int ntiles = K * npt * nnt;
    const int tid = threadIdx.x;
    const bool active = tid < ntiles;
    const int nt = tid % nnt, pt = (tid / nnt) % npt, m = active ? tid / (nnt * npt) : 0;
    const int p0 = pbase + pt * 8, n0 = nt * 4;

    double *E_s = reinterpret_cast<double *>(smem_raw);  // [kQMax]
    float *e_s = reinterpret_cast<float *>(E_s + kQMax);  // [kQMax]
    float *itau = e_s + kQMax;                            // [32]
    float *dec = itau + 32;                               // [32]
    float *coef = dec + 32;                               // [kQMax][K]
    float *u_s = coef + kQMax * K;                        // [kQMax][Ps]
    float *v_s = u_s + kQMax * Ps;                        // [kQMax][Npad]

    if (tid < K) itau[tid] = 1.f / tau[h * K + tid];
    const float log_cap = head_log_cap(tau, h, K);
    const size_t PN = size_t(P) * N;
    const size_t bh = size_t(b) * d.H + h;

    float S[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int p = p0 + i, nn = n0 + j;
            S[i][j] = (active && init && p < P && nn < N)
                          ? init[(bh * K + m) * PN + size_t(p) * N + nn]
                          : 0.f;
        }

    for (int ci = 0; ci < d.nc; ++ci) {
        const int c = REV ? d.nc - 1 - ci : ci;
        const int c0 = c * d.Q, n = min(d.Q, d.L - c0);
        __syncthreads();  // the previous chunk's shared-memory reads are done
        chunk_rates(d, b, h, c0, n, log_cap, dt, alpha, lam, e_s, E_s, nullptr);
        // the chunk's rows, four independent loads per thread in flight before their stores
        for (int i0 = tid; i0 < n * Ps; i0 += 4 * blockDim.x) {
            float v[4];
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                const int idx = i0 + r * int(blockDim.x), k = idx / Ps, pp = idx - k * Ps, p = pbase + pp;
                v[r] = (idx < n * Ps && p < P) ? to_f(U[blh(d, b, c0 + k, h) * P + p]) : 0.f;
            }
#pragma unroll
            for (int r = 0; r < 4; ++r)
                if (i0 + r * int(blockDim.x) < n * Ps) u_s[i0 + r * blockDim.x] = v[r];
        }
        for (int i0 = tid; i0 < n * Npad; i0 += 4 * blockDim.x) {
            float v[4];
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                const int idx = i0 + r * int(blockDim.x), k = idx / Npad, nn = idx - k * Npad;
                v[r] = (idx < n * Npad && nn < N) ? to_f(V[((size_t(b) * d.L + c0 + k) * d.G + g) * N + nn]) : 0.f;
            }
#pragma unroll
            for (int r = 0; r < 4; ++r)
                if (i0 + r * int(blockDim.x) < n * Npad) v_s[i0 + r * blockDim.x] = v[r];
        }
        __syncthreads();  // E_s, e_s ready
        const double Eend = E_s[n - 1];
        for (int idx = tid; idx < n * K; idx += blockDim.x) {
            const int k = idx / K, mm = idx - k * K;
            const float w = to_f(W[blh(d, b, c0 + k, h) * K + mm]);
            float cval;
            if (!REV) {
                const float kap = -expm1f(-e_s[k] * itau[mm]) * w;
                cval = kap * expf(-float(Eend - E_s[k]) * itau[mm]);
            } else {
                cval = w * expf(-float(E_s[k]) * itau[mm]);
            }
            coef[k * K + mm] = cval;
        }
        if (tid < K) dec[tid] = expf(-float(Eend) * itau[tid]);
        if (active) {  // emit the state entering this chunk (before its update)
            TS *dst = emit + ((bh * d.nc + c) * K + m) * PN;
#pragma unroll
            for (int i = 0; i < 8; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    if (p0 + i < P && n0 + j < N)
                        dst[size_t(p0 + i) * N + n0 + j] = cvt_state<TS>(S[i][j]);
        }
        __syncthreads();  // coef, dec ready
        if (active) {
            const float dm = dec[m];
#pragma unroll
            for (int i = 0; i < 8; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) S[i][j] *= dm;
            for (int k = 0; k < n; ++k) {
                const float cf = coef[k * K + m];
                const float4 ua = *reinterpret_cast<const float4 *>(u_s + k * Ps + pt * 8);
                const float4 ub = *reinterpret_cast<const float4 *>(u_s + k * Ps + pt * 8 + 4);
                const float4 vv = *reinterpret_cast<const float4 *>(v_s + k * Npad + n0);
                const float cu[8] = {cf * ua.x, cf * ua.y, cf * ua.z, cf * ua.w,
                                     cf * ub.x, cf * ub.y, cf * ub.z, cf * ub.w};
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    S[i][0] = fmaf(cu[i], vv.x, S[i][0]);
                    S[i][1] = fmaf(cu[i], vv.y, S[i][1]);
                    S[i][2] = fmaf(cu[i], vv.z, S[i][2]);
                    S[i][3] = fmaf(cu[i], vv.w, S[i][3]);
                }
            }
        }
    }
    if (active && fin) {
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j)
                if (p0 + i < P && n0 + j < N)
                    fin[(bh * K + m) * PN + size_t(p0 + i) * N + n0 + j] = S[i][j];
    }
}

size_t state_pass_smem(const ScanDims &d, int Ps) {
    const int Npad = ((d.N + 3) >> 2) * 4;
    return sizeof(double) * kQMax + sizeof(float) * (kQMax + 64 + size_t(kQMax) * d.K +
                                                     size_t(kQMax) * Ps + size_t(kQMax) * Npad);
}

// ---------------------------------------------------------------------------------------------
// Chunk output: y for one (b, h, chunk).  Thread tiles: 4x4 over (t, k) for Gamma o G,
// 4 t x 4 p for y (at most two tiles per thread).
template <typename T, typename TS>
__global__ void __launch_bounds__(kThreads) simt_chunk_fwd(
    ScanDims d, const T *__restrict__ x, const T *__restrict__ Bm, const T *__restrict__ Cm,
    const T *__restrict__ wr, const T *__restrict__ ww, const float *__restrict__ dt,
    const float *__restrict__ alpha, const float *__restrict__ lam,
    const float *__restrict__ tau, const float *__restrict__ Dv, const TS *__restrict__ S_in,
    T *__restrict__ y) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int g = h / (d.H / d.G);
    const int K = d.K, N = d.N, P = d.P, Q = d.Q;
    const int c0 = c * Q, n = min(Q, d.L - c0);
    const int P1 = P + 1, N1 = N + 1, Q1 = Q + 1;
    const int tid = threadIdx.x;

    double *E_s = reinterpret_cast<double *>(smem_raw);
    float *e_s = reinterpret_cast<float *>(E_s + kQMax);
    float *itau = e_s + kQMax;
    float *wr_s = itau + 32;            // [Q][K]
    float *kap_s = wr_s + Q * K;        // [Q][K]
    float *f_s = kap_s + Q * K;         // [Q][K]
    float *xs = f_s + Q * K;            // [Q][P1]
    float *Cs = xs + Q * P1;            // [Q][N1]
    float *Bs = Cs + Q * N1;            // [Q][N1]
    float *Ms = Bs + Q * N1;            // [Q][Q1]
    float *Ss = Ms + Q * Q1;            // [P][N1]

    if (tid < K) itau[tid] = 1.f / tau[h * K + tid];
    const float log_cap = head_log_cap(tau, h, K);
    chunk_rates(d, b, h, c0, n, log_cap, dt, alpha, lam, e_s, E_s, nullptr);
    // the chunk's rows, four independent loads per thread in flight before their stores
    for (int i0 = tid; i0 < Q * P; i0 += 4 * blockDim.x) {
        float v[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const int idx = i0 + r * int(blockDim.x), t = idx / P, p = idx - t * P;
            v[r] = (idx < Q * P && t < n) ? to_f(x[blh(d, b, c0 + t, h) * P + p]) : 0.f;
        }
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const int idx = i0 + r * int(blockDim.x), t = idx / P, p = idx - t * P;
            if (idx < Q * P) xs[t * P1 + p] = v[r];
        }
    }
    for (int i0 = tid; i0 < Q * N; i0 += 4 * blockDim.x) {
        float vc[4], vb[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const int idx = i0 + r * int(blockDim.x), t = idx / N, nn = idx - t * N;
            const size_t gi = ((size_t(b) * d.L + c0 + t) * d.G + g) * N + nn;
            const bool in = idx < Q * N && t < n;
            vc[r] = in ? to_f(Cm[gi]) : 0.f;
            vb[r] = in ? to_f(Bm[gi]) : 0.f;
        }
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const int idx = i0 + r * int(blockDim.x), t = idx / N, nn = idx - t * N;
            if (idx < Q * N) {
                Cs[t * N1 + nn] = vc[r];
                Bs[t * N1 + nn] = vb[r];
            }
        }
    }
    __syncthreads();
    for (int idx = tid; idx < Q * K; idx += blockDim.x) {
        const int t = idx / K, mm = idx - t * K;
        float w = 0.f, kp = 0.f, f = 0.f;
        if (t < n) {
            const size_t wi = blh(d, b, c0 + t, h) * K + mm;
            w = to_f(wr[wi]);
            kp = -expm1f(-e_s[t] * itau[mm]) * to_f(ww[wi]);
            f = w * expf(-float(E_s[t]) * itau[mm]);
        }
        wr_s[idx] = w;
        kap_s[idx] = kp;
        f_s[idx] = f;
    }
    __syncthreads();
    // Gamma o (C B^T), lower triangle
    const int qt = Q >> 2;
    for (int tile = tid; tile < qt * qt; tile += blockDim.x) {
        const int t0 = 4 * (tile / qt), k0 = 4 * (tile % qt);
        float G[4][4] = {};
        if (k0 <= t0 + 3) {
            for (int nn = 0; nn < N; ++nn) {
                float cv[4], bv[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    cv[i] = Cs[(t0 + i) * N1 + nn];
                    bv[i] = Bs[(k0 + i) * N1 + nn];
                }
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int j = 0; j < 4; ++j) G[i][j] = fmaf(cv[i], bv[j], G[i][j]);
            }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int t = t0 + i, k = k0 + j;
                float v = 0.f;
                if (k <= t && t < n) {
                    const float dE = float(E_s[t] - E_s[k]);
                    float gam = 0.f;
                    for (int mm = 0; mm < K; ++mm)
                        gam = fmaf(wr_s[t * K + mm] * kap_s[k * K + mm], expf(-dE * itau[mm]), gam);
                    v = gam * G[i][j];
                }
                Ms[t * Q1 + k] = v;
            }
    }
    __syncthreads();
    // y tiles
    const int npt4 = (P + 3) >> 2;
    const int ytiles = qt * npt4;
    float acc[2][4][4] = {};
    int tt0[2], pp0[2];
#pragma unroll
    for (int s = 0; s < 2; ++s) {
        const int tile = tid + s * blockDim.x;
        tt0[s] = 4 * (tile / npt4);
        pp0[s] = 4 * (tile % npt4);
        if (tile < ytiles) {
            const int kend = min(tt0[s] + 4, n);
            for (int k = 0; k < kend; ++k) {
                float mv[4], xv[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    mv[i] = Ms[(tt0[s] + i) * Q1 + k];
                    xv[i] = (pp0[s] + i < P) ? xs[k * P1 + pp0[s] + i] : 0.f;
                }
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int j = 0; j < 4; ++j) acc[s][i][j] = fmaf(mv[i], xv[j], acc[s][i][j]);
            }
        }
    }
    const size_t PN = size_t(P) * N;
    const TS *Sbase = S_in + ((size_t(b) * d.H + h) * d.nc + c) * K * PN;
    for (int mm = 0; mm < K; ++mm) {
        __syncthreads();
        for (int idx = tid; idx < P * N; idx += blockDim.x) {
            const int p = idx / N, nn = idx - p * N;
            Ss[p * N1 + nn] = to_f(Sbase[mm * PN + idx]);
        }
        __syncthreads();
#pragma unroll
        for (int s = 0; s < 2; ++s) {
            const int tile = tid + s * blockDim.x;
            if (tile >= ytiles) continue;
            float z[4][4] = {};
            for (int nn = 0; nn < N; ++nn) {
                float cv[4], sv[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    cv[i] = Cs[(tt0[s] + i) * N1 + nn];
                    sv[i] = (pp0[s] + i < P) ? Ss[(pp0[s] + i) * N1 + nn] : 0.f;
                }
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int j = 0; j < 4; ++j) z[i][j] = fmaf(cv[i], sv[j], z[i][j]);
            }
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float f = f_s[(tt0[s] + i) * K + mm];
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[s][i][j] = fmaf(f, z[i][j], acc[s][i][j]);
            }
        }
    }
    const float Dh = Dv[h];
#pragma unroll
    for (int s = 0; s < 2; ++s) {
        const int tile = tid + s * blockDim.x;
        if (tile >= ytiles) continue;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int t = tt0[s] + i;
            if (t >= n) continue;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int p = pp0[s] + j;
                if (p < P)
                    y[blh(d, b, c0 + t, h) * P + p] =
                        from_f<T>(acc[s][i][j] + Dh * xs[t * P1 + p]);
            }
        }
    }
}

size_t chunk_fwd_smem(const ScanDims &d) {
    const int Q = d.Q;
    return sizeof(double) * kQMax +
           sizeof(float) * (kQMax + 32 + 3 * size_t(Q) * d.K + size_t(Q) * (d.P + 1) +
                            2 * size_t(Q) * (d.N + 1) + size_t(Q) * (Q + 1) +
                            size_t(d.P) * (d.N + 1));
}

// ---------------------------------------------------------------------------------------------
// Chunk backward for one (b, h, chunk).  With G[t,k] = C_t . B_k, H[t,k] = dy_t . x_k,
// W_{t,k,m} = exp(-(E_t - E_k)/tau_m) (t >= k), u_{k,m} = exp(-(E_end - E_k)/tau_m),
// s = kappa u, f = w_read exp(-E_t/tau), U_m = B dS_out,m^T, Z_m = C S_in,m^T:
//   dx_k      = sum_m s_{k,m} U_m[k] + sum_{t>=k} Gamma_{t,k} G_{t,k} dy_t + D dy_k
//   dkappa_km = u_{k,m} x_k . U_m[k] + sum_{t>=k} w_read_{t,m} W_{t,k,m} G_{t,k} H_{t,k}
//   dw_read_tm= exp(-E_t/tau_m) dy_t . Z_m[t] + sum_{k<=t} kappa_{k,m} W_{t,k,m} G_{t,k} H_{t,k}
//   dC_t     += sum_m f_{t,m} S_in,m^T dy_t + sum_{k<=t} Gamma_{t,k} H_{t,k} B_k
//   dB_k     += sum_m s_{k,m} dS_out,m^T x_k + sum_{t>=k} Gamma_{t,k} H_{t,k} C_t
//   sum_m rho_t <dS_t, S_{t-1}>_m / tau_m = sum_{t'>=t} a_t' + sum_{k<t} b_k + c
//                                           + sum_{t'>=t, k<t} Gamma'_{t',k} G_{t',k} H_{t',k}
//        a_t = sum_m f_{t,m} dy_t.Z_m[t] / tau_m,  b_k = sum_m s_{k,m} x_k.U_m[k] / tau_m,
//        c = sum_m d_m <dS_out,m, S_in,m> / tau_m,  Gamma' = Gamma with kappa / tau
//   (every term carries its own decay, so this stays accurate when e_t is large)
//   de_t = -(that) + sum_m dkappa_{t,m} rho_{t,m} w_write_{t,m} / tau_m   (0 if e_t was clamped)
template <typename T, typename TS>
__global__ void __launch_bounds__(kThreads) simt_chunk_bwd(
    ScanDims d, const T *__restrict__ x, const T *__restrict__ Bm, const T *__restrict__ Cm,
    const T *__restrict__ wr, const T *__restrict__ ww, const T *__restrict__ dy,
    const float *__restrict__ dt, const float *__restrict__ alpha, const float *__restrict__ lam,
    const float *__restrict__ tau, const float *__restrict__ Dv, const TS *__restrict__ S_in,
    const TS *__restrict__ dS_out, T *__restrict__ dx, T *__restrict__ dwr_o,
    T *__restrict__ dww_o, float *__restrict__ ddt, float *__restrict__ dalpha,
    float *__restrict__ dlam, float *__restrict__ dD, float *__restrict__ dB_acc,
    float *__restrict__ dC_acc, float *__restrict__ dtau) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int g = h / (d.H / d.G);
    const int K = d.K, N = d.N, P = d.P, Q = d.Q;
    const int c0 = c * Q, n = min(Q, d.L - c0);
    const int P1 = P + 1, N1 = N + 1, Q1 = Q + 1;
    const int tid = threadIdx.x;
    const int QK = Q * K;

    double *E_s = reinterpret_cast<double *>(smem_raw);
    double *dtq_s = E_s + kQMax;    // [32] per mode: sum over the chunk of the dtau terms
    float *e_s = reinterpret_cast<float *>(dtq_s + 32);
    float *cl_s = e_s + kQMax;
    float *itau = cl_s + kQMax;     // [32]
    float *dec = itau + 32;         // [32]
    float *red = dec + 32;          // [32]
    float *cdm_s = red + 32;        // [32] per mode: <S_in, dS_out>
    float *a_s = cdm_s + 32;        // [kQMax]
    float *b_s = a_s + kQMax;       // [kQMax]
    float *rp_s = b_s + kQMax;      // [kQMax]
    float *wr_s = rp_s + kQMax;     // [Q][K] x 11
    float *ww_s = wr_s + QK;
    float *kap_s = ww_s + QK;
    float *rho_s = kap_s + QK;
    float *omr_s = rho_s + QK;
    float *fd_s = omr_s + QK;       // exp(-E_t/tau)
    float *u_s = fd_s + QK;         // exp(-(E_end - E_k)/tau)
    float *dwri = u_s + QK;         // intra part of dw_read
    float *dkpi = dwri + QK;        // intra part of dkappa
    float *xU = dkpi + QK;          // x_k . U_m[k]
    float *dyZ = xU + QK;           // dy_t . Z_m[t]
    float *xs = dyZ + QK;           // [Q][P1]
    float *dys = xs + Q * P1;       // [Q][P1]
    float *Bs = dys + Q * P1;       // [Q][N1]
    float *Cs = Bs + Q * N1;        // [Q][N1]
    float *un = Cs + Q * N1;        // union
    float *MG = un;                 // [Q][Q1]  Gamma o G
    float *MH = MG + Q * Q1;        // [Q][Q1]  Gamma o H
    float *XX = MH + Q * Q1;        // [Q][Q1]  Gamma' o G o H
    float *Ss = un;                 // [P][N1]
    float *dSs = Ss + P * N1;       // [P][N1]

    // ---- loads
    if (tid < K) itau[tid] = 1.f / tau[h * K + tid];
    if (tid < 32) {
        dtq_s[tid] = 0.0;
        cdm_s[tid] = 0.f;
    }
    const float log_cap = head_log_cap(tau, h, K);
    chunk_rates(d, b, h, c0, n, log_cap, dt, alpha, lam, e_s, E_s, cl_s);
    for (int idx = tid; idx < Q * P; idx += blockDim.x) {
        const int t = idx / P, p = idx - t * P;
        const size_t gi = blh(d, b, c0 + t, h) * P + p;
        xs[t * P1 + p] = t < n ? to_f(x[gi]) : 0.f;
        dys[t * P1 + p] = t < n ? to_f(dy[gi]) : 0.f;
    }
    for (int idx = tid; idx < Q * N; idx += blockDim.x) {
        const int t = idx / N, nn = idx - t * N;
        const size_t gi = ((size_t(b) * d.L + c0 + t) * d.G + g) * N + nn;
        Cs[t * N1 + nn] = t < n ? to_f(Cm[gi]) : 0.f;
        Bs[t * N1 + nn] = t < n ? to_f(Bm[gi]) : 0.f;
    }
    __syncthreads();
    const double Eend = E_s[n - 1];
    for (int idx = tid; idx < QK; idx += blockDim.x) {
        const int t = idx / K, mm = idx - t * K;
        float w_r = 0.f, w_w = 0.f, rho = 0.f, omr = 0.f, fd = 0.f, uu = 0.f;
        if (t < n) {
            const size_t wi = blh(d, b, c0 + t, h) * K + mm;
            w_r = to_f(wr[wi]);
            w_w = to_f(ww[wi]);
            const float z = e_s[t] * itau[mm];
            rho = expf(-z);
            omr = -expm1f(-z);
            fd = expf(-float(E_s[t]) * itau[mm]);
            uu = expf(-float(Eend - E_s[t]) * itau[mm]);
        }
        wr_s[idx] = w_r;
        ww_s[idx] = w_w;
        kap_s[idx] = omr * w_w;
        rho_s[idx] = rho;
        omr_s[idx] = omr;
        fd_s[idx] = fd;
        u_s[idx] = uu;
        dwri[idx] = 0.f;
        dkpi[idx] = 0.f;
        xU[idx] = 0.f;
        dyZ[idx] = 0.f;
    }
    if (tid < K) dec[tid] = expf(-float(Eend) * itau[tid]);
    __syncthreads();

    // ---- intra-chunk pairs: 4 t x 4 k tiles
    const int qt = Q >> 2;
    for (int tile = tid; tile < qt * qt; tile += blockDim.x) {
        const int t0 = 4 * (tile / qt), k0 = 4 * (tile % qt);
        float G[4][4] = {}, Hm[4][4] = {};
        if (k0 <= t0 + 3) {
            for (int nn = 0; nn < N; ++nn) {
                float cv[4], bv[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    cv[i] = Cs[(t0 + i) * N1 + nn];
                    bv[i] = Bs[(k0 + i) * N1 + nn];
                }
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int j = 0; j < 4; ++j) G[i][j] = fmaf(cv[i], bv[j], G[i][j]);
            }
            for (int p = 0; p < P; ++p) {
                float dv[4], xv[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    dv[i] = dys[(t0 + i) * P1 + p];
                    xv[i] = xs[(k0 + i) * P1 + p];
                }
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int j = 0; j < 4; ++j) Hm[i][j] = fmaf(dv[i], xv[j], Hm[i][j]);
            }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int t = t0 + i, k = k0 + j;
                float mg = 0.f, mh = 0.f, xx = 0.f;
                if (k <= t && t < n) {
                    const float dE = float(E_s[t] - E_s[k]);
                    const float gh = G[i][j] * Hm[i][j];
                    float gam = 0.f, gamt = 0.f;
                    for (int mm = 0; mm < K; ++mm) {
                        const float Wm = expf(-dE * itau[mm]);
                        const float a = wr_s[t * K + mm] * kap_s[k * K + mm] * Wm;
                        gam += a;
                        gamt = fmaf(a, itau[mm], gamt);
                        const float cw = Wm * gh;
                        atomicAdd(&dwri[t * K + mm], kap_s[k * K + mm] * cw);
                        atomicAdd(&dkpi[k * K + mm], wr_s[t * K + mm] * cw);
                    }
                    mg = gam * G[i][j];
                    mh = gam * Hm[i][j];
                    xx = gamt * gh;
                }
                MG[t * Q1 + k] = mg;
                MH[t * Q1 + k] = mh;
                XX[t * Q1 + k] = xx;
            }
    }
    __syncthreads();
    // exclusive row prefix of XX, then column suffix -> pair rectangle sums
    if (tid < Q) {
        float run = 0.f;
        for (int j = 0; j < Q; ++j) {
            const float v = XX[tid * Q1 + j];
            XX[tid * Q1 + j] = run;
            run += v;
        }
    }
    __syncthreads();
    if (tid < Q) {
        float s = 0.f;
        for (int tp = tid; tp < n; ++tp) s += XX[tp * Q1 + tid];
        rp_s[tid] = s;
    }

    // ---- register tiles: dx (4 k x 4 p), dC / dB (4 rows x 8 n)
    const int npt4 = (P + 3) >> 2, nnt8 = (N + 7) >> 3;
    const bool has_x = tid < qt * npt4, has_cb = tid < qt * nnt8;
    const int xr0 = 4 * (tid / npt4), xp0 = 4 * (tid % npt4);
    const int cr0 = 4 * (tid / nnt8), cn0 = 8 * (tid % nnt8);
    float adx[4][4] = {}, adC[4][8] = {}, adB[4][8] = {};
    if (has_x) {
        for (int t = xr0; t < n; ++t) {
            float mv[4], dv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                mv[i] = MG[t * Q1 + xr0 + i];
                dv[i] = (xp0 + i < P) ? dys[t * P1 + xp0 + i] : 0.f;
            }
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) adx[i][j] = fmaf(mv[i], dv[j], adx[i][j]);
        }
    }
    if (has_cb) {
        for (int k = 0; k < min(cr0 + 4, n); ++k) {  // dC_t += sum_{k<=t} (Gamma o H)[t,k] B_k
            float mv[4], bv[8];
#pragma unroll
            for (int i = 0; i < 4; ++i) mv[i] = MH[(cr0 + i) * Q1 + k];
#pragma unroll
            for (int j = 0; j < 8; ++j) bv[j] = (cn0 + j < N) ? Bs[k * N1 + cn0 + j] : 0.f;
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 8; ++j) adC[i][j] = fmaf(mv[i], bv[j], adC[i][j]);
        }
        for (int t = cr0; t < n; ++t) {  // dB_k += sum_{t>=k} (Gamma o H)[t,k] C_t
            float mv[4], cv[8];
#pragma unroll
            for (int i = 0; i < 4; ++i) mv[i] = MH[t * Q1 + cr0 + i];
#pragma unroll
            for (int j = 0; j < 8; ++j) cv[j] = (cn0 + j < N) ? Cs[t * N1 + cn0 + j] : 0.f;
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 8; ++j) adB[i][j] = fmaf(mv[i], cv[j], adB[i][j]);
        }
    }

    // ---- inter-chunk terms, mode by mode
    const size_t PN = size_t(P) * N;
    const size_t sbase = ((size_t(b) * d.H + h) * d.nc + c) * K * PN;
    float cpart = 0.f;
    for (int mm = 0; mm < K; ++mm) {
        __syncthreads();  // the union region / previous mode is no longer read
        float dot = 0.f;
        for (int idx = tid; idx < P * N; idx += blockDim.x) {
            const int p = idx / N, nn = idx - p * N;
            const float sv = to_f(S_in[sbase + mm * PN + idx]);
            const float dv = to_f(dS_out[sbase + mm * PN + idx]);
            Ss[p * N1 + nn] = sv;
            dSs[p * N1 + nn] = dv;
            dot = fmaf(sv, dv, dot);
        }
        cpart = fmaf(dec[mm] * itau[mm], dot, cpart);
        if (dtau) atomicAdd(&cdm_s[mm], dot);
        __syncthreads();
        if (has_x) {
            float Uq[4][4] = {}, Zq[4][4] = {};
            for (int nn = 0; nn < N; ++nn) {
                float bv[4], cv[4], dsv[4], sv[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    bv[i] = Bs[(xr0 + i) * N1 + nn];
                    cv[i] = Cs[(xr0 + i) * N1 + nn];
                    const bool ok = xp0 + i < P;
                    dsv[i] = ok ? dSs[(xp0 + i) * N1 + nn] : 0.f;
                    sv[i] = ok ? Ss[(xp0 + i) * N1 + nn] : 0.f;
                }
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        Uq[i][j] = fmaf(bv[i], dsv[j], Uq[i][j]);
                        Zq[i][j] = fmaf(cv[i], sv[j], Zq[i][j]);
                    }
            }
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int r = xr0 + i;
                const float sk = kap_s[r * K + mm] * u_s[r * K + mm];
                float xu = 0.f, dz = 0.f;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    adx[i][j] = fmaf(sk, Uq[i][j], adx[i][j]);
                    if (xp0 + j < P) {
                        xu = fmaf(xs[r * P1 + xp0 + j], Uq[i][j], xu);
                        dz = fmaf(dys[r * P1 + xp0 + j], Zq[i][j], dz);
                    }
                }
                if (r < n) {
                    atomicAdd(&xU[r * K + mm], xu);
                    atomicAdd(&dyZ[r * K + mm], dz);
                }
            }
        }
        if (has_cb) {
            float fr[4], sr[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int r = cr0 + i;
                fr[i] = wr_s[r * K + mm] * fd_s[r * K + mm];
                sr[i] = kap_s[r * K + mm] * u_s[r * K + mm];
            }
            for (int p = 0; p < P; ++p) {
                float fy[4], sx[4], sv[8], dsv[8];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    fy[i] = fr[i] * dys[(cr0 + i) * P1 + p];
                    sx[i] = sr[i] * xs[(cr0 + i) * P1 + p];
                }
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const bool ok = cn0 + j < N;
                    sv[j] = ok ? Ss[p * N1 + cn0 + j] : 0.f;
                    dsv[j] = ok ? dSs[p * N1 + cn0 + j] : 0.f;
                }
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        adC[i][j] = fmaf(fy[i], sv[j], adC[i][j]);
                        adB[i][j] = fmaf(sx[i], dsv[j], adB[i][j]);
                    }
            }
        }
    }
    const float cprime = block_sum(cpart, red);  // contains __syncthreads

    // ---- dD partial
    float dd = 0.f;
    for (int idx = tid; idx < n * P; idx += blockDim.x) {
        const int t = idx / P, p = idx - t * P;
        dd = fmaf(dys[t * P1 + p], xs[t * P1 + p], dd);
    }
    dd = block_sum(dd, red);
    if (tid == 0) atomicAdd(&dD[h], dd);

    // ---- stores of the tiles
    const float Dh = Dv[h];
    if (has_x) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int t = xr0 + i;
            if (t >= n) continue;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int p = xp0 + j;
                if (p < P)
                    dx[blh(d, b, c0 + t, h) * P + p] =
                        from_f<T>(adx[i][j] + Dh * dys[t * P1 + p]);
            }
        }
    }
    if (has_cb) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int t = cr0 + i;
            if (t >= n) continue;
            const size_t gi = ((size_t(b) * d.L + c0 + t) * d.G + g) * N;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int nn = cn0 + j;
                if (nn < N) {
                    atomicAdd(&dC_acc[gi + nn], adC[i][j]);
                    atomicAdd(&dB_acc[gi + nn], adB[i][j]);
                }
            }
        }
    }
    // ---- per-position scalars
    if (tid < n) {
        const int t = tid;
        float a = 0.f, bb = 0.f;
        for (int mm = 0; mm < K; ++mm) {
            a = fmaf(wr_s[t * K + mm] * fd_s[t * K + mm] * dyZ[t * K + mm], itau[mm], a);
            bb = fmaf(kap_s[t * K + mm] * u_s[t * K + mm] * xU[t * K + mm], itau[mm], bb);
        }
        a_s[t] = a;
        b_s[t] = bb;
    }
    __syncthreads();
    if (tid < n) {
        const int t = tid;
        float suf = 0.f, pre = 0.f;
        for (int j = t; j < n; ++j) suf += a_s[j];
        for (int j = 0; j < t; ++j) pre += b_s[j];
        const float R = suf + pre + cprime + rp_s[t];
        float de = -R;
        const size_t wi0 = blh(d, b, c0 + t, h) * K;
        for (int mm = 0; mm < K; ++mm) {
            const int q = t * K + mm;
            const float dk = u_s[q] * xU[q] + dkpi[q];
            const float dw = fd_s[q] * dyZ[q] + dwri[q];
            de = fmaf(dk * rho_s[q] * ww_s[q], itau[mm], de);
            dwr_o[wi0 + mm] = from_f<T>(dw);
            dww_o[wi0 + mm] = from_f<T>(dk * omr_s[q]);
            if (dtau) {
                // timescale gradient, the terms with S_in or dS_out, each weighted by the e_t it
                // spans (E_t, E_end - E_t); the pairs inside the chunk come from dtau_pairs
                const double Et = E_s[t], Eend = E_s[n - 1];
                const double tq = Et * double(wr_s[q]) * double(fd_s[q] * dyZ[q]) +
                                  (Eend - Et) * double(kap_s[q]) * double(u_s[q] * xU[q]) -
                                  double(e_s[t]) * double(dk) * double(rho_s[q]) * double(ww_s[q]);
                atomicAdd(&dtq_s[mm], tq);
            }
        }
        const size_t i = blh(d, b, c0 + t, h);
        const float e = e_s[t];
        const bool cl = cl_s[t] != 0.f;
        const float al = alpha[i], lm = lam[i], dtv = dt[i];
        const float ge = cl ? 0.f : de * e;
        ddt[i] = ge / dtv;
        dlam[i] = ge / (al * lm);
        dalpha[i] = -ge * logf(lm) / (al * al);
    }
    if (dtau) {  // dtau_m += (sum_t ... + E_end d_m <dS_out, S_in>_m) / tau_m^2
        __syncthreads();
        if (tid < K)
            atomicAdd(&dtau[h * K + tid],
                      float((dtq_s[tid] + E_s[n - 1] * double(dec[tid]) * double(cdm_s[tid])) *
                            double(itau[tid]) * double(itau[tid])));
    }
}

size_t chunk_bwd_smem(const ScanDims &d) {
    const size_t Q = d.Q, P1 = d.P + 1, N1 = d.N + 1;
    const size_t uni = std::max(3 * Q * (Q + 1), 2 * size_t(d.P) * N1);
    return sizeof(double) * (kQMax + 32) +
           sizeof(float) * (2 * kQMax + 4 * 32 + 3 * kQMax + 11 * Q * d.K + 2 * Q * P1 +
                            2 * Q * N1 + uni);
}

__global__ void f32_to_bf16_kernel(const float *__restrict__ in, __nv_bfloat16 *__restrict__ out,
                                   size_t n) {
    for (size_t i = blockIdx.x * size_t(blockDim.x) + threadIdx.x; i < n;
         i += size_t(gridDim.x) * blockDim.x)
        out[i] = __float2bfloat16_rn(in[i]);
}

int state_pass_ps(const ScanDims &d) {
    const int nnt = (d.N + 3) >> 2;
    const int per8 = d.K * nnt;  // tiles per 8 p-rows
    if (per8 > 512) return 0;
    int npt = std::max(1, 256 / per8);
    npt = std::min(npt, (d.P + 7) / 8);
    npt = std::max(1, std::min(npt, 512 / per8));
    return npt * 8;
}

template <typename T, typename TS>
cudaError_t run_state_pass(const ScanDims &d, bool rev, const void *U, const void *V,
                           const void *W, const ScanPtrs &p, const float *init, void *emit,
                           float *fin, cudaStream_t st) {
    const int Ps = state_pass_ps(d);
    const int ntiles = d.K * (Ps / 8) * ((d.N + 3) >> 2);
    // at least 256 threads: the ones beyond the register tiles only help stage each chunk's rows
    const int threads = std::max(((ntiles + 31) / 32) * 32, 256);
    const size_t smem = state_pass_smem(d, Ps);
    dim3 grid((d.P + Ps - 1) / Ps, d.H, d.B);
    if (rev) {
        auto k = simt_state_pass<T, TS, true>;
        cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        trace_begin("state_pass_rev_simt", st);
        k<<<grid, threads, smem, st>>>(d, Ps, (const T *)U, (const T *)V, (const T *)W, p.dt,
                                       p.alpha, p.lam, p.tau, init, (TS *)emit, fin);
        trace_end(st);
    } else {
        auto k = simt_state_pass<T, TS, false>;
        cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        trace_begin("state_pass_fwd_simt", st);
        k<<<grid, threads, smem, st>>>(d, Ps, (const T *)U, (const T *)V, (const T *)W, p.dt,
                                       p.alpha, p.lam, p.tau, init, (TS *)emit, fin);
        trace_end(st);
    }
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// N = 1 (the paper's own layer: scalar B, C per position): each (mode, p) is a scalar
// recurrence S <- rho S + kappa B x, y = sum_m w_read C S + D x, so the forward runs it directly
// (K fused multiply-adds per mode row and token) instead of the pairwise intra-chunk form.
// Per chunk, the coefficients of its positions and modes go to shared memory first:
// rho = exp(-e/tau), kappa B = -expm1(-e/tau) w_write B and (output kernel) w_read C.
constexpr int kN1Modes = 32;  // nmodes <= 32 (checked at the boundary)
constexpr int kN1P = 256;     // p per CTA of the N = 1 chunk kernels (one thread each)

template <typename T>
__device__ void n1_chunk_coefs(const ScanDims &d, int b, int h, int c0, int n, float log_cap,
                               const float *__restrict__ itau, const T *__restrict__ Bm,
                               const T *__restrict__ Cm, const T *__restrict__ ww,
                               const T *__restrict__ wr, const float *__restrict__ dt,
                               const float *__restrict__ alpha, const float *__restrict__ lam,
                               float *e_s, float *rho_s, float *kb_s, float *wc_s) {
    const int K = d.K, g = h / (d.H / d.G);
    for (int t = threadIdx.x; t < n; t += blockDim.x) {
        const size_t i = blh(d, b, c0 + t, h);
        bool cl = false;
        e_s[t] = token_rate(dt[i], alpha[i], lam[i], log_cap, &cl);
    }
    __syncthreads();
    for (int idx = threadIdx.x; idx < n * K; idx += blockDim.x) {
        const int t = idx / K, m = idx - t * K;
        const size_t i = blh(d, b, c0 + t, h);
        const size_t ig = (size_t(b) * d.L + c0 + t) * d.G + g;  // N = 1: one B, C per group
        const float z = e_s[t] * itau[m];
        rho_s[idx] = expf(-z);
        kb_s[idx] = -expm1f(-z) * to_f(ww[i * K + m]) * to_f(Bm[ig]);
        if (wc_s) wc_s[idx] = to_f(wr[i * K + m]) * to_f(Cm[ig]);
    }
    __syncthreads();
}

// The chunk's x rows of one 256-wide p block into shared memory (row stride 256 elements):
// 16-byte asynchronous copies when every row segment is a whole number of aligned 16-byte
// pieces (VEC), element loads otherwise.  Issued before the coefficients are computed, so the
// recurrence never waits on HBM; completed by n1_x_wait.
template <typename T, bool VEC>
__device__ __forceinline__ void n1_x_issue(const ScanDims &d, const T *__restrict__ x, int b, int h, int c0,
                                           int n, int p0, int np, T *x_s) {
    if constexpr (VEC) {
        constexpr int PER = 16 / sizeof(T);
        const int pieces = np / PER;
        for (int idx = threadIdx.x; idx < n * pieces; idx += blockDim.x) {
            const int t = idx / pieces, q = idx - t * pieces;
            const uint32_t dst = static_cast<uint32_t>(__cvta_generic_to_shared(x_s + t * kN1P + q * PER));
            const T *src = x + blh(d, b, c0 + t, h) * d.P + p0 + q * PER;
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    } else {
        for (int idx = threadIdx.x; idx < n * kN1P; idx += blockDim.x) {
            const int t = idx / kN1P, q = idx - t * kN1P;
            if (q < np) x_s[t * kN1P + q] = x[blh(d, b, c0 + t, h) * d.P + p0 + q];
        }
    }
}
template <bool VEC>
__device__ __forceinline__ void n1_x_wait() {
    if constexpr (VEC) asm volatile("cp.async.wait_all;" ::: "memory");
    __syncthreads();
}

struct N1Smem {  // dynamic shared memory of the N = 1 chunk kernels
    size_t e, itau, rho, kb, wc, x, total;
    __host__ __device__ N1Smem(size_t esz) {
        e = 0;
        itau = e + sizeof(float) * kQMax;
        rho = itau + sizeof(float) * kN1Modes;
        kb = rho + sizeof(float) * kQMax * kN1Modes;
        wc = kb + sizeof(float) * kQMax * kN1Modes;
        x = wc + sizeof(float) * kQMax * kN1Modes;
        total = x + esz * kQMax * kN1P;
    }
};

// Chunk-local pass: per chunk, the state the chunk alone leaves at its end (from zero) for each
// (mode, p), and (threads of the first p block) the chunk's decay prod_t rho_t per mode, the
// same products the recurrence applies.  One thread per p of a 256-wide block.
template <typename T, bool VEC, int KP>
__global__ void __launch_bounds__(kN1P) n1_local(ScanDims d, const T *__restrict__ x, const T *__restrict__ Bm,
                                                const T *__restrict__ ww, const float *__restrict__ dt,
                                                const float *__restrict__ alpha, const float *__restrict__ lam,
                                                const float *__restrict__ tau, float *__restrict__ loc,
                                                float *__restrict__ dec) {
    extern __shared__ __align__(16) unsigned char n1_smem[];
    const N1Smem L_(sizeof(T));
    float *e_s = reinterpret_cast<float *>(n1_smem + L_.e), *itau = reinterpret_cast<float *>(n1_smem + L_.itau);
    float *rho_s = reinterpret_cast<float *>(n1_smem + L_.rho), *kb_s = reinterpret_cast<float *>(n1_smem + L_.kb);
    T *x_s = reinterpret_cast<T *>(n1_smem + L_.x);
    const int K = d.K, P = d.P;
    const int npb = (P + kN1P - 1) / kN1P;
    const int c = blockIdx.x, h = blockIdx.y / npb, b = blockIdx.z, pb = blockIdx.y % npb;
    const int p0 = pb * kN1P, np = min(kN1P, P - p0), p = p0 + threadIdx.x;
    const size_t bh = size_t(b) * d.H + h;
    const int c0 = c * d.Q, n = min(d.Q, d.L - c0);
    n1_x_issue<T, VEC>(d, x, b, h, c0, n, p0, np, x_s);
    if (threadIdx.x < K) itau[threadIdx.x] = 1.f / tau[h * K + threadIdx.x];
    const float log_cap = head_log_cap(tau, h, K);
    __syncthreads();
    n1_chunk_coefs<T>(d, b, h, c0, n, log_cap, itau, Bm, nullptr, ww, nullptr, dt, alpha, lam, e_s, rho_s,
                      kb_s, nullptr);
    n1_x_wait<VEC>();
    if (pb == 0 && threadIdx.x < K) {
        float a = 1.f;
        for (int t = 0; t < n; ++t) a *= rho_s[t * K + threadIdx.x];
        dec[(bh * d.nc + c) * K + threadIdx.x] = a;
    }
    if (threadIdx.x >= np) return;
    float S[KP];
#pragma unroll
    for (int m = 0; m < KP; ++m) S[m] = 0.f;
#pragma unroll 4
    for (int t = 0; t < n; ++t) {
        const float xv = to_f(x_s[t * kN1P + threadIdx.x]);
        if ((K & 3) == 0) {  // rows of 16-byte pieces; packed float32 pairs (the same IEEE operations)
            const float4 *r4 = reinterpret_cast<const float4 *>(rho_s + t * K);
            const float4 *k4 = reinterpret_cast<const float4 *>(kb_s + t * K);
            const float2 xx = make_float2(xv, xv);
#pragma unroll
            for (int q = 0; q < KP / 4; ++q) {
                if (4 * q < K) {
                    const float4 r = r4[q], kv = k4[q];
                    const float2 a = __ffma2_rn(make_float2(r.x, r.y), make_float2(S[4 * q], S[4 * q + 1]),
                                                __fmul2_rn(make_float2(kv.x, kv.y), xx));
                    const float2 c2 = __ffma2_rn(make_float2(r.z, r.w), make_float2(S[4 * q + 2], S[4 * q + 3]),
                                                 __fmul2_rn(make_float2(kv.z, kv.w), xx));
                    S[4 * q] = a.x;
                    S[4 * q + 1] = a.y;
                    S[4 * q + 2] = c2.x;
                    S[4 * q + 3] = c2.y;
                }
            }
        } else {
#pragma unroll
            for (int m = 0; m < KP; ++m)
                if (m < K) S[m] = fmaf(rho_s[t * K + m], S[m], kb_s[t * K + m] * xv);
        }
    }
#pragma unroll
    for (int m = 0; m < KP; ++m)
        if (m < K) loc[((bh * d.nc + c) * K + m) * P + p] = S[m];
}

// Serial combine over chunks, one thread per (b, h, mode, p): S_in[c] = S, then
// S = decay_c S + local_c; the last S is the final state.  The local states and decays of 16
// chunks are loaded at once (all in flight) before their dependent updates.
template <typename TS>
__global__ void __launch_bounds__(256) n1_combine(ScanDims d, const float *__restrict__ loc,
                                                 const float *__restrict__ dec, const float *__restrict__ init,
                                                 TS *__restrict__ emit, float *__restrict__ fin) {
    constexpr int kBatch = 16;
    const size_t total = size_t(d.B) * d.H * d.K * d.P;
    const size_t idx = size_t(blockIdx.x) * blockDim.x + threadIdx.x;
    if (idx >= total) return;
    const int p = int(idx % d.P);
    const size_t bhm = idx / d.P;  // (b h) K + m
    const int m = int(bhm % d.K);
    const size_t bh = bhm / d.K;
    float S = init ? init[idx] : 0.f;  // [B, H, K, P] (N = 1)
    for (int c0 = 0; c0 < d.nc; c0 += kBatch) {
        float lv[kBatch], dv[kBatch];
#pragma unroll
        for (int j = 0; j < kBatch; ++j) {
            const int c = c0 + j;
            lv[j] = c < d.nc ? loc[((bh * d.nc + c) * d.K + m) * d.P + p] : 0.f;
            dv[j] = c < d.nc ? dec[(bh * d.nc + c) * d.K + m] : 0.f;
        }
#pragma unroll
        for (int j = 0; j < kBatch; ++j) {
            const int c = c0 + j;
            if (c < d.nc) {
                emit[((bh * d.nc + c) * d.K + m) * d.P + p] = from_f<TS>(S);
                S = fmaf(dv[j], S, lv[j]);
            }
        }
    }
    if (fin) fin[idx] = S;
}

// Chunk-parallel output: from the chunk's entering state, the recurrence again with
// y_t = sum_m w_read C S_m + D x_t after each update; one thread per p of a 256-wide block.
template <typename T, typename TS, bool VEC, int KP>
__global__ void __launch_bounds__(kN1P) n1_chunk_fwd(ScanDims d, const T *__restrict__ x,
                                                     const T *__restrict__ Bm, const T *__restrict__ Cm,
                                                     const T *__restrict__ wr, const T *__restrict__ ww,
                                                     const float *__restrict__ dt, const float *__restrict__ alpha,
                                                     const float *__restrict__ lam, const float *__restrict__ tau,
                                                     const float *__restrict__ Dp, const TS *__restrict__ S_in,
                                                     T *__restrict__ y) {
    extern __shared__ __align__(16) unsigned char n1_smem[];
    const N1Smem L_(sizeof(T));
    float *e_s = reinterpret_cast<float *>(n1_smem + L_.e), *itau = reinterpret_cast<float *>(n1_smem + L_.itau);
    float *rho_s = reinterpret_cast<float *>(n1_smem + L_.rho), *kb_s = reinterpret_cast<float *>(n1_smem + L_.kb);
    float *wc_s = reinterpret_cast<float *>(n1_smem + L_.wc);
    T *x_s = reinterpret_cast<T *>(n1_smem + L_.x);
    const int K = d.K, P = d.P;
    const int npb = (P + kN1P - 1) / kN1P;
    const int c = blockIdx.x, h = blockIdx.y / npb, b = blockIdx.z;
    const int p0 = (blockIdx.y % npb) * kN1P, np = min(kN1P, P - p0), p = p0 + threadIdx.x;
    const bool active = threadIdx.x < np;
    const size_t bh = size_t(b) * d.H + h;
    const int c0 = c * d.Q, n = min(d.Q, d.L - c0);
    n1_x_issue<T, VEC>(d, x, b, h, c0, n, p0, np, x_s);
    if (threadIdx.x < K) itau[threadIdx.x] = 1.f / tau[h * K + threadIdx.x];
    const float log_cap = head_log_cap(tau, h, K);
    float S[KP];
#pragma unroll
    for (int m = 0; m < KP; ++m)
        S[m] = (active && m < K) ? to_f(S_in[((bh * d.nc + c) * K + m) * P + p]) : 0.f;
    __syncthreads();
    n1_chunk_coefs<T>(d, b, h, c0, n, log_cap, itau, Bm, Cm, ww, wr, dt, alpha, lam, e_s, rho_s, kb_s,
                      wc_s);
    n1_x_wait<VEC>();
    if (!active) return;
    const float Dh = Dp[h];
#pragma unroll 4
    for (int t = 0; t < n; ++t) {
        const float xv = to_f(x_s[t * kN1P + threadIdx.x]);
        float ya[4] = {Dh * xv, 0.f, 0.f, 0.f};  // four independent partial readout sums
        if ((K & 3) == 0) {  // rows of 16-byte pieces; packed float32 pairs (the same IEEE operations)
            const float4 *r4 = reinterpret_cast<const float4 *>(rho_s + t * K);
            const float4 *k4 = reinterpret_cast<const float4 *>(kb_s + t * K);
            const float4 *w4 = reinterpret_cast<const float4 *>(wc_s + t * K);
            const float2 xx = make_float2(xv, xv);
            float2 y01 = make_float2(ya[0], ya[1]), y23 = make_float2(ya[2], ya[3]);
#pragma unroll
            for (int q = 0; q < KP / 4; ++q) {
                if (4 * q < K) {
                    const float4 r = r4[q], kv = k4[q], wv = w4[q];
                    const float2 a = __ffma2_rn(make_float2(r.x, r.y), make_float2(S[4 * q], S[4 * q + 1]),
                                                __fmul2_rn(make_float2(kv.x, kv.y), xx));
                    const float2 c2 = __ffma2_rn(make_float2(r.z, r.w), make_float2(S[4 * q + 2], S[4 * q + 3]),
                                                 __fmul2_rn(make_float2(kv.z, kv.w), xx));
                    S[4 * q] = a.x;
                    S[4 * q + 1] = a.y;
                    S[4 * q + 2] = c2.x;
                    S[4 * q + 3] = c2.y;
                    y01 = __ffma2_rn(make_float2(wv.x, wv.y), a, y01);
                    y23 = __ffma2_rn(make_float2(wv.z, wv.w), c2, y23);
                }
            }
            ya[0] = y01.x;
            ya[1] = y01.y;
            ya[2] = y23.x;
            ya[3] = y23.y;
        } else {
#pragma unroll
            for (int m = 0; m < KP; ++m) {
                if (m < K) {
                    S[m] = fmaf(rho_s[t * K + m], S[m], kb_s[t * K + m] * xv);
                    ya[m & 3] = fmaf(wc_s[t * K + m], S[m], ya[m & 3]);
                }
            }
        }
        y[blh(d, b, c0 + t, h) * P + p] = from_f<T>((ya[0] + ya[1]) + (ya[2] + ya[3]));
    }
}

template <typename T, typename TS>
cudaError_t fwd_n1(const ScanDims &d, const ScanPtrs &p, void *S_in, float *scratch, cudaStream_t st) {
    const int npb = (d.P + kN1P - 1) / kN1P;
    float *loc = scratch, *dec = scratch + size_t(d.B) * d.H * d.nc * d.K * d.P;
    // 16-byte copies of the x rows when x is 16-byte aligned and a head's row is whole pieces
    const bool vec = (reinterpret_cast<uintptr_t>(p.x) % 16 == 0) && ((size_t(d.P) * sizeof(T)) % 16 == 0);
    const size_t smem = N1Smem(sizeof(T)).total;
    cudaError_t e = cudaSuccess;
    const int KP = d.K <= 4 ? 4 : d.K <= 8 ? 8 : d.K <= 16 ? 16 : 32;
    auto pick_local = [&](auto kp) {
        constexpr int V = decltype(kp)::value;
        return vec ? n1_local<T, true, V> : n1_local<T, false, V>;
    };
    auto pick_out = [&](auto kp) {
        constexpr int V = decltype(kp)::value;
        return vec ? n1_chunk_fwd<T, TS, true, V> : n1_chunk_fwd<T, TS, false, V>;
    };
    using I4 = std::integral_constant<int, 4>;
    using I8 = std::integral_constant<int, 8>;
    using I16 = std::integral_constant<int, 16>;
    using I32 = std::integral_constant<int, 32>;
    auto kl = KP == 4 ? pick_local(I4{}) : KP == 8 ? pick_local(I8{}) : KP == 16 ? pick_local(I16{}) : pick_local(I32{});
    auto ko = KP == 4 ? pick_out(I4{}) : KP == 8 ? pick_out(I8{}) : KP == 16 ? pick_out(I16{}) : pick_out(I32{});
    if (d.nc > 0) {
        cudaFuncSetAttribute(kl, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        trace_begin("local_fwd_n1", st);
        kl<<<dim3(d.nc, d.H * npb, d.B), kN1P, smem, st>>>(d, (const T *)p.x, (const T *)p.Bm, (const T *)p.ww,
                                                           p.dt, p.alpha, p.lam, p.tau, loc, dec);
        trace_end(st);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    const size_t total = size_t(d.B) * d.H * d.K * d.P;
    trace_begin("combine_fwd_n1", st);
    n1_combine<TS><<<unsigned((total + 255) / 256), 256, 0, st>>>(d, loc, dec, p.h0, (TS *)S_in, p.h_final);
    trace_end(st);
    if ((e = cudaGetLastError()) != cudaSuccess || d.nc == 0) return e;  // L = 0: h_final = h0
    cudaFuncSetAttribute(ko, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    trace_begin("chunk_fwd_n1", st);
    ko<<<dim3(d.nc, d.H * npb, d.B), kN1P, smem, st>>>(
        d, (const T *)p.x, (const T *)p.Bm, (const T *)p.Cm, (const T *)p.wr, (const T *)p.ww, p.dt,
        p.alpha, p.lam, p.tau, p.D, (const TS *)S_in, (T *)p.y);
    trace_end(st);
    return cudaGetLastError();
}

bool uses_n1(const ScanDims &d) {  // grid y of the chunk kernels: heads x p blocks
    return d.N == 1 && d.Q <= kQMax && d.K <= kN1Modes && size_t(d.H) * ((d.P + kN1P - 1) / kN1P) <= 65535;
}

template <typename T, typename TS>
cudaError_t fwd_t(const ScanDims &d, const ScanPtrs &p, void *S_in, float *scratch, cudaStream_t st) {
    if (uses_n1(d)) return fwd_n1<T, TS>(d, p, S_in, scratch, st);
    cudaError_t e = run_state_pass<T, TS>(d, false, p.x, p.Bm, p.ww, p, p.h0, S_in, p.h_final, st);
    if (e != cudaSuccess || d.nc == 0) return e;  // L = 0: h_final = h0 was written
    const size_t smem = chunk_fwd_smem(d);
    auto k = simt_chunk_fwd<T, TS>;
    cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    trace_begin("chunk_fwd_simt", st);
    k<<<dim3(d.nc, d.H, d.B), kThreads, smem, st>>>(
        d, (const T *)p.x, (const T *)p.Bm, (const T *)p.Cm, (const T *)p.wr, (const T *)p.ww,
        p.dt, p.alpha, p.lam, p.tau, p.D, (const TS *)S_in, (T *)p.y);
    trace_end(st);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// N = 1 backward (the paper's layer shape).  The adjoint of the scalar recurrence per (mode, p),
// g_t = w_read_t C_t dy_t + rho_{t+1} g_{t+1}, is carried across chunks the way the forward
// carries the state: a reverse chunk-local pass gives each chunk's carry
// loc_c = rho_{c0} g^loc_{c0} (its own positions only) and its decay prod rho, a reverse serial
// combine turns them into the adjoint entering each chunk from the right (gamma_c, emitted in
// the dS_out layout) and dh0, and a chunk-parallel gradient kernel forms every gradient of the
// chunk from S_in and gamma in the pairwise chunked form (H = dY X^T over p, the per-mode pair
// sums with their own decays, and the S_in / gamma dot products over p).

// Reverse chunk-local pass: one thread per p of a 256-wide block (dy rows staged like x in the
// forward), the modes in registers; g walks the chunk from its last position to its first.
template <typename T, bool VEC, int KP>
__global__ void __launch_bounds__(kN1P) n1_rev_local(ScanDims d, const T *__restrict__ dy, const T *__restrict__ Cm,
                                                    const T *__restrict__ wr, const float *__restrict__ dt,
                                                    const float *__restrict__ alpha, const float *__restrict__ lam,
                                                    const float *__restrict__ tau, float *__restrict__ loc,
                                                    float *__restrict__ dec) {
    extern __shared__ __align__(16) unsigned char n1_smem[];
    const N1Smem L_(sizeof(T));
    float *e_s = reinterpret_cast<float *>(n1_smem + L_.e), *itau = reinterpret_cast<float *>(n1_smem + L_.itau);
    float *rho_s = reinterpret_cast<float *>(n1_smem + L_.rho), *wc_s = reinterpret_cast<float *>(n1_smem + L_.wc);
    float *kb_s = reinterpret_cast<float *>(n1_smem + L_.kb);
    T *y_s = reinterpret_cast<T *>(n1_smem + L_.x);
    const int K = d.K, P = d.P;
    const int npb = (P + kN1P - 1) / kN1P;
    const int c = blockIdx.x, h = blockIdx.y / npb, b = blockIdx.z, pb = blockIdx.y % npb;
    const int p0 = pb * kN1P, np = min(kN1P, P - p0), p = p0 + threadIdx.x;
    const size_t bh = size_t(b) * d.H + h;
    const int c0 = c * d.Q, n = min(d.Q, d.L - c0);
    n1_x_issue<T, VEC>(d, dy, b, h, c0, n, p0, np, y_s);
    if (threadIdx.x < K) itau[threadIdx.x] = 1.f / tau[h * K + threadIdx.x];
    const float log_cap = head_log_cap(tau, h, K);
    __syncthreads();
    // rho and (in the kb slot, unused here) kappa B; w_read C in the wc slot
    n1_chunk_coefs<T>(d, b, h, c0, n, log_cap, itau, Cm, Cm, wr, wr, dt, alpha, lam, e_s, rho_s, kb_s, wc_s);
    n1_x_wait<VEC>();
    if (pb == 0 && threadIdx.x < K) {
        float a = 1.f;
        for (int t = 0; t < n; ++t) a *= rho_s[t * K + threadIdx.x];
        dec[(bh * d.nc + c) * K + threadIdx.x] = a;
    }
    if (threadIdx.x >= np) return;
    // g = w_read C dy at the chunk's last position, then g = rho_{t+1} g + w_read C dy going left
    // (16-byte pieces of the coefficient rows when K is a multiple of 4, as in the forward)
    float g[KP];
#pragma unroll
    for (int m = 0; m < KP; ++m) g[m] = 0.f;
    if (n > 0) {
        const float dv = to_f(y_s[(n - 1) * kN1P + threadIdx.x]);
#pragma unroll
        for (int m = 0; m < KP; ++m)
            if (m < K) g[m] = wc_s[(n - 1) * K + m] * dv;
    }
#pragma unroll 4
    for (int t = n - 2; t >= 0; --t) {
        const float dv = to_f(y_s[t * kN1P + threadIdx.x]);
        if ((K & 3) == 0) {
            const float4 *r4 = reinterpret_cast<const float4 *>(rho_s + (t + 1) * K);
            const float4 *w4 = reinterpret_cast<const float4 *>(wc_s + t * K);
            const float2 dd = make_float2(dv, dv);
#pragma unroll
            for (int q = 0; q < KP / 4; ++q) {  // packed float32 pairs (the same IEEE operations)
                if (4 * q < K) {
                    const float4 r = r4[q], wv = w4[q];
                    const float2 a = __ffma2_rn(make_float2(r.x, r.y), make_float2(g[4 * q], g[4 * q + 1]),
                                                __fmul2_rn(make_float2(wv.x, wv.y), dd));
                    const float2 c2 = __ffma2_rn(make_float2(r.z, r.w), make_float2(g[4 * q + 2], g[4 * q + 3]),
                                                 __fmul2_rn(make_float2(wv.z, wv.w), dd));
                    g[4 * q] = a.x;
                    g[4 * q + 1] = a.y;
                    g[4 * q + 2] = c2.x;
                    g[4 * q + 3] = c2.y;
                }
            }
        } else {
#pragma unroll
            for (int m = 0; m < KP; ++m)
                if (m < K) g[m] = fmaf(rho_s[(t + 1) * K + m], g[m], wc_s[t * K + m] * dv);
        }
    }
#pragma unroll
    for (int m = 0; m < KP; ++m)
        if (m < K) loc[((bh * d.nc + c) * K + m) * P + p] = n > 0 ? rho_s[m] * g[m] : 0.f;
}

// Reverse serial combine: gamma of the last chunk is dh_final; going left, emit gamma_c (the
// adjoint entering chunk c from the right, in the dS_out layout), then
// gamma_{c-1} = decay_c gamma_c + loc_c; what leaves chunk 0 is dh0.
template <typename TS>
__global__ void __launch_bounds__(256) n1_combine_rev(ScanDims d, const float *__restrict__ loc,
                                                     const float *__restrict__ dec, const float *__restrict__ init,
                                                     TS *__restrict__ emit, float *__restrict__ fin) {
    constexpr int kBatch = 16;
    const size_t total = size_t(d.B) * d.H * d.K * d.P;
    const size_t idx = size_t(blockIdx.x) * blockDim.x + threadIdx.x;
    if (idx >= total) return;
    const int p = int(idx % d.P);
    const size_t bhm = idx / d.P;
    const int m = int(bhm % d.K);
    const size_t bh = bhm / d.K;
    float S = init ? init[idx] : 0.f;
    for (int c1 = d.nc - 1; c1 >= 0; c1 -= kBatch) {
        float lv[kBatch], dv[kBatch];
#pragma unroll
        for (int j = 0; j < kBatch; ++j) {
            const int c = c1 - j;
            lv[j] = c >= 0 ? loc[((bh * d.nc + c) * d.K + m) * d.P + p] : 0.f;
            dv[j] = c >= 0 ? dec[(bh * d.nc + c) * d.K + m] : 0.f;
        }
#pragma unroll
        for (int j = 0; j < kBatch; ++j) {
            const int c = c1 - j;
            if (c >= 0) {
                emit[((bh * d.nc + c) * d.K + m) * d.P + p] = from_f<TS>(S);
                S = fmaf(dv[j], S, lv[j]);
            }
        }
    }
    if (fin) fin[idx] = S;
}

constexpr int kN1BQ = 32;  // chunk of the N = 1 backward (shared-memory tiles [Q][P])
constexpr int kN1Timeout = 4;  // FRAC_ERR_TIMEOUT in the call's status word
// floats of the N1Arrays block (15 [Q][K] arrays and two [Q] arrays)
__host__ __device__ constexpr size_t n1_arrays_floats(int K) { return size_t(15) * kN1BQ * K + 2 * kN1BQ; }
constexpr int kGS = 36;    // row stride of its Gamma tile (rows read as 16-byte pieces)

struct N1BwdSmem {
    size_t E, Ef, e, cl, itau, red, cdot, dtq, qk, x, y, sin, gam, H, Gm, XR, total;
    int P;
    __host__ __device__ N1BwdSmem(int P_, int K, size_t esz) : P(P_) {
        E = 0;                                                   // double [Q]
        Ef = E + sizeof(double) * kN1BQ;                         // float2 [Q]: E as hi + lo
        e = Ef + sizeof(float) * 2 * kN1BQ;                      // float [Q]
        cl = e + sizeof(float) * kN1BQ;                          // float [Q]
        itau = cl + sizeof(float) * kN1BQ;                       // float [32]
        red = itau + sizeof(float) * 32;                         // float [64]
        cdot = red + sizeof(float) * 64;                         // float [32]
        dtq = cdot + sizeof(float) * 32;                         // float [32]: dtau sums per mode
        qk = dtq + sizeof(float) * 32;                           // float N1Arrays
        x = qk + sizeof(float) * n1_arrays_floats(K);            // T [Q][P]
        x = (x + 15) / 16 * 16;
        y = x + esz * kN1BQ * P;                                 // T [Q][P]
        y = (y + 15) / 16 * 16;
        sin = y + esz * kN1BQ * P;                               // float [K][P]
        gam = sin + sizeof(float) * K * P;                       // float [K][P]
        H = (gam + sizeof(float) * K * P + 15) / 16 * 16;         // float [Q][Q + 1]
        Gm = H + sizeof(float) * kN1BQ * (kN1BQ + 1);            // float [Q][kGS]
        XR = Gm + sizeof(float) * kN1BQ * kGS;                   // float [Q][Q + 1]
        total = XR + sizeof(float) * kN1BQ * (kN1BQ + 1);
    }
};

// The [Q][K] float arrays of the N = 1 gradient kernels (shared memory): per-(position, mode)
// coefficients, then the dot products over p and the pair sums.
struct N1Arrays {
    float *rho, *kap, *kb, *wc, *A, *u, *ww, *wr, *XG, *YS, *dwci, *dkbi;
    float *kbT, *wcT, *s;  // kappa B, w_read C and kappa B u, mode-major [K][Q]
    float *Bt, *Ct;        // [Q]
    __device__ N1Arrays(float *qk, int K) {
        const int QK = kN1BQ * K;
        rho = qk; kap = qk + QK; kb = qk + 2 * QK; wc = qk + 3 * QK; A = qk + 4 * QK; u = qk + 5 * QK;
        ww = qk + 6 * QK; wr = qk + 7 * QK; XG = qk + 8 * QK; YS = qk + 9 * QK; dwci = qk + 10 * QK;
        dkbi = qk + 11 * QK; kbT = qk + 12 * QK; wcT = qk + 13 * QK; s = qk + 14 * QK;
        Bt = qk + 15 * QK; Ct = Bt + kN1BQ;
    }
};

// Per-(position, mode) coefficients of one chunk: rho = exp(-e/tau), kappa = -expm1(-e/tau) w_write,
// kappa B, w_read C, A = exp(-E_t/tau) (entering state to position t), u = exp(-(E_end - E_t)/tau)
// (position t to the chunk's end) and s = kappa B u; zeros past the chunk's end.
template <typename T>
__device__ __forceinline__ void n1_bwd_coefs(const ScanDims &d, int b, int h, int g, int c0, int n, double Eend,
                                             const float *itau, const float *e_s, const double *E_s,
                                             const T *__restrict__ ww, const T *__restrict__ wr,
                                             const T *__restrict__ Bm, const T *__restrict__ Cm, const N1Arrays &a) {
    const int K = d.K;
    for (int idx = threadIdx.x; idx < kN1BQ * K; idx += blockDim.x) {
        const int t = idx / K, m = idx - t * K;
        float rho = 0.f, kap = 0.f, A = 0.f, u = 0.f, w_w = 0.f, w_r = 0.f, Bt = 0.f, Ct = 0.f;
        if (t < n) {
            const size_t wi = blh(d, b, c0 + t, h) * K + m;
            const size_t gi = (size_t(b) * d.L + c0 + t) * d.G + g;
            w_w = to_f(ww[wi]);
            w_r = to_f(wr[wi]);
            Bt = to_f(Bm[gi]);
            Ct = to_f(Cm[gi]);
            const float z = e_s[t] * itau[m];
            rho = expf(-z);
            kap = -expm1f(-z) * w_w;
            A = expf(-float(E_s[t]) * itau[m]);
            u = expf(-float(Eend - E_s[t]) * itau[m]);
        }
        a.rho[idx] = rho; a.kap[idx] = kap; a.kb[idx] = kap * Bt; a.wc[idx] = w_r * Ct;
        a.A[idx] = A; a.u[idx] = u; a.ww[idx] = w_w; a.wr[idx] = w_r;
        a.kbT[m * kN1BQ + t] = kap * Bt; a.wcT[m * kN1BQ + t] = w_r * Ct; a.s[m * kN1BQ + t] = kap * Bt * u;
        if (m == 0) {
            a.Bt[t] = Bt;
            a.Ct[t] = Ct;
        }
        a.XG[idx] = 0.f; a.YS[idx] = 0.f;
    }
}

// Sums NV (a power of two <= 32) values over the 32 lanes of a warp by halving exchanges: at
// offset o a lane keeps the half of its values picked by bit o of its lane index and adds its
// partner's copy of that half.  Returns the index of the total that v[0] then holds; lanes whose
// low 5 - log2(NV) bits are not all zero hold copies.
template <int NV>
__device__ __forceinline__ int warp_halving_sum(float (&v)[NV], int lane) {
    int cnt = NV, base = 0;
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
        if (cnt > 1) {
            const int half = cnt / 2;
            const bool up = (lane & o) != 0;
#pragma unroll
            for (int i = 0; i < NV / 2; ++i) {
                if (i < half) {
                    const float send = up ? v[i] : v[i + half];
                    const float keep = up ? v[i + half] : v[i];
                    v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
                }
            }
            if (up) base += half;
            cnt = half;
        } else {
            v[0] += __shfl_xor_sync(0xffffffffu, v[0], o);
        }
    }
    return base;
}

// Pair passes over k <= t.  Row pass, one warp per row t with the lanes on the columns k: the
// pair decays of every mode in registers (independent exponentials), Gamma_tk = sum_m w_read C_t
// kappa B_k exp(-(E_t - E_k)/tau_m) to put(t, k, .), Gamma' o H to XR, and the intra dw_read-like
// sums over k (a halving-exchange sum across the warp).  Column pass, one warp per column k with
// the lanes on the rows t: the intra dkappa B-like sums over t.  Every entry has one writer.
// exp(-x tau^-1) as 2^(-x tau^-1 log2 e) by the approximate hardware exp2 (relative error ~1e-6 over
// the arguments of the pair decays, inside the bf16 tolerance); FAST = false keeps expf
template <bool FAST>
__device__ __forceinline__ float pair_decay(float dE, float it) {
    if constexpr (FAST) {
        float y;
        asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(-dE * (it * 1.4426950408889634f)));
        return y;
    } else {
        return expf(-dE * it);
    }
}

template <int KP, bool FAST, typename PutGamma>
__device__ __forceinline__ void n1_pair_passes(int n, int K, const float *itau, const float2 *Ef_s,
                                               const N1Arrays &a, const float *H, float *XR, PutGamma put) {
    constexpr int Q1 = kN1BQ + 1;
    constexpr int kDup = 32 / KP - 1;  // lane bits holding copies after warp_halving_sum<KP>
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
    float it[KP];
#pragma unroll
    for (int m = 0; m < KP; ++m) it[m] = m < K ? itau[m] : 0.f;
    const float2 Elane = Ef_s[lane];
    for (int t = w; t < n; t += nw) {  // row pass
        const float2 Et = Ef_s[t];
        const bool ok = lane <= t;
        const float dE = (Et.x - Elane.x) + (Et.y - Elane.y);
        const float hv = ok ? H[t * Q1 + lane] : 0.f;
        float gam = 0.f, gamt = 0.f, dw[KP];
#pragma unroll
        for (int m = 0; m < KP; ++m) {
            float av = 0.f, kw = 0.f;
            if (m < K && ok) {
                kw = a.kbT[m * kN1BQ + lane] * pair_decay<FAST>(dE, it[m]);
                av = a.wc[t * K + m] * kw;
            }
            gam += av;
            gamt = fmaf(av, it[m], gamt);
            dw[m] = kw * hv;
        }
        if (ok) {
            put(t, lane, gam);
            XR[t * Q1 + lane] = gamt * hv;
        }
        const int m0 = warp_halving_sum<KP>(dw, lane);
        if ((lane & kDup) == 0 && m0 < K) a.dwci[t * K + m0] = dw[0];
    }
    for (int k = w; k < n; k += nw) {  // column pass
        const float2 Ek = Ef_s[k];
        const bool ok = lane >= k && lane < n;
        const float dE = (Elane.x - Ek.x) + (Elane.y - Ek.y);
        const float hv = ok ? H[lane * Q1 + k] : 0.f;
        float dk[KP];
#pragma unroll
        for (int m = 0; m < KP; ++m)
            dk[m] = (m < K && ok) ? a.wcT[m * kN1BQ + lane] * pair_decay<FAST>(dE, it[m]) * hv : 0.f;
        const int m0 = warp_halving_sum<KP>(dk, lane);
        if ((lane & kDup) == 0 && m0 < K) a.dkbi[k * K + m0] = dk[0];
    }
}

// Rectangle sums of Gamma' o H over pairs k < t <= t': each row of XR becomes its exclusive
// prefix (a warp scan per row), then rp_s[t] = sum over t' >= t of row t' at column t (a warp sum
// per column).  Ends with rp_s published.
__device__ __forceinline__ void n1_rect(int n, float *XR, float *rp_s) {
    constexpr int Q1 = kN1BQ + 1;
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
    for (int t = w; t < n; t += nw) {
        float incl = XR[t * Q1 + lane];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const float u = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += u;
        }
        const float excl = __shfl_up_sync(0xffffffffu, incl, 1);  // no cancellation of v
        XR[t * Q1 + lane] = lane > 0 ? excl : 0.f;
    }
    __syncthreads();
    for (int t = w; t < n; t += nw) {
        const float v = (lane >= t && lane < n) ? XR[lane * Q1 + t] : 0.f;
        const float sum = warp_sum(v);
        if (lane == 0) rp_s[t] = sum;
    }
    __syncthreads();
}

// Per-position gradients of one chunk, one thread per (position, mode) with 32 / KP positions per
// warp (the lanes of a position on consecutive modes).  a_t / b_k are the S_in / gamma terms of
// sum_m rho <g_t, S_{t-1}>_m / tau_m (suffix and exclusive prefix sums over the chunk, warp
// scans), c the <gamma, S_in> term, rp_s the pairs; then the mode-weight gradients per (t, m) and,
// summed over the position's lanes, dDelta, dalpha, dlambda, dB, dC and (when asked) the
// inter-chunk and per-position terms of dtau.  scratch: 96 floats no longer in use.
template <typename T, int KP>
__device__ __forceinline__ void n1_position_grads(
    const ScanDims &d, int b, int h, int g, int c0, int n, double Eend, const N1Arrays &a, const float *itau,
    const float *e_s, const double *E_s, const float *cl_s, const float *cdot, const float *rp_s, float *scratch,
    float *dtq, const float *__restrict__ dt, const float *__restrict__ alpha, const float *__restrict__ lam,
    T *__restrict__ dwr_o, T *__restrict__ dww_o, float *__restrict__ ddt, float *__restrict__ dalpha,
    float *__restrict__ dlam, float *__restrict__ dB_acc, float *__restrict__ dC_acc, float *__restrict__ dtau) {
    constexpr int RPW = 32 / KP;
    const int K = d.K, tid = threadIdx.x, w = tid >> 5, lane = tid & 31, nw = blockDim.x >> 5;
    const int m = lane % KP, sub = lane / KP;
    const bool mok = m < K;
    const float itm = mok ? itau[m] : 0.f;
    float *a_s = scratch, *b_s = scratch + 32, *R_s = scratch + 64;
    const int ngrp = (n + RPW - 1) / RPW;
    for (int gi = w; gi < ngrp; gi += nw) {
        const int t = gi * RPW + sub;
        float va = 0.f, vb = 0.f;
        if (t < n && mok) {
            const int q = t * K + m;
            va = a.wc[q] * a.A[q] * a.YS[q] * itm;
            vb = a.kb[q] * a.u[q] * a.XG[q] * itm;
        }
#pragma unroll
        for (int o = KP / 2; o >= 1; o >>= 1) {
            va += __shfl_xor_sync(0xffffffffu, va, o);
            vb += __shfl_xor_sync(0xffffffffu, vb, o);
        }
        if (m == 0 && t < n) {
            a_s[t] = va;
            b_s[t] = vb;
        }
    }
    __syncthreads();
    if (w == 0) {
        float cp = lane < K ? expf(-float(Eend) * itau[lane]) * itau[lane] * cdot[lane] : 0.f;
        cp = warp_sum(cp);
        const float av = lane < n ? a_s[lane] : 0.f, bv = lane < n ? b_s[lane] : 0.f;
        float suf = av, pre = bv;  // inclusive suffix sums of a, inclusive prefix sums of b
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const float us = __shfl_down_sync(0xffffffffu, suf, o);
            const float up = __shfl_up_sync(0xffffffffu, pre, o);
            if (lane + o < 32) suf += us;
            if (lane >= o) pre += up;
        }
        const float pre_x = __shfl_up_sync(0xffffffffu, pre, 1);  // exclusive prefix of b
        if (lane < n) R_s[lane] = suf + (lane > 0 ? pre_x : 0.f) + cp + rp_s[lane];
    }
    __syncthreads();
    for (int gi = w; gi < ngrp; gi += nw) {
        const int t = gi * RPW + sub;
        float de = 0.f, sB = 0.f, sC = 0.f;
        const size_t i = t < n ? blh(d, b, c0 + t, h) : 0;
        if (t < n && mok) {
            const int q = t * K + m;
            const float dkb = a.u[q] * a.XG[q] + a.dkbi[q];  // d(kappa B)
            const float dwc = a.A[q] * a.YS[q] + a.dwci[q];  // d(w_read C)
            const float dk = dkb * a.Bt[t];                  // d kappa
            de = dk * a.rho[q] * a.ww[q] * itm;
            dwr_o[i * K + m] = from_f<T>(dwc * a.Ct[t]);
            dww_o[i * K + m] = from_f<T>(dk * (-expm1f(-e_s[t] * itm)));
            sB = dkb * a.kap[q];
            sC = dwc * a.wr[q];
            if (dtau) {
                const double Et = E_s[t];
                const double tq = Et * double(a.wc[q] * a.A[q] * a.YS[q]) +
                                  (Eend - Et) * double(a.kb[q] * a.u[q] * a.XG[q]) -
                                  double(e_s[t]) * double(dk) * double(a.rho[q]) * double(a.ww[q]);
                atomicAdd(&dtq[m], float(tq));
            }
        }
#pragma unroll
        for (int o = KP / 2; o >= 1; o >>= 1) {
            de += __shfl_xor_sync(0xffffffffu, de, o);
            sB += __shfl_xor_sync(0xffffffffu, sB, o);
            sC += __shfl_xor_sync(0xffffffffu, sC, o);
        }
        if (m == 0 && t < n) {
            de -= R_s[t];
            const size_t gq = (size_t(b) * d.L + c0 + t) * d.G + g;
            atomicAdd(&dB_acc[gq], sB);
            atomicAdd(&dC_acc[gq], sC);
            const float e = e_s[t];
            const bool cl = cl_s[t] != 0.f;
            const float al = alpha[i], lm = lam[i], dtv = dt[i];
            const float ge = cl ? 0.f : de * e;
            ddt[i] = ge / dtv;
            dlam[i] = ge / (al * lm);
            dalpha[i] = -ge * logf(lm) / (al * al);
        }
    }
    if (dtau) {
        __syncthreads();
        if (tid < K) {
            const float it = itau[tid];
            const float chunk_term = float(Eend) * expf(-float(Eend) * it) * cdot[tid];
            atomicAdd(&dtau[h * K + tid], (dtq[tid] + chunk_term) * it * it);
        }
    }
}

// Gradients of one chunk of one head (one CTA, 256 threads; Q <= 32, all of P).
template <typename T, typename TS, bool VEC, int KP>
__global__ void __launch_bounds__(kThreads) n1_chunk_bwd(
    ScanDims d, const T *__restrict__ x, const T *__restrict__ Bm, const T *__restrict__ Cm,
    const T *__restrict__ wr, const T *__restrict__ ww, const T *__restrict__ dy,
    const float *__restrict__ dt, const float *__restrict__ alpha, const float *__restrict__ lam,
    const float *__restrict__ tau, const float *__restrict__ Dv, const TS *__restrict__ S_in,
    const TS *__restrict__ dS_out, T *__restrict__ dx, T *__restrict__ dwr_o, T *__restrict__ dww_o,
    float *__restrict__ ddt, float *__restrict__ dalpha, float *__restrict__ dlam, float *__restrict__ dD,
    float *__restrict__ dB_acc, float *__restrict__ dC_acc, float *__restrict__ dtau) {
    extern __shared__ __align__(16) unsigned char sm_raw[];
    const int K = d.K, P = d.P, Q = d.Q;
    const N1BwdSmem L_(P, K, sizeof(T));
    double *E_s = reinterpret_cast<double *>(sm_raw + L_.E);
    float2 *Ef_s = reinterpret_cast<float2 *>(sm_raw + L_.Ef);
    float *e_s = reinterpret_cast<float *>(sm_raw + L_.e), *cl_s = reinterpret_cast<float *>(sm_raw + L_.cl);
    float *itau = reinterpret_cast<float *>(sm_raw + L_.itau), *red = reinterpret_cast<float *>(sm_raw + L_.red);
    float *cdot = reinterpret_cast<float *>(sm_raw + L_.cdot);
    float *dtq = reinterpret_cast<float *>(sm_raw + L_.dtq);
    float *qk = reinterpret_cast<float *>(sm_raw + L_.qk);
    const N1Arrays a(qk, K);
    float *XG = a.XG, *YS = a.YS, *s_s = a.s;
    T *xs = reinterpret_cast<T *>(sm_raw + L_.x), *dys = reinterpret_cast<T *>(sm_raw + L_.y);
    float *Sin = reinterpret_cast<float *>(sm_raw + L_.sin), *Gam = reinterpret_cast<float *>(sm_raw + L_.gam);
    float *H = reinterpret_cast<float *>(sm_raw + L_.H), *Gm = reinterpret_cast<float *>(sm_raw + L_.Gm);
    float *XR = reinterpret_cast<float *>(sm_raw + L_.XR);
    constexpr int Q1 = kN1BQ + 1;
    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
    const int g = h / (d.H / d.G);
    const int c0 = c * Q, n = min(Q, d.L - c0);
    const size_t bh = size_t(b) * d.H + h;

    // ---- P0: tiles, states, rates and per-(position, mode) coefficients
    if constexpr (VEC) {
        constexpr int PER = 16 / sizeof(T);
        const int pieces = P / PER;
        for (int idx = tid; idx < n * pieces; idx += blockDim.x) {
            const int t = idx / pieces, q = idx - t * pieces;
            const size_t src = blh(d, b, c0 + t, h) * P + q * PER;
            const uint32_t dx_ = static_cast<uint32_t>(__cvta_generic_to_shared(xs + t * P + q * PER));
            const uint32_t dy_ = static_cast<uint32_t>(__cvta_generic_to_shared(dys + t * P + q * PER));
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dx_), "l"(x + src) : "memory");
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dy_), "l"(dy + src) : "memory");
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    } else {
        for (int idx = tid; idx < n * P; idx += blockDim.x) {
            const int t = idx / P, q = idx - t * P;
            xs[t * P + q] = x[blh(d, b, c0 + t, h) * P + q];
            dys[t * P + q] = dy[blh(d, b, c0 + t, h) * P + q];
        }
    }
    for (int idx = tid; idx < (kN1BQ - n) * P; idx += blockDim.x) {  // rows past a ragged end
        const int t = n + idx / P, q = idx % P;
        xs[t * P + q] = from_f<T>(0.f);
        dys[t * P + q] = from_f<T>(0.f);
    }
    const size_t sbase = (bh * d.nc + c) * size_t(K) * P;
    for (int idx = tid; idx < K * P; idx += blockDim.x) {
        Sin[idx] = to_f(S_in[sbase + idx]);
        Gam[idx] = to_f(dS_out[sbase + idx]);
    }
    if (tid < K) itau[tid] = 1.f / tau[h * K + tid];
    if (tid < 64) red[tid] = 0.f;
    if (tid < 32) cdot[tid] = dtq[tid] = 0.f;
    const float log_cap = head_log_cap(tau, h, K);
    chunk_rates(d, b, h, c0, n, log_cap, dt, alpha, lam, e_s, E_s, cl_s);
    __syncthreads();
    const double Eend = E_s[n - 1];
    n1_bwd_coefs<T>(d, b, h, g, c0, n, Eend, itau, e_s, E_s, ww, wr, Bm, Cm, a);
    for (int idx = tid; idx < kN1BQ * Q1; idx += blockDim.x) H[idx] = 0.f;
    if (tid < kN1BQ) {  // E as an unevaluated float pair: pair differences without FP64
        const double Ev = tid < n ? E_s[tid] : 0.0;
        const float hi = float(Ev);
        Ef_s[tid] = make_float2(hi, float(Ev - double(hi)));
    }
    if constexpr (VEC) asm volatile("cp.async.wait_all;" ::: "memory");
    __syncthreads();

    // ---- P1: H = dY X^T and the dot products over p of x with gamma, dy with S_in and gamma with
    // S_in: one warp per 4 x 4 output tile, the lanes on consecutive p (no bank conflicts), the
    // 16 partial sums reduced across the warp by halving exchanges (lane l ends with one value)
    {
        const int w = tid >> 5, lane = tid & 31, nw = blockDim.x >> 5;
        const int qt = Q / 4, mt = (K + 3) / 4;
        const int nH = qt * (qt + 1) / 2;  // tiles on or below the diagonal
        for (int item = w; item < nH + qt * mt; item += nw) {
            float v[16], v2[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] = v2[i] = 0.f;
            float vc[4] = {0.f, 0.f, 0.f, 0.f};
            int r0, c0t;
            const bool isH = item < nH;
            if (isH) {  // item -> (row tile, column tile <= row tile)
                int rt = 0, rem = item;
                while (rem > rt) rem -= ++rt;
                r0 = 4 * rt;
                c0t = 4 * rem;
                for (int q = lane; q < P; q += 32) {
                    float dv[4], xv[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        dv[i] = to_f(dys[(r0 + i) * P + q]);
                        xv[i] = to_f(xs[(c0t + i) * P + q]);
                    }
#pragma unroll
                    for (int i = 0; i < 4; ++i)
#pragma unroll
                        for (int j = 0; j < 4; ++j) v[4 * i + j] = fmaf(dv[i], xv[j], v[4 * i + j]);
                }
            } else {
                const int it = item - nH;
                r0 = 4 * (it / mt);
                c0t = 4 * (it % mt);  // first mode
                for (int q = lane; q < P; q += 32) {
                    float xv[4], dv[4], gv[4], sv[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        xv[i] = to_f(xs[(r0 + i) * P + q]);
                        dv[i] = to_f(dys[(r0 + i) * P + q]);
                        gv[i] = c0t + i < K ? Gam[(c0t + i) * P + q] : 0.f;
                        sv[i] = c0t + i < K ? Sin[(c0t + i) * P + q] : 0.f;
                    }
#pragma unroll
                    for (int i = 0; i < 4; ++i)
#pragma unroll
                        for (int j = 0; j < 4; ++j) {
                            v[4 * i + j] = fmaf(xv[i], gv[j], v[4 * i + j]);
                            v2[4 * i + j] = fmaf(dv[i], sv[j], v2[4 * i + j]);
                        }
                    if (r0 == 0)
#pragma unroll
                        for (int j = 0; j < 4; ++j) vc[j] = fmaf(gv[j], sv[j], vc[j]);
                }
            }
            // halving exchanges: after offsets 16, 8, 4, 2 lane l holds value
            // 8 b4 + 4 b3 + 2 b2 + b1 (bk = bit k of l) summed over 16 lanes; offset 1 completes it
            auto reduce16 = [&](float *a) {
#pragma unroll
                for (int o = 16, cnt = 8; o >= 2; o >>= 1, cnt >>= 1) {
                    const bool up = (lane & o) != 0;
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        if (i < cnt) {
                            const float send = up ? a[i] : a[i + cnt];
                            const float keep = up ? a[i + cnt] : a[i];
                            a[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
                        }
                    }
                }
                a[0] += __shfl_xor_sync(0xffffffffu, a[0], 1);
            };
            const int vi = 8 * ((lane >> 4) & 1) + 4 * ((lane >> 3) & 1) + 2 * ((lane >> 2) & 1) + ((lane >> 1) & 1);
            const int ri = vi >> 2, ci = vi & 3;
            reduce16(v);
            if (isH) {
                if ((lane & 1) == 0) H[(r0 + ri) * Q1 + c0t + ci] = v[0];
            } else {
                reduce16(v2);
                if ((lane & 1) == 0 && c0t + ci < K) {
                    XG[(r0 + ri) * K + c0t + ci] = v[0];
                    YS[(r0 + ri) * K + c0t + ci] = v2[0];
                }
                if (r0 == 0) {
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const float sc = warp_sum(vc[j]);
                        if (lane == 0 && c0t + j < K) cdot[c0t + j] = sc;
                    }
                }
            }
        }
    }
    __syncthreads();

    // ---- P2: pair passes (n1_pair_passes); Gamma into the row-major Gm tile
    for (int idx = tid; idx < kN1BQ * kGS; idx += blockDim.x) Gm[idx] = 0.f;
    for (int idx = tid; idx < kN1BQ * Q1; idx += blockDim.x) XR[idx] = 0.f;
    __syncthreads();
    n1_pair_passes<KP, false>(n, K, itau, Ef_s, a, H, XR, [&](int t, int k, float v) { Gm[t * kGS + k] = v; });
    __syncthreads();

    // ---- P3: rectangle sums of Gamma' o H over pairs k < t <= t' (row prefix, column suffix)
    float *rp_s = red + 32;  // [Q <= 32] (block_sum below uses red[0 .. 8))
    n1_rect(n, XR, rp_s);

    // ---- P4: dx[k][p] = sum_m s_{k,m} gamma_m[p] + sum_{t>=k} Gamma[t][k] dy_t[p] + D dy_k[p]
    // (one thread per p).  Gamma is zero above the diagonal and on rows past the chunk's end, so
    // every row adds to all 32 accumulators, read as 16-byte broadcast pieces.
    const float Dh = Dv[h];
    float ddv = 0.f;  // sum dy x for dD
    for (int q = tid; q < P; q += blockDim.x) {
        float acc[kN1BQ];
#pragma unroll
        for (int k = 0; k < kN1BQ; ++k) acc[k] = 0.f;
#pragma unroll 1
        for (int t = 0; t < n; ++t) {
            const float dv = to_f(dys[t * P + q]);
            ddv = fmaf(dv, to_f(xs[t * P + q]), ddv);
            const float4 *g4 = reinterpret_cast<const float4 *>(Gm + t * kGS);
#pragma unroll
            for (int k4 = 0; k4 < kN1BQ / 4; ++k4) {
                const float4 gv = g4[k4];
                acc[4 * k4] = fmaf(gv.x, dv, acc[4 * k4]);
                acc[4 * k4 + 1] = fmaf(gv.y, dv, acc[4 * k4 + 1]);
                acc[4 * k4 + 2] = fmaf(gv.z, dv, acc[4 * k4 + 2]);
                acc[4 * k4 + 3] = fmaf(gv.w, dv, acc[4 * k4 + 3]);
            }
        }
#pragma unroll 1
        for (int m = 0; m < K; ++m) {
            const float gv = Gam[m * P + q];
            const float4 *s4 = reinterpret_cast<const float4 *>(s_s + m * kN1BQ);
#pragma unroll
            for (int k4 = 0; k4 < kN1BQ / 4; ++k4) {
                const float4 sv = s4[k4];
                acc[4 * k4] = fmaf(sv.x, gv, acc[4 * k4]);
                acc[4 * k4 + 1] = fmaf(sv.y, gv, acc[4 * k4 + 1]);
                acc[4 * k4 + 2] = fmaf(sv.z, gv, acc[4 * k4 + 2]);
                acc[4 * k4 + 3] = fmaf(sv.w, gv, acc[4 * k4 + 3]);
            }
        }
#pragma unroll
        for (int k = 0; k < kN1BQ; ++k)
            if (k < n) dx[blh(d, b, c0 + k, h) * P + q] = from_f<T>(fmaf(Dh, to_f(dys[k * P + q]), acc[k]));
    }
    ddv = block_sum(ddv, red);  // contains __syncthreads (also publishes rp_s)
    if (tid == 0) atomicAdd(&dD[h], ddv);

    // ---- P5: per-position scalars (XR is free now)
    n1_position_grads<T, KP>(d, b, h, g, c0, n, Eend, a, itau, e_s, E_s, cl_s, cdot, rp_s, XR, dtq, dt, alpha, lam,
                         dwr_o, dww_o, ddt, dalpha, dlam, dB_acc, dC_acc, dtau);
}

// ----------------------------------------------------------------------------------------------
// Tensor-core variant of the N = 1 gradient kernel (bf16 inputs and states, P a multiple of 128,
// chunk 32).  The contractions over p and over positions run on tcgen05:
//   P1: one M = 128 chain over K = p of the rows [dy (32) | x (32) | gamma (KS) | S_in (KS)] (A,
//       from row 0) against the rows [x | gamma | S_in] (B, from row 32), K-major, gives in one
//       accumulator H = dY X^T, YS = dY S_in^T, XG = X gamma^T and diag(gamma S_in^T); every
//       product is of two bf16 values, so only the order of the fp32 sums differs.
//   P4: dx^T = [dY ; gamma]^T [Gamma ; s^T] per 128 p: A is the same tiles read MN-major (M = p,
//       K = position or mode), B the Gamma and s = kappa B u coefficients as bf16 hi + lo pairs
//       (K doubled), so the fp32 coefficients keep ~16 mantissa bits.
// The tiles arrive by TMA as 128-byte-swizzled 64-column panels of 64 + 2 KS rows (KS = 16 or 32
// rows for the modes); the phases between stay on the CUDA cores (the shared functions above).
struct N1BwdTcSmem {
    size_t pan, bimg, E, Ef, e, cl, itau, red, cdot, dtq, qk, H, XR, bars, total;
    uint32_t panel, bimg_rows;
    int KS;
    __host__ __device__ N1BwdTcSmem(int P, int K) {
        KS = K <= 16 ? 16 : 32;
        panel = uint32_t(64 + 2 * KS) * 128;                       // bytes of one 64-column panel
        pan = 0;                                                   // [P / 64] panels (1024-aligned)
        bimg = pan + size_t(P / 64) * panel;                       // B of P4: [2 (32 + KS)][128 B]
        bimg_rows = uint32_t(2 * (32 + KS));
        E = bimg + size_t(bimg_rows) * 128;                        // double [Q]
        Ef = E + sizeof(double) * kN1BQ;                           // float2 [Q]
        e = Ef + sizeof(float) * 2 * kN1BQ;                        // float [Q]
        cl = e + sizeof(float) * kN1BQ;                            // float [Q]
        itau = cl + sizeof(float) * kN1BQ;                         // float [32]
        red = itau + sizeof(float) * 32;                           // float [64]
        cdot = red + sizeof(float) * 64;                           // float [32]
        dtq = cdot + sizeof(float) * 32;                           // float [32]
        qk = dtq + sizeof(float) * 32;                             // float N1Arrays
        H = qk + sizeof(float) * n1_arrays_floats(K);              // float [Q][Q + 1]
        XR = H + sizeof(float) * kN1BQ * (kN1BQ + 1);              // float [Q][Q + 1]
        bars = (XR + sizeof(float) * kN1BQ * (kN1BQ + 1) + 7) / 8 * 8;  // 3 mbarriers, TMEM slot
        total = bars + 32 + 1024;                                  // + slack to align the base
    }
};
// TMEM columns of the variant: P1's accumulator (32 + 2 KS) and P4's (64 per 128 p), reused.
__host__ __device__ inline uint32_t n1_tc_tmem_cols(int P, int K) {
    const uint32_t need = uint32_t(std::max(32 + 2 * (K <= 16 ? 16 : 32), P / 2));
    uint32_t c = 32;
    while (c < need) c <<= 1;
    return c;
}

__device__ __forceinline__ void st_bf16_pair(unsigned char *img, uint32_t row_hi, uint32_t row_lo, uint32_t col,
                                             float v) {
    const __nv_bfloat16 hi = __float2bfloat16_rn(v);
    const __nv_bfloat16 lo = __float2bfloat16_rn(v - __bfloat162float(hi));
    *reinterpret_cast<__nv_bfloat16 *>(img + tc::sw128_offset(row_hi, col)) = hi;
    *reinterpret_cast<__nv_bfloat16 *>(img + tc::sw128_offset(row_lo, col)) = lo;
}

template <int KP>
__global__ void __launch_bounds__(kThreads) n1_chunk_bwd_tc(
    const __grid_constant__ CUtensorMap mapX, const __grid_constant__ CUtensorMap mapDY,
    const __grid_constant__ CUtensorMap mapS, const __grid_constant__ CUtensorMap mapG, ScanDims d,
    const __nv_bfloat16 *__restrict__ Bm, const __nv_bfloat16 *__restrict__ Cm,
    const __nv_bfloat16 *__restrict__ wr, const __nv_bfloat16 *__restrict__ ww, const float *__restrict__ dt,
    const float *__restrict__ alpha, const float *__restrict__ lam, const float *__restrict__ tau,
    const float *__restrict__ Dv, __nv_bfloat16 *__restrict__ dx, __nv_bfloat16 *__restrict__ dwr_o,
    __nv_bfloat16 *__restrict__ dww_o, float *__restrict__ ddt, float *__restrict__ dalpha,
    float *__restrict__ dlam, float *__restrict__ dD, float *__restrict__ dB_acc, float *__restrict__ dC_acc,
    float *__restrict__ dtau, int *__restrict__ err, uint32_t tmem_cols) {
    using namespace tc;
    using bf16 = __nv_bfloat16;
    constexpr int KS = KP <= 16 ? 16 : 32;
    constexpr int N1 = 32 + 2 * KS;
    constexpr int Q1 = kN1BQ + 1;
    extern __shared__ __align__(1024) unsigned char sm_raw0[];
    unsigned char *sm = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(sm_raw0) + 1023) &
                                                          ~uintptr_t(1023));
    const int K = d.K, P = d.P, Q = d.Q;
    const N1BwdTcSmem L_(P, K);
    double *E_s = reinterpret_cast<double *>(sm + L_.E);
    float2 *Ef_s = reinterpret_cast<float2 *>(sm + L_.Ef);
    float *e_s = reinterpret_cast<float *>(sm + L_.e), *cl_s = reinterpret_cast<float *>(sm + L_.cl);
    float *itau = reinterpret_cast<float *>(sm + L_.itau), *red = reinterpret_cast<float *>(sm + L_.red);
    float *cdot = reinterpret_cast<float *>(sm + L_.cdot), *dtq = reinterpret_cast<float *>(sm + L_.dtq);
    const N1Arrays a(reinterpret_cast<float *>(sm + L_.qk), K);
    float *H = reinterpret_cast<float *>(sm + L_.H), *XR = reinterpret_cast<float *>(sm + L_.XR);
    uint64_t *bars = reinterpret_cast<uint64_t *>(sm + L_.bars);  // copies in, P1 done, P4 done
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bars + 3);
    unsigned char *img = sm + L_.bimg;
    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z, tid = threadIdx.x, w = tid >> 5, lane = tid & 31;
    const int g = h / (d.H / d.G);
    const int c0 = c * Q, n = min(Q, d.L - c0);
    const size_t bh = size_t(b) * d.H + h;
    const int NP = P / 64;
    const uint32_t pan_a = smem_u32(sm + L_.pan), img_a = smem_u32(img);

    // ---- P0: barriers, TMEM, the tile copies, rates and coefficients
    if (tid == 0) {
        for (int i = 0; i < 3; ++i) mbar_init(&bars[i], 1);
        fence_barrier_init();
    }
    if (w == 0) tmem_alloc_once(tslot, tmem_cols);
    for (uint32_t i = tid; i < L_.bimg_rows * 8; i += blockDim.x)
        reinterpret_cast<uint4 *>(img)[i] = make_uint4(0u, 0u, 0u, 0u);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    bool issued1 = false, issued2 = false;  // (thread 0) MMA groups committed
    if (tid == 0) {
        mbar_arrive_expect_tx(&bars[0], uint32_t(NP) * L_.panel);
        const int sc = int(bh * d.nc + c);
        for (int j = 0; j < NP; ++j) {
            unsigned char *pj = sm + L_.pan + size_t(j) * L_.panel;
            tma_load_3d(pj, &mapDY, &bars[0], h * P + 64 * j, c0, b);
            tma_load_3d(pj + 32 * 128, &mapX, &bars[0], h * P + 64 * j, c0, b);
            tma_load_3d(pj + 64 * 128, &mapG, &bars[0], 64 * j, 0, sc);
            tma_load_3d(pj + (64 + KS) * 128, &mapS, &bars[0], 64 * j, 0, sc);
        }
    }
    if (tid < K) itau[tid] = 1.f / tau[h * K + tid];
    if (tid < 64) red[tid] = 0.f;
    if (tid < 32) cdot[tid] = dtq[tid] = 0.f;
    const float log_cap = head_log_cap(tau, h, K);
    chunk_rates(d, b, h, c0, n, log_cap, dt, alpha, lam, e_s, E_s, cl_s);
    __syncthreads();
    const double Eend = E_s[n - 1];
    n1_bwd_coefs<bf16>(d, b, h, g, c0, n, Eend, itau, e_s, E_s, ww, wr, Bm, Cm, a);
    for (int idx = tid; idx < kN1BQ * Q1; idx += blockDim.x) XR[idx] = 0.f;
    if (tid < kN1BQ) {
        const double Ev = tid < n ? E_s[tid] : 0.0;
        const float hi = float(Ev);
        Ef_s[tid] = make_float2(hi, float(Ev - double(hi)));
    }

    // ---- P1 on the tensor cores
    int bad = !mbar_wait(&bars[0], 0);
    bad = __syncthreads_or(bad);
    if (!bad && tid == 0) {
        tc_fence_after();
        constexpr uint32_t id1 = idesc_bf16(128, N1, false, false);
        for (int j = 0; j < NP; ++j)
            for (int kk = 0; kk < 4; ++kk) {
                const uint32_t a0 = pan_a + uint32_t(j) * L_.panel + kk * 32;
                mma_bf16(tmem, desc_sw128(a0, 16, 1024), desc_sw128(a0 + 32 * 128, 16, 1024), id1, (j | kk) != 0);
            }
        mma_commit(&bars[1]);
        issued1 = true;
    }
    if (!bad) bad = !mbar_wait(&bars[1], 0);
    bad = __syncthreads_or(bad);
    if (!bad) {
        tc_fence_after();
        if (w == 0) {  // lanes = dy rows t: H row t (columns 0..31), YS row t (columns 32 + KS ..)
            float hv[32], ys[KS];
            tmem_ld32(tmem, hv);
            if constexpr (KS == 16) tmem_ld16(tmem + 32 + KS, ys);
            else tmem_ld32(tmem + 32 + KS, ys);
            tmem_ld_wait();
            float dd = 0.f;
#pragma unroll
            for (int k = 0; k < 32; ++k) {
                H[lane * Q1 + k] = hv[k];
                if (k == lane && lane < n) dd = hv[k];  // sum_p dy x of row t (for dD)
            }
#pragma unroll
            for (int m = 0; m < KS; ++m)
                if (m < K) a.YS[lane * K + m] = ys[m];
            dd = warp_sum(dd);
            if (lane == 0) atomicAdd(&dD[h], dd);
        } else if (w == 1) {  // lanes = x rows t: XG row t (columns 32 ..)
            float xg[KS];
            if constexpr (KS == 16) tmem_ld16(tmem + (32u << 16) + 32, xg);
            else tmem_ld32(tmem + (32u << 16) + 32, xg);
            tmem_ld_wait();
#pragma unroll
            for (int m = 0; m < KS; ++m)
                if (m < K) a.XG[lane * K + m] = xg[m];
        } else if (w == 2) {  // lanes = gamma rows m: <gamma_m, S_in,m> on the diagonal
            float cv[KS];
            if constexpr (KS == 16) tmem_ld16(tmem + (64u << 16) + 32 + KS, cv);
            else tmem_ld32(tmem + (64u << 16) + 32 + KS, cv);
            tmem_ld_wait();
            float v = 0.f;
#pragma unroll
            for (int m = 0; m < KS; ++m)
                if (m == lane) v = cv[m];
            if (lane < K) cdot[lane] = v;
        }
    }
    __syncthreads();

    // ---- P2: pair passes; Gamma (hi, lo) into rows t and 32 + KS + t of P4's B, column k, and
    // s = kappa B u into rows 32 + m and 64 + KS + m
    if (!bad) {
        n1_pair_passes<KP, true>(n, K, itau, Ef_s, a, H, XR, [&](int t, int k, float v) {
            st_bf16_pair(img, uint32_t(t), uint32_t(32 + KS + t), uint32_t(k), v);
        });
        for (int idx = tid; idx < K * kN1BQ; idx += blockDim.x) {
            const int m = idx / kN1BQ, k = idx - m * kN1BQ;
            st_bf16_pair(img, uint32_t(32 + m), uint32_t(64 + KS + m), uint32_t(k), a.s[idx]);
        }
        fence_async_smem();
    }
    tc_fence_before();
    __syncthreads();

    // ---- P4 on the tensor cores (issued now, read after P3 and P5)
    if (!bad && tid == 0) {
        tc_fence_after();
        constexpr uint32_t id4 = idesc_bf16(128, 64, true, true);
        constexpr int half = 2 + KS / 16;  // K steps of 16 rows per (hi or lo) half
        for (int i = 0; i < NP / 2; ++i)
            for (int st = 0; st < 2 * half; ++st) {
                const int sh = st % half;
                const int ra = sh < 2 ? 16 * sh : 64 + 16 * (sh - 2);  // dy rows, then gamma rows
                const uint32_t ad = pan_a + uint32_t(2 * i) * L_.panel + uint32_t(ra) * 128;
                const uint32_t bd = img_a + uint32_t(st) * 16 * 128;
                mma_bf16(tmem + 64 * i, desc_sw128(ad, L_.panel, 1024), desc_sw128(bd, L_.bimg_rows * 128, 1024),
                         id4, st > 0);
            }
        mma_commit(&bars[2]);
        issued2 = true;
    }

    // ---- P3 and P5 on the CUDA cores meanwhile
    float *rp_s = red + 32;
    if (!bad) {
        n1_rect(n, XR, rp_s);
        n1_position_grads<bf16, KP>(d, b, h, g, c0, n, Eend, a, itau, e_s, E_s, cl_s, cdot, rp_s, XR, dtq, dt, alpha,
                                lam, dwr_o, dww_o, ddt, dalpha, dlam, dB_acc, dC_acc, dtau);
    }

    // ---- P4 epilogue: dx[k][p] = (dx^T)[p][k] + D dy[k][p], one thread per p
    if (!bad) bad = !mbar_wait(&bars[2], 0);
    bad = __syncthreads_or(bad);
    if (!bad) {
        tc_fence_after();
        const float Dh = Dv[h];
        for (int i = w / 4; i < NP / 2; i += 2) {
            const int p = 128 * i + 32 * (w & 3) + lane;
            float acc[32];
            tmem_ld32(tmem + (uint32_t(32 * (w & 3)) << 16) + 64 * i, acc);
            tmem_ld_wait();
            const unsigned char *pp = sm + L_.pan + size_t(p >> 6) * L_.panel;
#pragma unroll
            for (int k = 0; k < kN1BQ; ++k) {
                if (k < n) {
                    const float dyv = __bfloat162float(*reinterpret_cast<const bf16 *>(pp + sw128_offset(k, p & 63)));
                    dx[blh(d, b, c0 + k, h) * P + p] = __float2bfloat16_rn(fmaf(Dh, dyv, acc[k]));
                }
            }
        }
    }
    if (bad && tid == 0) {  // a wait gave up: record it, let copies and MMAs in flight finish
        atomicExch(err, kN1Timeout);
        mbar_wait(&bars[0], 0);
        if (issued1) mbar_wait(&bars[1], 0);
        if (issued2) mbar_wait(&bars[2], 0);
    }
    tc_fence_before();
    __syncthreads();
    if (w == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, tmem_cols);
    }
}

bool n1_bwd_fits(const ScanDims &d, size_t esz) {
    return d.N == 1 && d.Q <= kN1BQ && d.K <= 32 && N1BwdSmem(d.P, d.K, esz).total <= 227 * 1024 &&
           size_t(d.H) * ((d.P + kN1P - 1) / kN1P) <= 65535;
}

// Whether the tensor-core variant of the N = 1 gradient kernel takes a bf16 call: P a multiple of
// 128 up to 512, chunk 32, x, dy and the per-chunk states 16-byte aligned, and its shared memory
// within the per-CTA limit.
bool n1_bwd_tc_ok(const ScanDims &d, const ScanPtrs &p, const void *S_in, const void *dS_out) {
    auto al16 = [](const void *q) { return (reinterpret_cast<uintptr_t>(q) & 15u) == 0; };
    return d.N == 1 && d.Q == kN1BQ && d.P % 128 == 0 && d.P <= 512 && d.K <= 32 && al16(p.x) && al16(p.dy) &&
           al16(S_in) && al16(dS_out) && N1BwdTcSmem(d.P, d.K).total <= 227 * 1024;
}

// Launches n1_chunk_bwd_tc; *launched stays false (and nothing is enqueued) when a tensor map
// cannot be encoded, so that the caller runs the CUDA-core kernel instead.
cudaError_t launch_n1_bwd_tc(const ScanDims &d, const ScanPtrs &p, void *S_in, void *dS_out, float *dB_acc,
                             float *dC_acc, int *err, cudaStream_t st, bool *launched) {
    using bf = __nv_bfloat16;
    *launched = false;
    const int KS = d.K <= 16 ? 16 : 32;
    const uint64_t HP = uint64_t(d.H) * d.P;
    const uint64_t chunks = uint64_t(d.B) * d.H * d.nc;
    CUtensorMap mapX, mapDY, mapS, mapG;
    if (!tc_make_map3(&mapX, p.x, HP, d.L, d.B, HP * 2, uint64_t(d.L) * HP * 2, 64, kN1BQ, 1) ||
        !tc_make_map3(&mapDY, p.dy, HP, d.L, d.B, HP * 2, uint64_t(d.L) * HP * 2, 64, kN1BQ, 1) ||
        !tc_make_map3(&mapS, S_in, d.P, d.K, chunks, uint64_t(d.P) * 2, uint64_t(d.K) * d.P * 2, 64, KS, 1) ||
        !tc_make_map3(&mapG, dS_out, d.P, d.K, chunks, uint64_t(d.P) * 2, uint64_t(d.K) * d.P * 2, 64, KS, 1))
        return cudaSuccess;
    const size_t smem = N1BwdTcSmem(d.P, d.K).total;
    const uint32_t cols = n1_tc_tmem_cols(d.P, d.K);
    const int KP = d.K <= 4 ? 4 : d.K <= 8 ? 8 : d.K <= 16 ? 16 : 32;
    auto k = KP == 4 ? n1_chunk_bwd_tc<4> : KP == 8 ? n1_chunk_bwd_tc<8> : KP == 16 ? n1_chunk_bwd_tc<16>
                                                                                  : n1_chunk_bwd_tc<32>;
    cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    trace_begin("chunk_bwd_n1_tc", st);
    k<<<dim3(d.nc, d.H, d.B), kThreads, smem, st>>>(
        mapX, mapDY, mapS, mapG, d, (const bf *)p.Bm, (const bf *)p.Cm, (const bf *)p.wr, (const bf *)p.ww, p.dt,
        p.alpha, p.lam, p.tau, p.D, (bf *)p.dx, (bf *)p.dwr, (bf *)p.dww, p.ddt, p.dalpha, p.dlam, p.dD, dB_acc,
        dC_acc, p.dtau, err, cols);
    trace_end(st);
    *launched = true;
    return cudaGetLastError();
}

template <typename T, typename TS>
cudaError_t bwd_n1(const ScanDims &d, const ScanPtrs &p, void *S_in, void *dS_out, float *dB_acc,
                   float *dC_acc, float *scratch, bool reuse, int *err, cudaStream_t st) {
    const int npb = (d.P + kN1P - 1) / kN1P;
    float *loc = scratch, *dec = scratch + size_t(d.B) * d.H * d.nc * d.K * d.P;
    const bool vec = (reinterpret_cast<uintptr_t>(p.x) % 16 == 0) && (reinterpret_cast<uintptr_t>(p.dy) % 16 == 0) &&
                     ((size_t(d.P) * sizeof(T)) % 16 == 0);
    const int KP = d.K <= 4 ? 4 : d.K <= 8 ? 8 : d.K <= 16 ? 16 : 32;
    using I4 = std::integral_constant<int, 4>;
    using I8 = std::integral_constant<int, 8>;
    using I16 = std::integral_constant<int, 16>;
    using I32 = std::integral_constant<int, 32>;
    auto pick = [&](auto f) { return KP == 4 ? f(I4{}) : KP == 8 ? f(I8{}) : KP == 16 ? f(I16{}) : f(I32{}); };
    const size_t n1smem = N1Smem(sizeof(T)).total;
    const size_t total = size_t(d.B) * d.H * d.K * d.P;
    cudaError_t e = cudaSuccess;
    if (!reuse && d.nc > 0) {  // the forward's per-chunk entering states
        auto kl = pick([&](auto kp) {
            constexpr int V = decltype(kp)::value;
            return vec ? n1_local<T, true, V> : n1_local<T, false, V>;
        });
        cudaFuncSetAttribute(kl, cudaFuncAttributeMaxDynamicSharedMemorySize, int(n1smem));
        trace_begin("local_fwd_n1", st);
        kl<<<dim3(d.nc, d.H * npb, d.B), kN1P, n1smem, st>>>(d, (const T *)p.x, (const T *)p.Bm, (const T *)p.ww,
                                                             p.dt, p.alpha, p.lam, p.tau, loc, dec);
        trace_end(st);
        trace_begin("combine_fwd_n1", st);
        n1_combine<TS><<<unsigned((total + 255) / 256), 256, 0, st>>>(d, loc, dec, p.h0, (TS *)S_in, nullptr);
        trace_end(st);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    const size_t ngn = size_t(d.B) * d.L * d.G * d.N;
    if ((e = cudaMemsetAsync(p.dD, 0, sizeof(float) * d.H, st)) != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(dB_acc, 0, sizeof(float) * ngn, st)) != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(dC_acc, 0, sizeof(float) * ngn, st)) != cudaSuccess) return e;
    if (p.dtau && (e = cudaMemsetAsync(p.dtau, 0, sizeof(float) * d.H * d.K, st)) != cudaSuccess) return e;
    if (d.nc > 0) {  // the adjoint's chunk carries
        auto kr = pick([&](auto kp) {
            constexpr int V = decltype(kp)::value;
            return vec ? n1_rev_local<T, true, V> : n1_rev_local<T, false, V>;
        });
        cudaFuncSetAttribute(kr, cudaFuncAttributeMaxDynamicSharedMemorySize, int(n1smem));
        trace_begin("local_rev_n1", st);
        kr<<<dim3(d.nc, d.H * npb, d.B), kN1P, n1smem, st>>>(d, (const T *)p.dy, (const T *)p.Cm, (const T *)p.wr,
                                                             p.dt, p.alpha, p.lam, p.tau, loc, dec);
        trace_end(st);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    trace_begin("combine_rev_n1", st);
    n1_combine_rev<TS><<<unsigned((total + 255) / 256), 256, 0, st>>>(d, loc, dec, p.dh_final, (TS *)dS_out, p.dh0);
    trace_end(st);
    if ((e = cudaGetLastError()) != cudaSuccess || d.nc == 0) return e;  // L = 0: dh0 = dh_final
    bool done = false;
    if constexpr (std::is_same<T, __nv_bfloat16>::value && std::is_same<TS, __nv_bfloat16>::value) {
        if (n1_bwd_tc_ok(d, p, S_in, dS_out)) {
            if ((e = launch_n1_bwd_tc(d, p, S_in, dS_out, dB_acc, dC_acc, err, st, &done)) != cudaSuccess) return e;
        }
    }
    if (!done) {
        const size_t smem = N1BwdSmem(d.P, d.K, sizeof(T)).total;
        auto kb = pick([&](auto kp) {
            constexpr int V = decltype(kp)::value;
            return vec ? n1_chunk_bwd<T, TS, true, V> : n1_chunk_bwd<T, TS, false, V>;
        });
        cudaFuncSetAttribute(kb, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        trace_begin("chunk_bwd_n1", st);
        kb<<<dim3(d.nc, d.H, d.B), kThreads, smem, st>>>(
            d, (const T *)p.x, (const T *)p.Bm, (const T *)p.Cm, (const T *)p.wr, (const T *)p.ww, (const T *)p.dy,
            p.dt, p.alpha, p.lam, p.tau, p.D, (const TS *)S_in, (const TS *)dS_out, (T *)p.dx, (T *)p.dwr,
            (T *)p.dww, p.ddt, p.dalpha, p.dlam, p.dD, dB_acc, dC_acc, p.dtau);
        trace_end(st);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    if ((e = dtau_pairs_launch(d, sizeof(T) == 2 ? 1 : 0, p, st)) != cudaSuccess) return e;
    if (sizeof(T) == 2 && ngn > 0) {
        const unsigned blocks = unsigned(std::min<size_t>((ngn + 255) / 256, 4096));
        trace_begin("f32_to_bf16", st);
        f32_to_bf16_kernel<<<blocks, 256, 0, st>>>(dB_acc, (__nv_bfloat16 *)p.dB, ngn);
        trace_end(st);
        trace_begin("f32_to_bf16", st);
        f32_to_bf16_kernel<<<blocks, 256, 0, st>>>(dC_acc, (__nv_bfloat16 *)p.dC, ngn);
        trace_end(st);
        e = cudaGetLastError();
    }
    return e;
}

template <typename T, typename TS>
cudaError_t bwd_t(const ScanDims &d, const ScanPtrs &p, void *S_in, void *dS_out, float *dB_acc,
                  float *dC_acc, float *n1_scratch, bool reuse, int *err, cudaStream_t st) {
    if (uses_n1(d) && n1_bwd_fits(d, sizeof(T)))
        return bwd_n1<T, TS>(d, p, S_in, dS_out, dB_acc, dC_acc, n1_scratch, reuse, err, st);
    cudaError_t e = cudaSuccess;
    if (!reuse) e = run_state_pass<T, TS>(d, false, p.x, p.Bm, p.ww, p, p.h0, S_in, nullptr, st);
    if (e != cudaSuccess) return e;
    e = run_state_pass<T, TS>(d, true, p.dy, p.Cm, p.wr, p, p.dh_final, dS_out, p.dh0, st);
    if (e != cudaSuccess) return e;
    const size_t ngn = size_t(d.B) * d.L * d.G * d.N;
    if ((e = cudaMemsetAsync(p.dD, 0, sizeof(float) * d.H, st)) != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(dB_acc, 0, sizeof(float) * ngn, st)) != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(dC_acc, 0, sizeof(float) * ngn, st)) != cudaSuccess) return e;
    if (p.dtau && (e = cudaMemsetAsync(p.dtau, 0, sizeof(float) * d.H * d.K, st)) != cudaSuccess) return e;
    if (d.nc == 0) return cudaSuccess;  // L = 0: dh0 = dh_final was written, dD = 0
    const size_t smem = chunk_bwd_smem(d);
    auto k = simt_chunk_bwd<T, TS>;
    cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    trace_begin("chunk_bwd_simt", st);
    k<<<dim3(d.nc, d.H, d.B), kThreads, smem, st>>>(
        d, (const T *)p.x, (const T *)p.Bm, (const T *)p.Cm, (const T *)p.wr, (const T *)p.ww,
        (const T *)p.dy, p.dt, p.alpha, p.lam, p.tau, p.D, (const TS *)S_in,
        (const TS *)dS_out, (T *)p.dx, (T *)p.dwr, (T *)p.dww, p.ddt, p.dalpha, p.dlam, p.dD,
        dB_acc, dC_acc, p.dtau);
    trace_end(st);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if ((e = dtau_pairs_launch(d, sizeof(T) == 2 ? 1 : 0, p, st)) != cudaSuccess) return e;
    if (sizeof(T) == 2 && ngn > 0) {
        const unsigned blocks = unsigned(std::min<size_t>((ngn + 255) / 256, 4096));
        trace_begin("f32_to_bf16", st);
        f32_to_bf16_kernel<<<blocks, 256, 0, st>>>(dB_acc, (__nv_bfloat16 *)p.dB, ngn);
        trace_end(st);
        trace_begin("f32_to_bf16", st);
        f32_to_bf16_kernel<<<blocks, 256, 0, st>>>(dC_acc, (__nv_bfloat16 *)p.dC, ngn);
        trace_end(st);
        e = cudaGetLastError();
    }
    return e;
}

}  // namespace

int simt_pick_chunk(const ScanDims &d0, int requested) {
    if (d0.N == 1) {  // the N = 1 kernels: chunk 32 unless 16 is asked for (the backward's tiles)
        for (int Q : {32, 16}) {
            if (requested && requested != Q) continue;
            ScanDims d = d0;
            d.Q = Q;
            if (uses_n1(d) && n1_bwd_fits(d, 4)) return Q;
        }
    }
    const int cands[3] = {64, 32, 16};
    for (int qi = 0; qi < 3; ++qi) {
        const int Q = cands[qi];
        if (requested && requested != Q) continue;
        ScanDims d = d0;
        d.Q = Q;
        const int qt = Q / 4;
        if (state_pass_ps(d) == 0) continue;
        if (qt * ((d.P + 3) / 4) > kThreads) continue;     // dx tiles (and <= 2 y tiles per thread)
        if (qt * ((d.N + 7) / 8) > kThreads) continue;     // dB / dC tiles
        if (chunk_fwd_smem(d) > 227 * 1024) continue;
        if (chunk_bwd_smem(d) > 227 * 1024) continue;
        if (state_pass_smem(d, state_pass_ps(d)) > 227 * 1024) continue;
        return Q;
    }
    return 0;
}

size_t simt_state_elems(const ScanDims &d) {
    return size_t(d.B) * d.H * d.nc * d.K * d.P * d.N;
}

size_t simt_n1_scratch_elems(const ScanDims &d) {
    return uses_n1(d) ? size_t(d.B) * d.H * d.nc * d.K * (size_t(d.P) + 1) : 0;
}

cudaError_t simt_scan_fwd(const ScanDims &d, int dtype, const ScanPtrs &p, void *S_in, float *n1_scratch,
                          cudaStream_t st) {
    if (dtype == 0) return fwd_t<float, float>(d, p, S_in, n1_scratch, st);
    return fwd_t<__nv_bfloat16, __nv_bfloat16>(d, p, S_in, n1_scratch, st);
}

cudaError_t simt_scan_bwd(const ScanDims &d, int dtype, const ScanPtrs &p, void *S_in,
                          void *dS_out, float *dB_acc, float *dC_acc, float *n1_scratch, bool reuse,
                          int *err, cudaStream_t st) {
    if (dtype == 0) return bwd_t<float, float>(d, p, S_in, dS_out, dB_acc, dC_acc, n1_scratch, reuse, err, st);
    return bwd_t<__nv_bfloat16, __nv_bfloat16>(d, p, S_in, dS_out, dB_acc, dC_acc, n1_scratch, reuse, err, st);
}

}  // namespace frac
