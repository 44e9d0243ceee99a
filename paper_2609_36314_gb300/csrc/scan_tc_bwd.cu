// Tensor-core backward of the chunked Frac scan (bf16 inputs, chunk 128, headdim 64).
//
// With S_in / dS_out the per-chunk states of the forward and reverse state passes, every
// gradient of a chunk follows from chunk-local quantities (the adjoint of the recurrence of
// Sec. 3.2, written in the chunked order of App. E).  With G[t,k] = C_t.B_k, H[t,k] = dy_t.x_k,
// W_{t,k,m} = exp(-(E_t - E_k)/tau_m) (k <= t), u = exp(-(E_end - E)/tau), s = kappa u,
// f = w_read exp(-E/tau), Gamma = sum_m w_read kappa W and Gamma' = the same with kappa/tau:
//   dx_k       = sum_m s_{k,m} (B dS_out,m^T)[k] + sum_{t>=k} Gamma_{t,k} G_{t,k} dy_t + D dy_k
//   dkappa_k,m = u_{k,m} x_k.(B dS_out,m^T)[k] + sum_{t>=k} w_read_{t,m} W G H
//   dw_read_t,m= exp(-E_t/tau_m) dy_t.(C S_in,m^T)[t] + sum_{k<=t} kappa_{k,m} W G H
//   dC = sum_h (f o dy) S_in + (Gamma o H) B,   dB = sum_h (s o x) dS_out + (Gamma o H)^T C
//   rho_t <dS_t, S_{t-1}>/tau summed over modes = suffix(a) + prefix(b) + c + rect(Gamma' o G o H)
// (see the CUDA-core kernels for the same formulas; every term carries its own decay).
//
//   tc_bwd_intra  (b, c, h): G, H on the tensor cores; per-position passes for Gamma, Gamma',
//                 the intra parts of dw_read / dkappa and the pair rectangle sums; dx_intra =
//                 (Gamma o G)^T dy on the tensor cores; Gamma o H added over heads (fp32, L2).
//   tc_bwd_inter  (b, c, h, 32-wide P-slice): Z = C S_in^T and U = B dS_out^T on the tensor
//                 cores; epilogue to dx, dw_read, dkappa and the a, b terms.
//   tc_bwd_dcdb   (b, c, group of heads): dC and dB accumulated in tensor memory over the heads
//                 of the group (and the head-summed intra term, once per chunk).
//   tc_bwd_final  (b, h, c): per-position gradients of Delta, alpha, lambda, w_write, bf16 casts.
// All mbarrier waits are bounded; a timeout sets FRAC_ERR_TIMEOUT in the status word.
#include <cuda.h>

#include <algorithm>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"
#include "tc_util.cuh"

namespace frac {
namespace {

using namespace tc;
using bf16 = __nv_bfloat16;
constexpr int kThreads = 128;
constexpr int BP = 64;   // headdim of the tensor-core backward
constexpr int XS = 129;  // padded row stride (floats) of the fp32 pair tiles

struct BwdArgs {
    ScanDims d;
    const bf16 *x, *dy, *wr, *ww;
    const float *dt, *alpha, *lam, *tau, *D;
    const bf16 *S_in, *dS_out;
    float *dx_acc, *dwr_acc, *dkap_acc, *ab_acc, *rect, *cdot, *mh_total, *dB_acc, *dC_acc;
    bf16 *dx, *dwr, *dww;
    float *ddt, *dalpha, *dlam, *dD;
    int *err;
    int hg;  // heads per dC/dB group
};

__device__ __forceinline__ float head_log_cap(const float *tau, int h, int K) {
    float tmax = 0.f;
    for (int m = 0; m < K; ++m) tmax = fmaxf(tmax, tau[h * K + m]);
    return logf(64.f * tmax);
}

__device__ __forceinline__ void store_bf16x8(unsigned char *p, const float *v) {
    *reinterpret_cast<uint4 *>(p) = make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                                               pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7]));
}

__device__ __forceinline__ void load_bf16x32(const bf16 *src, float *v) {
    const uint4 *s4 = reinterpret_cast<const uint4 *>(src);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const uint4 u = s4[q];
        const __nv_bfloat162 *h2 = reinterpret_cast<const __nv_bfloat162 *>(&u);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = __bfloat1622float2(h2[i]);
            v[8 * q + 2 * i] = f.x;
            v[8 * q + 2 * i + 1] = f.y;
        }
    }
}

__device__ __forceinline__ unsigned char *align1024(unsigned char *p) {
    return reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

// ============================================================================= intra
constexpr int kIntraThreads = 256;  // two groups of four warps share the 128 TMEM lanes

struct IntraSmem {
    int rcb, x, dy, mg, xx, total;
    __host__ __device__ IntraSmem() {
        rcb = ((TQ * XS * 4 + 1023) / 1024) * 1024;  // C + B tiles (<= 64 KB), then fp32 G*H
        x = 16384;                 // x chunk [128 t][64 p], 128-byte swizzle
        dy = 16384;                // dy chunk
        mg = 2 * 16384;            // Gamma o G, [t][k] K-major
        xx = TQ * XS * 4;          // fp32 Gamma' G H, then its row prefix sums
        total = rcb + x + dy + mg + xx + 3 * TQ * KMAX * 4 + TQ * 8 + 64 * 4 + 64 + 64 + 64;
    }
};

__global__ void __launch_bounds__(kIntraThreads, 1)
    tc_bwd_intra(const __grid_constant__ CUtensorMap mapC, const __grid_constant__ CUtensorMap mapB,
                 const __grid_constant__ CUtensorMap mapX, const __grid_constant__ CUtensorMap mapDY,
                 BwdArgs a) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char *base = align1024(smem_raw);
    const ScanDims &d = a.d;
    const int K = d.K, N = d.N, P = d.P;
    const IntraSmem L;
    unsigned char *sC = base;
    unsigned char *sB = sC + (N / 64) * 16384;
    float *GHs = reinterpret_cast<float *>(base);          // reuses the C/B region
    unsigned char *sX = base + L.rcb;
    unsigned char *sDY = sX + L.x;
    unsigned char *sMG = sDY + L.dy;
    float *XX = reinterpret_cast<float *>(sMG + L.mg);
    float *wr_s = XX + TQ * XS;                              // [128][KMAX]
    float *kap_s = wr_s + TQ * KMAX;                         // [128][KMAX]
    float *part = kap_s + TQ * KMAX;                         // [128][KMAX] partial sums of group 1
    float2 *E_s = reinterpret_cast<float2 *>(part + TQ * KMAX);  // hi / lo pairs
    float *l2t = reinterpret_cast<float *>(E_s + TQ);
    float *tau_s = l2t + 32;
    double *wsum = reinterpret_cast<double *>(tau_s + 32);
    uint64_t *bars = reinterpret_cast<uint64_t *>(wsum + 8);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bars + 3);
    volatile int *abort_s = reinterpret_cast<volatile int *>(tslot + 1);

    const int tid = threadIdx.x, grp = tid >> 7, t = tid & 127, w4 = (tid >> 5) & 3;
    const int h = blockIdx.x, c = blockIdx.y, b = blockIdx.z;
    const int g = h / (d.H / d.G);
    const int c0 = c * TQ, n = min(TQ, d.L - c0);

    if (tid == 0) {
        for (int i = 0; i < 3; ++i) mbar_init(&bars[i], 1);
        *abort_s = 0;
        fence_barrier_init();
    }
    if (tid < K) {
        const float tv = a.tau[h * K + tid];
        tau_s[tid] = tv;
        l2t[tid] = kLog2e / tv;
    }
    if (tid < 32) tmem_alloc_once(tslot, 512);
    // per-position inputs of row t, all loads issued before anything waits on them
    float dtv = 1.f, alv = 1.f, lmv = 1.f;
    float wr_t[KMAX], ww_t[KMAX];
    if (t < n) {
        const size_t i = blh(d, b, c0 + t, h);
        dtv = a.dt[i];
        alv = a.alpha[i];
        lmv = a.lam[i];
        load_weights(a.wr + i * K, K, wr_t);
        load_weights(a.ww + i * K, K, ww_t);
    } else {
#pragma unroll
        for (int m = 0; m < KMAX; ++m) wr_t[m] = ww_t[m] = 0.f;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    const uint32_t lane_base = tmem + (uint32_t(w4 * 32) << 16);
    const uint32_t colG = 0, colH = 128, colX = 256;

    if (tid == 0) {
        mbar_arrive_expect_tx(&bars[0], uint32_t(2 * (N / 64) * 16384 + 2 * 16384));
        for (int jb = 0; jb < N / 64; ++jb) {
            tma_load_3d(sC + jb * 16384, &mapC, &bars[0], g * N + 64 * jb, c0, b);
            tma_load_3d(sB + jb * 16384, &mapB, &bars[0], g * N + 64 * jb, c0, b);
        }
        tma_load_3d(sX, &mapX, &bars[0], h * P, c0, b);
        tma_load_3d(sDY, &mapDY, &bars[0], h * P, c0, b);
    }
    float tmax = 0.f;
    for (int m = 0; m < K; ++m) tmax = fmaxf(tmax, tau_s[m]);
    const float log_cap = logf(64.f * tmax);
    float e = 0.f;
    if (t < n) {
        bool cl;
        e = token_rate(dtv, alv, lmv, log_cap, &cl);
    }
    const double Et = group_scan128(double(e), wsum);
    const float2 Et2 = split_f2(Et);
    if (grp == 0) E_s[t] = Et2;
    float l2r[KMAX];  // log2(e) / tau per mode, in registers
#pragma unroll
    for (int m = 0; m < KMAX; ++m) {
        l2r[m] = m < K ? l2t[m] : 0.f;
        float kp = 0.f;
        if (m < K && t < n) kp = -expm1f(-e / tau_s[m]) * ww_t[m];
        if (grp == 0) {
            wr_s[t * KMAX + m] = wr_t[m];
            kap_s[t * KMAX + m] = kp;
        }
    }
    __syncthreads();
    if (tid == 0) {
        if (!mbar_wait(&bars[0], 0)) {
            *abort_s = 1;
        } else {
            tc_fence_after();
            const uint32_t idG = idesc_bf16(128, 128, false, false);
            for (int ks = 0; ks < N / 16; ++ks) {
                const uint32_t koff = (ks / 4) * 16384 + (ks % 4) * 32;
                mma_bf16(tmem + colG, desc_sw128(smem_u32(sC) + koff, 16, 1024),
                         desc_sw128(smem_u32(sB) + koff, 16, 1024), idG, ks > 0);
            }
            for (int ks = 0; ks < BP / 16; ++ks) {  // H = dY X^T, K = p
                mma_bf16(tmem + colH, desc_sw128(smem_u32(sDY) + ks * 32, 16, 1024),
                         desc_sw128(smem_u32(sX) + ks * 32, 16, 1024), idG, ks > 0);
            }
            mma_commit(&bars[1]);
        }
    }
    __syncthreads();
    if (!*abort_s && !mbar_wait(&bars[1], 0)) *abort_s = 1;
    __syncthreads();
    tc_fence_after();
    // ---- row pass (row t; group 0 takes k in [0,32) and [96,128), group 1 takes [32,96)):
    // Gamma, Gamma', intra dw_read, Gamma o G tile, Gamma o H summed over heads in L2, Gamma' G H
    // and G H pair tiles
    float dwr_i[KMAX];
#pragma unroll
    for (int m = 0; m < KMAX; ++m) dwr_i[m] = 0.f;
    if (!*abort_s) {
        float *mh_row = a.mh_total + (((size_t(b) * d.nc + c) * d.G + g) * TQ + t) * TQ;
        for (int half = 0; half < 2; ++half) {
            const int k32 = grp == 0 ? (half == 0 ? 0 : 96) : (half == 0 ? 32 : 64);
            float gv[32], hv[32];
            tmem_ld32(lane_base + colG + k32, gv);
            tmem_ld32(lane_base + colH + k32, hv);
            tmem_ld_wait();
#pragma unroll
            for (int kk = 0; kk < 32; ++kk) {
                const int k = k32 + kk;
                float gam = 0.f, gamt = 0.f, gh = 0.f;
                if (k <= t && t < n) {
                    const float dE = diff_f2(Et2, E_s[k]);
                    gh = gv[kk] * hv[kk];
#pragma unroll
                    for (int m = 0; m < KMAX; ++m) {
                        if (m < K) {
                            const float W = ex2_approx(-dE * l2r[m]);
                            const float kp = kap_s[k * KMAX + m];
                            const float aa = wr_t[m] * kp * W;
                            gam += aa;
                            gamt = fmaf(aa, l2r[m], gamt);  // times log2(e) / tau
                            dwr_i[m] = fmaf(kp * W, gh, dwr_i[m]);
                        }
                    }
                }
                gv[kk] = gam * gv[kk];  // Gamma o G
                hv[kk] = gam * hv[kk];  // Gamma o H
                XX[t * XS + k] = gamt * (1.f / kLog2e) * gh;
                GHs[t * XS + k] = gh;
            }
            unsigned char *tile = sMG + (k32 >> 6) * 16384;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int c8 = ((k32 & 63) >> 3) + q;
                *reinterpret_cast<uint4 *>(tile + t * 128 + ((c8 ^ (t & 7)) * 16)) =
                    make_uint4(pack_bf16x2(gv[8 * q], gv[8 * q + 1]), pack_bf16x2(gv[8 * q + 2], gv[8 * q + 3]),
                               pack_bf16x2(gv[8 * q + 4], gv[8 * q + 5]), pack_bf16x2(gv[8 * q + 6], gv[8 * q + 7]));
            }
            if (t < n && k32 <= t) {
#pragma unroll
                for (int q = 0; q < 8; ++q)
                    if (k32 + 4 * q <= t)
                        atomicAdd(reinterpret_cast<float4 *>(mh_row + k32 + 4 * q),
                                  make_float4(hv[4 * q], hv[4 * q + 1], hv[4 * q + 2], hv[4 * q + 3]));
            }
        }
        if (grp == 1) {
#pragma unroll
            for (int m = 0; m < KMAX; ++m) part[t * KMAX + m] = dwr_i[m];
        }
    }
    fence_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (!*abort_s && grp == 0 && t < n) {
        float *o = a.dwr_acc + blh(d, b, c0 + t, h) * K;
#pragma unroll
        for (int m = 0; m < KMAX; ++m)
            if (m < K) o[m] = dwr_i[m] + part[t * KMAX + m];
    }
    if (tid == 0 && !*abort_s) {  // dx_intra = (Gamma o G)^T dY: M = k, N = p, K = t
        const uint32_t idX = idesc_bf16(128, BP, true, true);
        for (int ks = 0; ks < TQ / 16; ++ks)
            mma_bf16(tmem + colX, desc_sw128(smem_u32(sMG) + ks * 2048, 16384, 1024),
                     desc_sw128(smem_u32(sDY) + ks * 2048, 16384, 1024), idX, ks > 0);
        mma_commit(&bars[2]);
    }
    __syncthreads();  // part[] is reused below
    // ---- column pass (column k = t; group g takes rows t' = k + g, k + g + 2, ...): intra dkappa
    float dk[KMAX];
#pragma unroll
    for (int m = 0; m < KMAX; ++m) dk[m] = 0.f;
    if (!*abort_s) {
        // all lanes of a warp walk the same rows tt (broadcast loads of E, w_read); rows above the
        // diagonal (tt < k) contribute nothing
        const int k = t;
        const float2 Ek = E_s[k];
        float dk2[KMAX];
#pragma unroll
        for (int m = 0; m < KMAX; ++m) dk2[m] = 0.f;
        // group grp takes the rows of parity grp, starting at this warp's first column; four
        // rows per step (two accumulator sets) keep several exponentials in flight
        for (int tt0 = (t & ~31) + grp; tt0 < n; tt0 += 8) {
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int tt = tt0 + 2 * u;
                if (tt < n && tt >= k) {
                    const float dE = diff_f2(E_s[tt], Ek);
                    const float gh = GHs[tt * XS + k];
#pragma unroll
                    for (int m = 0; m < KMAX; ++m) {
                        if (m < K) {
                            const float v = wr_s[tt * KMAX + m] * ex2_approx(-dE * l2r[m]);
                            if (u & 1)
                                dk2[m] = fmaf(v, gh, dk2[m]);
                            else
                                dk[m] = fmaf(v, gh, dk[m]);
                        }
                    }
                }
            }
        }
#pragma unroll
        for (int m = 0; m < KMAX; ++m) dk[m] += dk2[m];
        if (grp == 1) {
#pragma unroll
            for (int m = 0; m < KMAX; ++m) part[k * KMAX + m] = dk[m];
        }
    }
    // exclusive row prefix of XX (row t, group 0)
    if (!*abort_s && grp == 0) {
        float run = 0.f;
        for (int j = 0; j < TQ; ++j) {
            const float v = XX[t * XS + j];
            XX[t * XS + j] = run;
            run += v;
        }
    }
    __syncthreads();
    if (!*abort_s && grp == 0 && t < n) {
        float *o = a.dkap_acc + blh(d, b, c0 + t, h) * K;
#pragma unroll
        for (int m = 0; m < KMAX; ++m)
            if (m < K) o[m] = dk[m] + part[t * KMAX + m];
        float sr = 0.f;
        for (int tp = t; tp < n; ++tp) sr += XX[tp * XS + t];
        a.rect[blh(d, b, c0 + t, h)] = sr;
    }
    __syncthreads();
    if (!*abort_s && !mbar_wait(&bars[2], 0)) *abort_s = 1;
    __syncthreads();
    tc_fence_after();
    if (!*abort_s) {  // dx_intra row: group g takes columns [32 g, 32 g + 32)
        float v[32];
        tmem_ld32(lane_base + colX + grp * 32, v);
        tmem_ld_wait();
        if (t < n) {
            float4 *o = reinterpret_cast<float4 *>(a.dx_acc + blh(d, b, c0 + t, h) * P + grp * 32);
#pragma unroll
            for (int q = 0; q < 8; ++q) o[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        }
    }
    if (*abort_s && tid == 0) atomicExch(a.err, kTimeoutCode);
    tc_fence_before();
    __syncthreads();
    if (tid < 32) tmem_dealloc(tmem, 512);
}

// ============================================================================= inter
struct InterSmem {
    int cb, s, total;
    __host__ __device__ InterSmem(int K, int N) {
        cb = (N / 64) * 16384;           // one of C / B
        s = (N / 64) * (K * TPS * 128);  // one of S_in / dS_out slices
        total = 2 * cb + 2 * s + 64 + 64;
    }
};

__global__ void __launch_bounds__(kThreads, 1)
    tc_bwd_inter(const __grid_constant__ CUtensorMap mapC, const __grid_constant__ CUtensorMap mapB,
                 const __grid_constant__ CUtensorMap mapS, const __grid_constant__ CUtensorMap mapD,
                 BwdArgs a) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char *base = align1024(smem_raw);
    const ScanDims &d = a.d;
    const int K = d.K, N = d.N, P = d.P;
    const InterSmem L(K, N);
    unsigned char *sC = base, *sB = sC + L.cb, *sS = sB + L.cb, *sD = sS + L.s;
    double *wsum = reinterpret_cast<double *>(sD + L.s);
    uint64_t *bars = reinterpret_cast<uint64_t *>(wsum + 4);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bars + 2);
    volatile int *abort_s = reinterpret_cast<volatile int *>(tslot + 1);
    __shared__ float itau[32];

    const int tid = threadIdx.x, w = tid >> 5, r = tid;
    const int npart = P / TPS;
    const int h = blockIdx.x / npart, p0 = (blockIdx.x % npart) * TPS;
    const int c = blockIdx.y, b = blockIdx.z;
    const int g = h / (d.H / d.G);
    const int c0 = c * TQ, n = min(TQ, d.L - c0);
    const uint32_t ZN = uint32_t(K * TPS);

    if (tid == 0) {
        mbar_init(&bars[0], 1);
        mbar_init(&bars[1], 1);
        *abort_s = 0;
        fence_barrier_init();
    }
    if (tid < K) itau[tid] = 1.f / a.tau[h * K + tid];
    if (w == 0) tmem_alloc_once(tslot, 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    const uint32_t lane_base = tmem + (uint32_t(w * 32) << 16);
    if (tid == 0) {
        mbar_arrive_expect_tx(&bars[0], uint32_t(2 * L.cb + 2 * L.s));
        const int srow = int(((size_t(b) * d.H + h) * d.nc + c) * K);
        for (int jb = 0; jb < N / 64; ++jb) {
            tma_load_3d(sC + jb * 16384, &mapC, &bars[0], g * N + 64 * jb, c0, b);
            tma_load_3d(sB + jb * 16384, &mapB, &bars[0], g * N + 64 * jb, c0, b);
            tma_load_3d(sS + jb * (K * TPS * 128), &mapS, &bars[0], 64 * jb, p0, srow);
            tma_load_3d(sD + jb * (K * TPS * 128), &mapD, &bars[0], 64 * jb, p0, srow);
        }
    }
    // per-position coefficients of row r
    const float log_cap = head_log_cap(a.tau, h, K);
    float e = 0.f;
    if (r < n) {
        const size_t i = blh(d, b, c0 + r, h);
        bool cl;
        e = token_rate(a.dt[i], a.alpha[i], a.lam[i], log_cap, &cl);
    }
    const double Er = block_scan128(double(e), wsum);
    __shared__ double Eend_s;
    if (r == n - 1) Eend_s = Er;
    __syncthreads();
    const double Eend = Eend_s;
    float s_r[KMAX], u_r[KMAX], fd_r[KMAX], f_r[KMAX];
#pragma unroll
    for (int m = 0; m < KMAX; ++m) {
        s_r[m] = u_r[m] = fd_r[m] = f_r[m] = 0.f;
        if (m < K && r < n) {
            const size_t wi = blh(d, b, c0 + r, h) * K + m;
            const float kp = -expm1f(-e * itau[m]) * to_f(a.ww[wi]);
            u_r[m] = expf(-float(Eend - Er) * itau[m]);
            s_r[m] = kp * u_r[m];
            fd_r[m] = expf(-float(Er) * itau[m]);
            f_r[m] = to_f(a.wr[wi]) * fd_r[m];
        }
    }
    float xr[32], dyr[32];
    if (r < n) {
        load_bf16x32(a.x + blh(d, b, c0 + r, h) * P + p0, xr);
        load_bf16x32(a.dy + blh(d, b, c0 + r, h) * P + p0, dyr);
    } else {
#pragma unroll
        for (int p = 0; p < 32; ++p) xr[p] = dyr[p] = 0.f;
    }
    if (tid == 0) {
        if (!mbar_wait(&bars[0], 0)) {
            *abort_s = 1;
        } else {
            tc_fence_after();
            const uint32_t idZ = idesc_bf16(128, int(ZN), false, false);
            for (int ks = 0; ks < N / 16; ++ks) {
                const uint32_t koff = (ks / 4) * 16384 + (ks % 4) * 32;
                const uint32_t soff = (ks / 4) * (K * TPS * 128) + (ks % 4) * 32;
                mma_bf16(tmem, desc_sw128(smem_u32(sC) + koff, 16, 1024),
                         desc_sw128(smem_u32(sS) + soff, 16, 1024), idZ, ks > 0);
                mma_bf16(tmem + ZN, desc_sw128(smem_u32(sB) + koff, 16, 1024),
                         desc_sw128(smem_u32(sD) + soff, 16, 1024), idZ, ks > 0);
            }
            mma_commit(&bars[1]);
        }
    }
    // <dS_out, S_in> of this P-slice per mode, straight from the two tiles in shared memory (both
    // carry the same swizzle, so the byte-for-byte dot product is the element dot product);
    // it runs while the tensor cores work
    if (mbar_wait(&bars[0], 0)) {
        const int tpm = kThreads / K;  // threads per mode
        const int m = tid / tpm, jl = tid % tpm;
        float acc = 0.f;
        for (int jb = 0; jb < N / 64; ++jb) {
            const uint4 *ps = reinterpret_cast<const uint4 *>(sS + jb * (K * TPS * 128) + m * 4096);
            const uint4 *pd = reinterpret_cast<const uint4 *>(sD + jb * (K * TPS * 128) + m * 4096);
            for (int q = jl; q < 256; q += tpm) {
                const uint4 u = ps[q], v = pd[q];
                const __nv_bfloat162 *a2 = reinterpret_cast<const __nv_bfloat162 *>(&u);
                const __nv_bfloat162 *b2 = reinterpret_cast<const __nv_bfloat162 *>(&v);
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const float2 fa = __bfloat1622float2(a2[i]), fb = __bfloat1622float2(b2[i]);
                    acc = fmaf(fa.x, fb.x, fmaf(fa.y, fb.y, acc));
                }
            }
        }
        for (int o = tpm >> 1; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        if (jl == 0) atomicAdd(a.cdot + ((size_t(b) * d.H + h) * d.nc + c) * K + m, acc);
    } else {
        *abort_s = 1;
    }
    __syncthreads();
    if (!*abort_s && !mbar_wait(&bars[1], 0)) *abort_s = 1;
    __syncthreads();
    tc_fence_after();
    if (!*abort_s) {
        float dx[32];
#pragma unroll
        for (int p = 0; p < 32; ++p) dx[p] = 0.f;
        float aa = 0.f, bb = 0.f;
        float *dwr = a.dwr_acc + blh(d, b, c0 + r, h) * K;
        float *dkp = a.dkap_acc + blh(d, b, c0 + r, h) * K;
#pragma unroll
        for (int m = 0; m < KMAX; ++m) {
            if (m >= K) break;
            float z[32], u[32];
            tmem_ld32(lane_base + m * TPS, z);
            tmem_ld32(lane_base + ZN + m * TPS, u);
            tmem_ld_wait();
            float dyz = 0.f, xu = 0.f;
#pragma unroll
            for (int p = 0; p < 32; ++p) {
                dyz = fmaf(dyr[p], z[p], dyz);
                xu = fmaf(xr[p], u[p], xu);
                dx[p] = fmaf(s_r[m], u[p], dx[p]);
            }
            if (r < n) {
                atomicAdd(dwr + m, fd_r[m] * dyz);
                atomicAdd(dkp + m, u_r[m] * xu);
            }
            aa = fmaf(f_r[m] * dyz, itau[m], aa);
            bb = fmaf(s_r[m] * xu, itau[m], bb);
        }
        if (r < n) {
            atomicAdd(a.ab_acc + blh(d, b, c0 + r, h) * 2, aa);
            atomicAdd(a.ab_acc + blh(d, b, c0 + r, h) * 2 + 1, bb);
            float4 *o = reinterpret_cast<float4 *>(a.dx_acc + blh(d, b, c0 + r, h) * P + p0);
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                float4 v = o[q];
                v.x += dx[4 * q]; v.y += dx[4 * q + 1]; v.z += dx[4 * q + 2]; v.w += dx[4 * q + 3];
                o[q] = v;
            }
        }
    }
    if (*abort_s && tid == 0) atomicExch(a.err, kTimeoutCode);
    tc_fence_before();
    __syncthreads();
    if (w == 0) tmem_dealloc(tmem, 512);
}

// ============================================================================= dC / dB
struct DcdbSmem {
    int s, gen, total;
    __host__ __device__ DcdbSmem(int K, int N) {
        s = (N / 64) * (K * TPS * 128);  // S_in / dS_out slice; also holds the B / C chunk
        if (s < (N / 64) * 16384) s = (N / 64) * 16384;
        gen = (K * TPS / 64) * 16384;    // generated [128][(m, p)] operand; also Gamma o H
        if (gen < 2 * 16384) gen = 2 * 16384;
        total = 2 * s + gen + 64 + 64;
    }
};

__global__ void __launch_bounds__(kThreads, 1)
    tc_bwd_dcdb(const __grid_constant__ CUtensorMap mapS, const __grid_constant__ CUtensorMap mapD,
                const __grid_constant__ CUtensorMap mapB, const __grid_constant__ CUtensorMap mapC,
                BwdArgs a) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char *base = align1024(smem_raw);
    const ScanDims &d = a.d;
    const int K = d.K, N = d.N, P = d.P;
    const DcdbSmem L(K, N);
    unsigned char *sS = base, *sD = sS + L.s, *sG = sD + L.s;
    double *wsum = reinterpret_cast<double *>(sG + L.gen);
    uint64_t *bars = reinterpret_cast<uint64_t *>(wsum + 4);  // tma, mma
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bars + 2);
    volatile int *abort_s = reinterpret_cast<volatile int *>(tslot + 1);
    __shared__ float itau[32];
    __shared__ double Eend_s;

    const int tid = threadIdx.x, w = tid >> 5, t = tid;
    const int hg = blockIdx.x, c = blockIdx.y, b = blockIdx.z;
    const int h_first = hg * a.hg;
    const int g = h_first / (d.H / d.G);
    const int c0 = c * TQ, n = min(TQ, d.L - c0);
    const uint32_t KP = uint32_t(K * TPS);  // contraction length per P-slice
    const uint32_t colC = 0, colB = 128;

    if (tid == 0) {
        mbar_init(&bars[0], 1);
        mbar_init(&bars[1], 1);
        *abort_s = 0;
        fence_barrier_init();
    }
    if (w == 0) tmem_alloc_once(tslot, 256);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    const uint32_t lane_base = tmem + (uint32_t(w * 32) << 16);
    uint32_t tma_phase = 0, mma_phase = 0;
    bool first = true;  // first MMA into the accumulators overwrites them

    // helpers ---------------------------------------------------------------
    auto wait_mma = [&]() {
        if (!mbar_wait(&bars[1], mma_phase)) *abort_s = 1;
        mma_phase ^= 1;
    };

    // head-summed intra term, once per chunk and B/C group (by the group's first block):
    // dC = M_H B, dB = M_H^T C
    if (h_first % (d.H / d.G) == 0) {
        if (tid == 0) {
            mbar_arrive_expect_tx(&bars[0], uint32_t(2 * (N / 64) * 16384));
            for (int jb = 0; jb < N / 64; ++jb) {
                tma_load_3d(sS + jb * 16384, &mapB, &bars[0], g * N + 64 * jb, c0, b);
                tma_load_3d(sD + jb * 16384, &mapC, &bars[0], g * N + 64 * jb, c0, b);
            }
        }
        const float *mrow = a.mh_total + (((size_t(b) * d.nc + c) * d.G + g) * TQ + t) * TQ;
        for (int k8 = 0; k8 < TQ; k8 += 8) {
            float v[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) v[i] = mrow[k8 + i];
            const int c8 = (k8 & 63) >> 3;
            store_bf16x8(sG + (k8 >> 6) * 16384 + t * 128 + ((c8 ^ (t & 7)) * 16), v);
        }
        fence_async_smem();
        __syncthreads();
        if (tid == 0) {
            if (!mbar_wait(&bars[0], tma_phase)) {
                *abort_s = 1;
            } else {
                tc_fence_after();
                const uint32_t idC = idesc_bf16(128, N, false, true);
                const uint32_t idB = idesc_bf16(128, N, true, true);
                for (int ks = 0; ks < TQ / 16; ++ks) {
                    // dC[t, n] += sum_k M[t, k] B[k, n]
                    mma_bf16(tmem + colC,
                             desc_sw128(smem_u32(sG) + (ks / 4) * 16384 + (ks % 4) * 32, 16, 1024),
                             desc_sw128(smem_u32(sS) + ks * 2048, 16384, 1024), idC, ks > 0);
                    // dB[k, n] += sum_t M[t, k] C[t, n]
                    mma_bf16(tmem + colB, desc_sw128(smem_u32(sG) + ks * 2048, 16384, 1024),
                             desc_sw128(smem_u32(sD) + ks * 2048, 16384, 1024), idB, ks > 0);
                }
                mma_commit(&bars[1]);
            }
        }
        tma_phase ^= 1;
        __syncthreads();
        if (!*abort_s) wait_mma();
        __syncthreads();
        first = false;
    }

    for (int hh = 0; hh < a.hg && !*abort_s; ++hh) {
        const int h = h_first + hh;
        if (tid < K) itau[tid] = 1.f / a.tau[h * K + tid];
        __syncthreads();
        const float log_cap = head_log_cap(a.tau, h, K);
        float e = 0.f;
        if (t < n) {
            const size_t i = blh(d, b, c0 + t, h);
            bool cl;
            e = token_rate(a.dt[i], a.alpha[i], a.lam[i], log_cap, &cl);
        }
        const double Et = block_scan128(double(e), wsum);
        if (t == n - 1) Eend_s = Et;
        __syncthreads();
        const double Eend = Eend_s;
        float f_t[KMAX], s_t[KMAX];
#pragma unroll
        for (int m = 0; m < KMAX; ++m) {
            f_t[m] = s_t[m] = 0.f;
            if (m < K && t < n) {
                const size_t wi = blh(d, b, c0 + t, h) * K + m;
                f_t[m] = to_f(a.wr[wi]) * expf(-float(Et) * itau[m]);
                s_t[m] = -expm1f(-e * itau[m]) * to_f(a.ww[wi]) * expf(-float(Eend - Et) * itau[m]);
            }
        }
        const int srow = int(((size_t(b) * d.H + h) * d.nc + c) * K);
        for (int ps = 0; ps < P / TPS && !*abort_s; ++ps) {
            const int p0 = ps * TPS;
            if (tid == 0) {
                mbar_arrive_expect_tx(&bars[0], uint32_t(2 * (N / 64) * (K * TPS * 128)));
                for (int jb = 0; jb < N / 64; ++jb) {
                    tma_load_3d(sS + jb * (K * TPS * 128), &mapS, &bars[0], 64 * jb, p0, srow);
                    tma_load_3d(sD + jb * (K * TPS * 128), &mapD, &bars[0], 64 * jb, p0, srow);
                }
            }
            // dC += (f o dy)[t, (m, p)] S_in[(m, p), n]
            for (int pass = 0; pass < 2; ++pass) {
                float src[32];
                if (t < n)
                    load_bf16x32((pass == 0 ? a.dy : a.x) + blh(d, b, c0 + t, h) * P + p0, src);
                else
#pragma unroll
                    for (int p = 0; p < 32; ++p) src[p] = 0.f;
#pragma unroll
                for (int m = 0; m < KMAX; ++m) {
                    if (m >= K) break;
                    const float cm = pass == 0 ? f_t[m] : s_t[m];
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        float v[8];
#pragma unroll
                        for (int i = 0; i < 8; ++i) v[i] = cm * src[8 * q + i];
                        const int kidx = m * TPS + 8 * q;  // (m, p) index of the first element
                        const int c8 = (kidx & 63) >> 3;
                        store_bf16x8(sG + (kidx >> 6) * 16384 + t * 128 + ((c8 ^ (t & 7)) * 16), v);
                    }
                }
                fence_async_smem();
                tc_fence_before();
                __syncthreads();
                tc_fence_after();
                if (tid == 0) {
                    bool ok = true;
                    if (pass == 0 && !mbar_wait(&bars[0], tma_phase)) ok = false;
                    if (!ok) {
                        *abort_s = 1;
                    } else {
                        tc_fence_after();
                        const uint32_t id = idesc_bf16(128, N, false, true);
                        unsigned char *bt = pass == 0 ? sS : sD;
                        for (int ks = 0; ks < int(KP) / 16; ++ks)
                            mma_bf16(tmem + (pass == 0 ? colC : colB),
                                     desc_sw128(smem_u32(sG) + (ks / 4) * 16384 + (ks % 4) * 32, 16, 1024),
                                     desc_sw128(smem_u32(bt) + ks * 2048, K * TPS * 128, 1024), id,
                                     (first && ks == 0) ? 0u : 1u);
                        mma_commit(&bars[1]);
                    }
                }
                __syncthreads();
                if (!*abort_s) wait_mma();  // the generated operand buffer is reused next
                __syncthreads();
                if (pass == 1) first = false;  // both accumulators now hold data
            }
            tma_phase ^= 1;
        }
    }
    // accumulate the group's dC / dB into the fp32 outputs (every lane takes part in the
    // warp-collective tensor-memory loads; rows beyond the sequence end store nothing)
    tc_fence_after();
    if (!*abort_s) {
        const size_t gi = ((size_t(b) * d.L + c0 + min(t, n - 1)) * d.G + g) * N;
        for (int n32 = 0; n32 < N; n32 += 32) {
            float vc[32], vb[32];
            tmem_ld32(lane_base + colC + n32, vc);
            tmem_ld32(lane_base + colB + n32, vb);
            tmem_ld_wait();
            if (t < n) {
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    atomicAdd(reinterpret_cast<float4 *>(a.dC_acc + gi + n32 + 4 * q),
                              make_float4(vc[4 * q], vc[4 * q + 1], vc[4 * q + 2], vc[4 * q + 3]));
                    atomicAdd(reinterpret_cast<float4 *>(a.dB_acc + gi + n32 + 4 * q),
                              make_float4(vb[4 * q], vb[4 * q + 1], vb[4 * q + 2], vb[4 * q + 3]));
                }
            }
        }
    }
    if (*abort_s && tid == 0) atomicExch(a.err, kTimeoutCode);
    tc_fence_before();
    __syncthreads();
    if (w == 0) tmem_dealloc(tmem, 256);
}

// ============================================================================= final
__global__ void __launch_bounds__(kThreads) tc_bwd_final(BwdArgs a) {
    const ScanDims &d = a.d;
    const int K = d.K, P = d.P;
    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z, t = threadIdx.x;
    const int c0 = c * TQ, n = min(TQ, d.L - c0);
    __shared__ double wsum[4];
    __shared__ float itau[32];
    __shared__ double tot_s[2];
    __shared__ float red[4];
    if (t < K) itau[t] = 1.f / a.tau[h * K + t];
    __syncthreads();
    const float log_cap = head_log_cap(a.tau, h, K);
    float e = 0.f;
    bool cl = false;
    const size_t i = (t < n) ? blh(d, b, c0 + t, h) : 0;
    if (t < n) e = token_rate(a.dt[i], a.alpha[i], a.lam[i], log_cap, &cl);
    const double Et = block_scan128(double(e), wsum);
    const float av = t < n ? a.ab_acc[i * 2] : 0.f;
    const float bv = t < n ? a.ab_acc[i * 2 + 1] : 0.f;
    const double pa = block_scan128(double(av), wsum);  // inclusive prefix of a
    const double pb = block_scan128(double(bv), wsum);  // inclusive prefix of b
    if (t == n - 1) {
        tot_s[0] = pa;
        tot_s[1] = Et;
    }
    __syncthreads();
    const double Eend = tot_s[1];
    float cprime = 0.f;
    for (int m = 0; m < K; ++m)
        cprime = fmaf(expf(-float(Eend) * itau[m]) * itau[m],
                      a.cdot[((size_t(b) * d.H + h) * d.nc + c) * K + m], cprime);
    float dd = 0.f;
    if (t < n) {
        const double suf_a = tot_s[0] - (pa - av);
        const double pre_b = pb - bv;
        const float R = float(suf_a + pre_b) + cprime + a.rect[i];
        float de = -R;
        for (int m = 0; m < K; ++m) {
            const float z = e * itau[m];
            const float rho = expf(-z), omr = -expm1f(-z);
            const float ww = to_f(a.ww[i * K + m]);
            const float dk = a.dkap_acc[i * K + m];
            de = fmaf(dk * rho * ww, itau[m], de);
            a.dwr[i * K + m] = from_f<bf16>(a.dwr_acc[i * K + m]);
            a.dww[i * K + m] = from_f<bf16>(dk * omr);
        }
        const float al = a.alpha[i], lm = a.lam[i], dtv = a.dt[i];
        const float ge = cl ? 0.f : de * e;
        a.ddt[i] = ge / dtv;
        a.dlam[i] = ge / (al * lm);
        a.dalpha[i] = -ge * logf(lm) / (al * al);
        const float Dh = a.D[h];
        for (int p32 = 0; p32 < P; p32 += 32) {
            float dyv[32], xv[32];
            load_bf16x32(a.dy + i * P + p32, dyv);
            load_bf16x32(a.x + i * P + p32, xv);
            const float4 *src = reinterpret_cast<const float4 *>(a.dx_acc + i * P + p32);
            uint4 *o = reinterpret_cast<uint4 *>(a.dx + i * P + p32);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float4 u0 = src[2 * q], u1 = src[2 * q + 1];
                const float v[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
                float r8[8];
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    r8[k] = v[k] + Dh * dyv[8 * q + k];
                    dd = fmaf(dyv[8 * q + k], xv[8 * q + k], dd);
                }
                o[q] = make_uint4(pack_bf16x2(r8[0], r8[1]), pack_bf16x2(r8[2], r8[3]),
                                  pack_bf16x2(r8[4], r8[5]), pack_bf16x2(r8[6], r8[7]));
            }
        }
    }
    dd = warp_sum(dd);
    if ((t & 31) == 0) red[t >> 5] = dd;
    __syncthreads();
    if (t == 0) atomicAdd(a.dD + h, red[0] + red[1] + red[2] + red[3]);
}

__global__ void f32_to_bf16_tc(const float *__restrict__ in, bf16 *__restrict__ out, size_t n) {
    for (size_t i = blockIdx.x * size_t(blockDim.x) + threadIdx.x; i < n; i += size_t(gridDim.x) * blockDim.x)
        out[i] = __float2bfloat16_rn(in[i]);
}

int pick_hg(const ScanDims &d) {
    const int hpg = d.H / d.G;
    for (int hg = 16; hg >= 1; --hg)
        if (hpg % hg == 0) return hg;
    return 1;
}

}  // namespace

bool tc_bwd_supported(const ScanDims &d, int dtype) { return tc_supported(d, dtype) && d.P == BP; }

size_t tc_bwd_workspace_bytes(const ScanDims &d, TcBwdWorkspace *l, char *base) {
    auto ru = [](size_t v) { return (v + 255) / 256 * 256; };
    const size_t blh_ = size_t(d.B) * d.L * d.H;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        char *p = base ? base + off : nullptr;
        off += ru(bytes);
        return p;
    };
    const size_t st = tc_state_elems(d) * 2;
    l->S_in = take(st);
    l->dS_out = take(st);
    l->dx_acc = (float *)take(blh_ * d.P * 4);
    l->dwr_acc = (float *)take(blh_ * d.K * 4);
    l->dkap_acc = (float *)take(blh_ * d.K * 4);
    l->ab_acc = (float *)take(blh_ * 2 * 4);
    l->rect = (float *)take(blh_ * 4);
    l->cdot = (float *)take(size_t(d.B) * d.H * d.nc * d.K * 4);
    l->mh_total = (float *)take(size_t(d.B) * d.nc * d.G * TQ * TQ * 4);
    l->dB_acc = (float *)take(size_t(d.B) * d.L * d.G * d.N * 4);
    l->dC_acc = (float *)take(size_t(d.B) * d.L * d.G * d.N * 4);
    return off;
}

cudaError_t tc_scan_bwd(const ScanDims &d, const ScanPtrs &p, const TcBwdWorkspace &ws, int *err,
                        bool reuse_states, cudaStream_t st) {
    cudaError_t e;
    const size_t ngn = size_t(d.B) * d.L * d.G * d.N;
    const size_t blh_ = size_t(d.B) * d.L * d.H;
    if ((e = cudaMemsetAsync(p.dD, 0, sizeof(float) * d.H, st))) return e;
    if ((e = cudaMemsetAsync(ws.dB_acc, 0, sizeof(float) * ngn, st))) return e;
    if ((e = cudaMemsetAsync(ws.dC_acc, 0, sizeof(float) * ngn, st))) return e;
    if ((e = cudaMemsetAsync(ws.cdot, 0, sizeof(float) * d.B * d.H * d.nc * d.K, st))) return e;
    if ((e = cudaMemsetAsync(ws.ab_acc, 0, sizeof(float) * blh_ * 2, st))) return e;
    if ((e = cudaMemsetAsync(ws.mh_total, 0, sizeof(float) * d.B * d.nc * d.G * TQ * TQ, st))) return e;
    if (!reuse_states &&
        (e = tc_state_pass_launch(d, false, p.x, p.Bm, p.ww, p.dt, p.alpha, p.lam, p.tau, p.h0,
                                  ws.S_in, nullptr, err, st)))
        return e;
    if ((e = tc_state_pass_launch(d, true, p.dy, p.Cm, p.wr, p.dt, p.alpha, p.lam, p.tau,
                                  p.dh_final, ws.dS_out, p.dh0, err, st)))
        return e;
    if (d.nc == 0) return cudaSuccess;
    const uint64_t GN = uint64_t(d.G) * d.N, HP = uint64_t(d.H) * d.P;
    CUtensorMap mapC, mapB, mapX, mapDY, mapS, mapD;
    const uint64_t srows = uint64_t(d.B) * d.H * d.nc * d.K;
    if (!tc_make_map3(&mapC, p.Cm, GN, d.L, d.B, GN * 2, uint64_t(d.L) * GN * 2, 64, TQ, 1) ||
        !tc_make_map3(&mapB, p.Bm, GN, d.L, d.B, GN * 2, uint64_t(d.L) * GN * 2, 64, TQ, 1) ||
        !tc_make_map3(&mapX, p.x, HP, d.L, d.B, HP * 2, uint64_t(d.L) * HP * 2, 64, TQ, 1) ||
        !tc_make_map3(&mapDY, p.dy, HP, d.L, d.B, HP * 2, uint64_t(d.L) * HP * 2, 64, TQ, 1) ||
        !tc_make_map3(&mapS, ws.S_in, d.N, d.P, srows, uint64_t(d.N) * 2, uint64_t(d.P) * d.N * 2, 64,
                      TPS, d.K) ||
        !tc_make_map3(&mapD, ws.dS_out, d.N, d.P, srows, uint64_t(d.N) * 2, uint64_t(d.P) * d.N * 2, 64,
                      TPS, d.K))
        return cudaErrorInvalidValue;
    BwdArgs a;
    a.d = d;
    a.x = (const bf16 *)p.x; a.dy = (const bf16 *)p.dy;
    a.wr = (const bf16 *)p.wr; a.ww = (const bf16 *)p.ww;
    a.dt = p.dt; a.alpha = p.alpha; a.lam = p.lam; a.tau = p.tau; a.D = p.D;
    a.S_in = (const bf16 *)ws.S_in; a.dS_out = (const bf16 *)ws.dS_out;
    a.dx_acc = ws.dx_acc; a.dwr_acc = ws.dwr_acc; a.dkap_acc = ws.dkap_acc; a.ab_acc = ws.ab_acc;
    a.rect = ws.rect; a.cdot = ws.cdot; a.mh_total = ws.mh_total;
    a.dB_acc = ws.dB_acc; a.dC_acc = ws.dC_acc;
    a.dx = (bf16 *)p.dx; a.dwr = (bf16 *)p.dwr; a.dww = (bf16 *)p.dww;
    a.ddt = p.ddt; a.dalpha = p.dalpha; a.dlam = p.dlam; a.dD = p.dD;
    a.err = err;
    a.hg = pick_hg(d);

    {
        const size_t smem = IntraSmem().total + 1024;
        cudaFuncSetAttribute(tc_bwd_intra, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        trace_begin("bwd_intra_tc", st);
        tc_bwd_intra<<<dim3(d.H, d.nc, d.B), kIntraThreads, smem, st>>>(mapC, mapB, mapX, mapDY, a);
        trace_end(st);
        if ((e = cudaGetLastError())) return e;
    }
    {
        const size_t smem = InterSmem(d.K, d.N).total + 1024;
        cudaFuncSetAttribute(tc_bwd_inter, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        trace_begin("bwd_inter_tc", st);
        tc_bwd_inter<<<dim3(d.H * (d.P / TPS), d.nc, d.B), kThreads, smem, st>>>(mapC, mapB, mapS, mapD, a);
        trace_end(st);
        if ((e = cudaGetLastError())) return e;
    }
    {
        const size_t smem = DcdbSmem(d.K, d.N).total + 1024;
        cudaFuncSetAttribute(tc_bwd_dcdb, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        trace_begin("bwd_dcdb_tc", st);
        tc_bwd_dcdb<<<dim3(d.H / a.hg, d.nc, d.B), kThreads, smem, st>>>(mapS, mapD, mapB, mapC, a);
        trace_end(st);
        if ((e = cudaGetLastError())) return e;
    }
    trace_begin("bwd_final_tc", st);
    tc_bwd_final<<<dim3(d.nc, d.H, d.B), kThreads, 0, st>>>(a);
    trace_end(st);
    if ((e = cudaGetLastError())) return e;
    if (ngn > 0) {
        const unsigned blocks = unsigned(std::min<size_t>((ngn + 255) / 256, 4096));
        trace_begin("f32_to_bf16", st);
        f32_to_bf16_tc<<<blocks, 256, 0, st>>>(ws.dB_acc, (bf16 *)p.dB, ngn);
        f32_to_bf16_tc<<<blocks, 256, 0, st>>>(ws.dC_acc, (bf16 *)p.dC, ngn);
        trace_end(st);
        e = cudaGetLastError();
    }
    return e;
}

}  // namespace frac
