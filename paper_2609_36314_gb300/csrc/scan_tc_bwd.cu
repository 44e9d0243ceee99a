// Tensor-core backward of the chunked Frac scan (bf16 inputs, chunk 128, headdim 64).
//
// With S_in / dS_out the per-chunk states of the forward and reverse state passes, every
// gradient of a chunk follows from chunk-local quantities (the adjoint of the recurrence of
// Sec. 3.2, written in the chunked order of App. F).  With G[t,k] = C_t.B_k, H[t,k] = dy_t.x_k,
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
//   tc_bwd_state  (b, c, group of heads): per (head, mode) Z = C S_in^T and U = B dS_out^T,
//                 dx += (s o B) dS_out^T, dC += (f o dY) S_in and dB += (s o X) dS_out on the
//                 tensor cores (dC, dB summed over the group's heads in TMEM); epilogue to
//                 dw_read, dkappa, the a, b terms and <dS_out, S_in>; the head-summed intra term.
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
    float *coef;  // per position: f, s, u, exp(-E/tau) for every mode [B, L, H, 4, K]
    const float *ek;  // per position: {E hi, E lo, 0, 0, kappa[K]} [B, L, H, tc_ek_width(K)]
    bf16 *dx, *dwr, *dww;
    float *ddt, *dalpha, *dlam, *dD;
    float *inter_acc, *dtau;  // both null unless the timescale gradient is wanted
    int *err;
    int hg;      // heads per dC/dB group
    int pf_sms;  // SMs of the device: CTAs of the persistent intra kernel
};

__device__ __forceinline__ void store_bf16x8(unsigned char *p, const float *v) {
    *reinterpret_cast<uint4 *>(p) = make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                                               pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7]));
}

__device__ __forceinline__ unsigned char *align1024(unsigned char *p) {
    return reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

// ============================================================================= intra
constexpr int kIntraThreads = 256;  // two groups of four warps share the 128 TMEM lanes
constexpr int kIntraLaunch = kIntraThreads + 32;  // a ninth warp issues the MMAs and TMA loads

struct IntraSmem {
    int rcb, x, dy, mg, xx, total;
    __host__ __device__ IntraSmem() {
        rcb = ((TQ * XS * 4 + 1023) / 1024) * 1024;  // C + B tiles (<= 64 KB), then fp32 G*H
        x = 16384;                 // x chunk [128 t][64 p], 128-byte swizzle
        dy = 16384;                // dy chunk
        mg = 2 * 16384;            // Gamma o G, [t][k] K-major
        xx = TQ * XS * 4;          // fp32 Gamma' G H, then its row prefix sums
        total = rcb + x + dy + mg + xx + 4 * TQ * KMAX * 4 + TQ * 8 + 64 * 4 + 64 + 64 + 64 +
                12 * TQ * 4 + TQ * 16 +  // + the next item's per-position inputs
                3 * 64 * KMAX * 4 +      // + the 16-anchor factors V16, V16 / tau, U16
                KMAX * 4;                // + the next item's time constants
    }
};

__global__ void __launch_bounds__(kIntraLaunch, 1)
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
    float *Vs = part + TQ * KMAX;                            // [128][KMAX] kappa exp(-(E_a - E_k)/tau)
    float2 *E_s = reinterpret_cast<float2 *>(Vs + TQ * KMAX);  // hi / lo pairs
    float *l2t = reinterpret_cast<float *>(E_s + TQ);
    float *inv_tau_s = l2t + 32;  // 1 / tau per mode
    float2 *wsum = reinterpret_cast<float2 *>(inv_tau_s + 32);
    // bars: 0 C, B, x of the item loaded | 1 G, H, Gamma MMAs done | 2 dx MMA done | 3 dy loaded |
    //       the compute threads (256 arrive): 4 U, V operands written | 5 Gamma o G tile written
    //       and G read | 6 C / B region and x tile read | 7 dx read from TMEM
    uint64_t *bars = reinterpret_cast<uint64_t *>(wsum + 8);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bars + 8);
    volatile int *abort_s = reinterpret_cast<volatile int *>(tslot + 1);
    // the next item's per-position inputs, staged by cp.async: {E hi, E lo, 0, 0, kappa[K]} from
    // tc_coef [128][12] floats and w_read [128] x 16 bytes
    float *pf_e = reinterpret_cast<float *>(tslot + 4);
    unsigned char *pf_w = reinterpret_cast<unsigned char *>(pf_e + 12 * TQ);
    // the lower-left 16 x 16 quarter of each diagonal 32 x 32 block, factored through E at the
    // block's 16th position: V16 [64 (block, k mod 16)][KMAX] = kappa exp(-(E_a16 - E_k)/tau),
    // V16 / tau, and U16 [64 (block, t mod 16 of the lower half)][KMAX] = w_read exp(-(E_t - E_a16)/tau)
    float *V16s = reinterpret_cast<float *>(pf_w + TQ * 16);
    float *V16ps = V16s + 64 * KMAX;
    float *U16s = V16ps + 64 * KMAX;
    float *pf_tau = U16s + 64 * KMAX;  // the next item's mode time constants [KMAX] (staged)

    const int tid = threadIdx.x, grp = tid >> 7, t = tid & 127, w4 = (tid >> 5) & 3;
    // persistent: items (h, c, b) in launch order, gridDim.x CTAs apart
    const int nitems = d.H * d.nc * d.B;
    auto item_hcb = [&](int item) { return make_int3(item % d.H, (item / d.H) % d.nc, item / (d.H * d.nc)); };
    // the issuing thread: the item's C, B and x tiles (bars[0]) / its dy tile (bars[3]) by TMA
    auto load_cbx = [&](int item) {
        const int3 hcb = item_hcb(item);
        const int h_ = hcb.x, c_ = hcb.y, b_ = hcb.z;
        const int g_ = h_ / (d.H / d.G);
        mbar_arrive_expect_tx(&bars[0], uint32_t(2 * (N / 64) * 16384 + 16384));
        for (int jb = 0; jb < N / 64; ++jb) {
            tma_load_3d(sC + jb * 16384, &mapC, &bars[0], g_ * N + 64 * jb, c_ * TQ, b_);
            tma_load_3d(sB + jb * 16384, &mapB, &bars[0], g_ * N + 64 * jb, c_ * TQ, b_);
        }
        tma_load_3d(sX, &mapX, &bars[0], h_ * P, c_ * TQ, b_);
    };
    auto load_dy = [&](int item) {
        const int3 hcb = item_hcb(item);
        const int h_ = hcb.x, c_ = hcb.y, b_ = hcb.z;
        mbar_arrive_expect_tx(&bars[3], 16384u);
        tma_load_3d(sDY, &mapDY, &bars[3], h_ * P, c_ * TQ, b_);
    };
    // its position's {E, kappa} and w_read of the item into the staging area (group 0: {E, kappa},
    // group 1: w_read)
    const int ekw = tc_ek_width(K);
    auto stage_inputs = [&](int item) {
        const int3 hcb = item_hcb(item);
        const int h_ = hcb.x, c_ = hcb.y, b_ = hcb.z;
        // rows past the end of a ragged chunk take the last row's E (zero token rates there)
        const int tt = min(c_ * TQ + t, d.L - 1);
        const size_t i = blh(d, b_, tt, h_);
        if (grp == 0) {
            for (int q = 0; q < 1 + K / 4; ++q) cp_async_bytes(pf_e + t * 12 + 4 * q, a.ek + i * ekw + 4 * q, 16);
            if (t < K / 4) cp_async_bytes(pf_tau + 4 * t, a.tau + h_ * K + 4 * t, 16);
        } else if (c_ * TQ + t < d.L) {
            cp_async_bytes(pf_w + t * 16, a.wr + i * K, 2 * K);
        }
        cp_async_commit();
    };

    if (tid == 0) {
        for (int i = 0; i < 4; ++i) mbar_init(&bars[i], 1);
        for (int i = 4; i < 8; ++i) mbar_init(&bars[i], kIntraThreads);
        *abort_s = 0;
        fence_barrier_init();
    }
    if (tid < 32) tmem_alloc_once(tslot, 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    const uint32_t lane_base = tmem + (uint32_t(w4 * 32) << 16);
    // TMEM: G, H, the factored Gamma and Gamma' blocks; dx_intra replaces G after the row pass
    const uint32_t colG = 0, colH = 128, colGam = 256, colGamP = 384, colX = 0;
    if (int(blockIdx.x) < nitems) {
        if (tid == kIntraThreads) {
            load_cbx(blockIdx.x);
            load_dy(blockIdx.x);
        }
        if (tid < kIntraThreads) stage_inputs(blockIdx.x);
    }

    if (tid == kIntraThreads) {
        // the issuing thread: an item's G = C B^T once its C and B tiles are in (and the previous
        // item's dx has left TMEM), H = dY X^T once dY is in, the Gamma blocks once the threads
        // have written U and V, dx_intra once they have written the Gamma o G tile; then the
        // next item's dy (its tile free once dx_intra is done) and C, B, x (once read)
        int kk = 0;
        for (int item = blockIdx.x; item < nitems && !*abort_s; item += gridDim.x, ++kk) {
            const int ph = kk & 1;
            unsigned char *sU = reinterpret_cast<unsigned char *>(XX), *sV = sU + 16384, *sVp = sV + 4096;
            const uint32_t idG = idesc_bf16(128, 128, false, false);
            if ((kk > 0 && !mbar_wait(&bars[7], (kk - 1) & 1)) || !mbar_wait(&bars[0], ph)) {
                *abort_s = 1;
                break;
            }
            tc_fence_after();
            for (int ks = 0; ks < N / 16; ++ks) {
                const uint32_t koff = (ks / 4) * 16384 + (ks % 4) * 32;
                mma_bf16(tmem + colG, desc_sw128(smem_u32(sC) + koff, 16, 1024),
                         desc_sw128(smem_u32(sB) + koff, 16, 1024), idG, ks > 0);
            }
            if (!mbar_wait(&bars[3], ph)) {
                *abort_s = 1;
                break;
            }
            tc_fence_after();
            for (int ks = 0; ks < BP / 16; ++ks)  // H = dY X^T, K = p
                mma_bf16(tmem + colH, desc_sw128(smem_u32(sDY) + ks * 32, 16, 1024),
                         desc_sw128(smem_u32(sX) + ks * 32, 16, 1024), idG, ks > 0);
            if (!mbar_wait(&bars[4], ph)) {
                *abort_s = 1;
                break;
            }
            tc_fence_after();
            const uint32_t idT = idesc_tf32(128, 32);
            for (int J = 0; J < 4; ++J) {
                mma_tf32(tmem + colGam + 32 * J, desc_sw128(smem_u32(sU) + 32 * J, 16, 1024),
                         desc_sw128(smem_u32(sV) + 32 * J, 16, 1024), idT, 0);
                mma_tf32(tmem + colGamP + 32 * J, desc_sw128(smem_u32(sU) + 32 * J, 16, 1024),
                         desc_sw128(smem_u32(sVp) + 32 * J, 16, 1024), idT, 0);
            }
            mma_commit(&bars[1]);
            if (!mbar_wait(&bars[5], ph)) {
                *abort_s = 1;
                break;
            }
            tc_fence_after();
            const uint32_t idX = idesc_bf16(128, BP, true, true);  // dx_intra = (Gamma o G)^T dY
            for (int ks = 0; ks < TQ / 16; ++ks)
                mma_bf16(tmem + colX, desc_sw128(smem_u32(sMG) + ks * 2048, 16384, 1024),
                         desc_sw128(smem_u32(sDY) + ks * 2048, 16384, 1024), idX, ks > 0);
            mma_commit(&bars[2]);
            if (item + int(gridDim.x) < nitems) {
                if (!mbar_wait(&bars[2], ph)) {
                    *abort_s = 1;
                    break;
                }
                load_dy(item + gridDim.x);
                if (!mbar_wait(&bars[6], ph)) {
                    *abort_s = 1;
                    break;
                }
                load_cbx(item + gridDim.x);
            }
        }
    }

    int kk_item = 0;
    for (int item = blockIdx.x; item < nitems && tid < kIntraThreads; item += gridDim.x, ++kk_item) {
        const int ph = kk_item & 1;  // parity of this item's phase on every barrier
        const int3 hcb = item_hcb(item);
        const int h = hcb.x, c = hcb.y, b = hcb.z;
        const int g = h / (d.H / d.G);
        const int c0 = c * TQ, n = min(TQ, d.L - c0);
        // per-position inputs of row t from the staging area, and the mode time constants
        cp_async_wait_all();
        sync_first256();
        float wr_t[KMAX], kap_t[KMAX];
        float2 Et2 = make_float2(0.f, 0.f);  // in-chunk cumulative log-decay (hi, lo)
#pragma unroll
        for (int m = 0; m < KMAX; ++m) wr_t[m] = kap_t[m] = 0.f;
        {
            const float4 e4 = *reinterpret_cast<const float4 *>(pf_e + t * 12);
            Et2 = make_float2(e4.x, e4.y);
        }
        if (t < n) {
#pragma unroll
            for (int m = 0; m < KMAX; ++m)
                if (m < K) kap_t[m] = pf_e[t * 12 + 4 + m];
            load_weights(reinterpret_cast<const bf16 *>(pf_w + t * 16), K, wr_t);
        }
        if (tid < K) {
            const float tv = pf_tau[tid];
            inv_tau_s[tid] = 1.f / tv;
            l2t[tid] = kLog2e / tv;
        }
        sync_first256();  // the staging area is free again: the next item's inputs
        if (item + int(gridDim.x) < nitems) stage_inputs(item + gridDim.x);
        if (grp == 0) E_s[t] = Et2;
        float l2r[KMAX];  // log2(e) / tau per mode, in registers (the table tid < K wrote)
#pragma unroll
        for (int m = 0; m < KMAX; ++m) l2r[m] = m < K ? l2t[m] : 0.f;
        if (grp == 0) {
#pragma unroll
            for (int q = 0; q < KMAX / 4; ++q) {
                *reinterpret_cast<float4 *>(wr_s + t * KMAX + 4 * q) =
                    make_float4(wr_t[4 * q], wr_t[4 * q + 1], wr_t[4 * q + 2], wr_t[4 * q + 3]);
                *reinterpret_cast<float4 *>(kap_s + t * KMAX + 4 * q) =
                    make_float4(kap_t[4 * q], kap_t[4 * q + 1], kap_t[4 * q + 2], kap_t[4 * q + 3]);
            }
        }
        tc_fence_before();
        sync_first256();
        tc_fence_after();
        // ---- Gamma below the diagonal 32 x 32 blocks, factored through the log-decay E_a at the end
        // of the column block J (as in the forward output kernel): Gamma[t, k in J] =
        // sum_m U_J[t, m] V[k, m] and Gamma'[t, k] = sum_m U_J[t, m] V[k, m] / tau_m, tf32 products.
        // Operand tiles (128-byte swizzled) in the XX region: U [128 t][4 J x 8 m],
        // V and V / tau [32 k mod 32][4 J x 8 m]; V also as fp32 in Vs for the intra dw_read.
        unsigned char *sU = reinterpret_cast<unsigned char *>(XX), *sV = sU + 16384, *sVp = sV + 4096;
        if (grp == 0) {
            const int I = t >> 5;
            unsigned char *row = sU + t * 128;
#pragma unroll
            for (int J = 0; J < 4; ++J) {
                uint32_t u[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
                if (J < I) {  // blocks at or above the row's own are zero (I is uniform in a warp)
                    const float dE = diff_f2(Et2, E_s[32 * J + 31]);
#pragma unroll
                    for (int m = 0; m < KMAX; ++m)
                        u[m] = (m < K && t < n) ? to_tf32(wr_t[m] * ex2_approx(-dE * l2r[m])) : 0u;
                }
                *reinterpret_cast<uint4 *>(row + (((2 * J) ^ (t & 7)) * 16)) = make_uint4(u[0], u[1], u[2], u[3]);
                *reinterpret_cast<uint4 *>(row + (((2 * J + 1) ^ (t & 7)) * 16)) = make_uint4(u[4], u[5], u[6], u[7]);
            }
            if ((t & 31) >= 16) {  // lower half of its block: U16 against the anchor 32 I + 15
                const float dE = diff_f2(Et2, E_s[32 * I + 15]);
#pragma unroll
                for (int m = 0; m < KMAX; ++m)
                    U16s[(16 * I + (t & 15)) * KMAX + m] = (m < K && t < n) ? wr_t[m] * ex2_approx(-dE * l2r[m]) : 0.f;
            }
        } else {
            const int J = t >> 5, r = t & 31;
            const float dE = diff_f2(E_s[32 * J + 31], Et2);
            uint32_t v[8], vp[8];
#pragma unroll
            for (int m = 0; m < KMAX; ++m) {
                const float vv = m < K ? kap_t[m] * ex2_approx(-dE * l2r[m]) : 0.f;
                Vs[t * KMAX + m] = vv;
                v[m] = to_tf32(vv);
                vp[m] = m < K ? to_tf32(vv * inv_tau_s[m]) : 0u;
            }
            unsigned char *row = sV + r * 128, *rowp = sVp + r * 128;
            *reinterpret_cast<uint4 *>(row + (((2 * J) ^ (r & 7)) * 16)) = make_uint4(v[0], v[1], v[2], v[3]);
            *reinterpret_cast<uint4 *>(row + (((2 * J + 1) ^ (r & 7)) * 16)) = make_uint4(v[4], v[5], v[6], v[7]);
            *reinterpret_cast<uint4 *>(rowp + (((2 * J) ^ (r & 7)) * 16)) = make_uint4(vp[0], vp[1], vp[2], vp[3]);
            *reinterpret_cast<uint4 *>(rowp + (((2 * J + 1) ^ (r & 7)) * 16)) = make_uint4(vp[4], vp[5], vp[6], vp[7]);
            if (r < 16) {  // left half of its block: V16 against the anchor 32 J + 15
                const float dE16 = diff_f2(E_s[32 * J + 15], Et2);
#pragma unroll
                for (int m = 0; m < KMAX; ++m) {
                    const float v16 = m < K ? kap_t[m] * ex2_approx(-dE16 * l2r[m]) : 0.f;
                    V16s[(16 * J + r) * KMAX + m] = v16;
                    V16ps[(16 * J + r) * KMAX + m] = m < K ? v16 * inv_tau_s[m] : 0.f;
                }
            }
        }
        fence_async_smem();
        mbar_arrive(&bars[4]);  // U, V written: the Gamma MMAs may go
        if (!*abort_s && !mbar_wait(&bars[1], ph)) *abort_s = 1;
        sync_first256();
        tc_fence_after();
        // U rows as fp32 [128 t][4 J][8 m] in the x tile (free now) for the column pass, before the
        // row pass overwrites the operand tiles with XX.  Group g copies four of the eight 16-byte
        // pieces of row t: piece c = (a t) xor (4 g + c4), with a t the product by the generator of
        // GF(8) (x^3 + x + 1).  For eight neighbouring threads both the destination pieces c and the
        // swizzled source pieces c xor t = ((a + 1) t) xor (4 g + c4) are all different, so neither
        // the reads nor the writes meet a bank conflict
        float *Ufp = reinterpret_cast<float *>(sX);
        {
            const unsigned char *row = sU + t * 128;
            const int t7 = t & 7, at = ((t7 << 1) & 7) ^ ((t7 >> 2) * 3);
#pragma unroll
            for (int c4 = 0; c4 < 4; ++c4) {
                const int c8 = at ^ (4 * grp + c4);
                *reinterpret_cast<uint4 *>(Ufp + t * 32 + 4 * c8) =
                    *reinterpret_cast<const uint4 *>(row + ((c8 ^ (t & 7)) * 16));
            }
        }
        sync_first256();
        // ---- row pass (row t = this warp's row block I; group 0 takes column blocks 0, 1, group 1
        // blocks 2, 3): Gamma o G tile, Gamma o H summed over heads in L2, Gamma' G H and G H tiles,
        // intra dw_read.  Blocks below the diagonal take the factored Gamma from TMEM, the diagonal
        // block sums its pairs k <= t directly, blocks above it are zero.
        float dwr_i[KMAX];
#pragma unroll
        for (int m = 0; m < KMAX; ++m) dwr_i[m] = 0.f;
        if (!*abort_s) {
            const int I = t >> 5;
            float *mh_row = a.mh_total + (((size_t(b) * d.nc + c) * d.G + g) * TQ + t) * TQ;
            // 8-column work items (column block kc, eighth q8) alternate between the two groups, so
            // that both take half of every block, the diagonal one included; loops stay rolled (the
            // fully unrolled pass overflowed the instruction cache)
            float acc[KMAX];
#pragma unroll
            for (int m = 0; m < KMAX; ++m) acc[m] = 0.f;
            // the Gamma o G tile (bf16) and the head-summed Gamma o H for 8 columns from k0
            auto store_item = [&](const float *gv, const float *hv, unsigned char *mg, int k0) {
                *reinterpret_cast<uint4 *>(mg) = make_uint4(pack_bf16x2(gv[0], gv[1]), pack_bf16x2(gv[2], gv[3]),
                                                            pack_bf16x2(gv[4], gv[5]), pack_bf16x2(gv[6], gv[7]));
                if (t < n && k0 <= t) {
                    atomicAdd(reinterpret_cast<float4 *>(mh_row + k0), make_float4(hv[0], hv[1], hv[2], hv[3]));
                    if (k0 + 4 <= t)
                        atomicAdd(reinterpret_cast<float4 *>(mh_row + k0 + 4), make_float4(hv[4], hv[5], hv[6], hv[7]));
                }
            };
            // the diagonal block I in 16 x 16 quarters: the two on the diagonal sum their pairs
            // k <= t directly, the lower-left one is factored through E at 32 I + 15 (U16 V16,
            // both factors <= 1), the upper-right one is zero.  Each step gives every lane 8
            // columns: the direct step the lane's own diagonal quarter (upper rows: left half,
            // lower rows: right half), the other step the rest (lower rows: factored, upper: zero).
            auto diag_item = [&](int kc, bool dstep) {
                const bool upper = (t & 31) < 16;
                const int q8l = (dstep == upper) ? grp : grp + 2;  // this lane's 8 columns
                const int k0 = 32 * kc + 8 * q8l;
                unsigned char *mg = sMG + (kc >> 1) * 16384 + t * 128 + ((((kc & 1) * 4 + q8l) ^ (t & 7)) * 16);
                float gv[8], hv[8];
                {
                    float ga[8], gb[8], ha[8], hb[8];
                    tmem_ld8(lane_base + colG + 32 * kc + 8 * grp, ga);
                    tmem_ld8(lane_base + colG + 32 * kc + 8 * grp + 16, gb);
                    tmem_ld8(lane_base + colH + 32 * kc + 8 * grp, ha);
                    tmem_ld8(lane_base + colH + 32 * kc + 8 * grp + 16, hb);
                    tmem_ld_wait();
                    const bool lo = q8l == grp;
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) {
                        gv[kk] = lo ? ga[kk] : gb[kk];
                        hv[kk] = lo ? ha[kk] : hb[kk];
                    }
                }
                if (dstep) {
                    // branch-free over the eight columns: a pair above the diagonal (k > t) runs
                    // the same arithmetic with its decay exponent clamped to zero (every factor
                    // finite) and a zero G H, and its Gamma is masked to zero
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) {
                        const int k = k0 + kk;
                        const bool valid = k <= t && t < n;
                        const float dE = fmaxf(diff_f2(Et2, E_s[k]), 0.f);
                        const float gh = valid ? gv[kk] * hv[kk] : 0.f;
                        const float4 ka = *reinterpret_cast<const float4 *>(kap_s + k * KMAX);
                        const float4 kb = *reinterpret_cast<const float4 *>(kap_s + k * KMAX + 4);
                        const float kpv[8] = {ka.x, ka.y, ka.z, ka.w, kb.x, kb.y, kb.z, kb.w};
                        // modes in packed float32 pairs (K is even)
                        float2 gam2 = make_float2(0.f, 0.f), gamt2 = make_float2(0.f, 0.f);
                        const float2 ndE = make_float2(-dE, -dE), gh2 = make_float2(gh, gh);
#pragma unroll
                        for (int m = 0; m < KMAX; m += 2) {
                            if (m < K) {
                                const float2 l2 = make_float2(l2r[m], l2r[m + 1]);
                                const float2 x2 = __fmul2_rn(ndE, l2);
                                const float2 kpW = __fmul2_rn(make_float2(kpv[m], kpv[m + 1]),
                                                              make_float2(ex2_approx(x2.x), ex2_approx(x2.y)));
                                const float2 aa = __fmul2_rn(make_float2(wr_t[m], wr_t[m + 1]), kpW);
                                gam2 = __fadd2_rn(gam2, aa);
                                gamt2 = __ffma2_rn(aa, l2, gamt2);  // times log2(e) / tau
                                const float2 dw = __ffma2_rn(kpW, gh2, make_float2(dwr_i[m], dwr_i[m + 1]));
                                dwr_i[m] = dw.x;
                                dwr_i[m + 1] = dw.y;
                            }
                        }
                        float gam = gam2.x + gam2.y;
                        const float gamt = gamt2.x + gamt2.y;
                        gam = valid ? gam : 0.f;
                        gv[kk] = gam * gv[kk];
                        hv[kk] = gam * hv[kk];
                        XX[t * XS + k] = gamt * (1.f / kLog2e) * gh;
                        GHs[t * XS + k] = gh;
                    }
                } else if (!upper) {
                    const float *u16 = U16s + (16 * kc + (t & 15)) * KMAX;
                    const float4 ua = *reinterpret_cast<const float4 *>(u16), ub = *reinterpret_cast<const float4 *>(u16 + 4);
                    const float uu[8] = {ua.x, ua.y, ua.z, ua.w, ub.x, ub.y, ub.z, ub.w};
                    float a16[KMAX];
#pragma unroll
                    for (int m = 0; m < KMAX; ++m) a16[m] = 0.f;
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) {
                        const int k = k0 + kk, j16 = 16 * kc + (k & 15);
                        const float gh = t < n ? gv[kk] * hv[kk] : 0.f;
                        const float4 v0 = *reinterpret_cast<const float4 *>(V16s + j16 * KMAX);
                        const float4 v1 = *reinterpret_cast<const float4 *>(V16s + j16 * KMAX + 4);
                        const float4 p0 = *reinterpret_cast<const float4 *>(V16ps + j16 * KMAX);
                        const float4 p1 = *reinterpret_cast<const float4 *>(V16ps + j16 * KMAX + 4);
                        const float vk[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
                        const float pk[8] = {p0.x, p0.y, p0.z, p0.w, p1.x, p1.y, p1.z, p1.w};
                        float2 g2 = make_float2(0.f, 0.f), gp2 = make_float2(0.f, 0.f);
                        const float2 gh2 = make_float2(gh, gh);
#pragma unroll
                        for (int m = 0; m < KMAX; m += 2) {  // packed float32 pairs of modes
                            const float2 u2 = make_float2(uu[m], uu[m + 1]), v2 = make_float2(vk[m], vk[m + 1]);
                            g2 = __ffma2_rn(u2, v2, g2);
                            gp2 = __ffma2_rn(u2, make_float2(pk[m], pk[m + 1]), gp2);
                            const float2 a2 = __ffma2_rn(v2, gh2, make_float2(a16[m], a16[m + 1]));
                            a16[m] = a2.x;
                            a16[m + 1] = a2.y;
                        }
                        const float gam = g2.x + g2.y, gamp = gp2.x + gp2.y;
                        XX[t * XS + k] = gamp * gh;
                        GHs[t * XS + k] = gh;
                        gv[kk] *= gam;
                        hv[kk] *= gam;
                    }
                    // intra dw_read of these pairs: exp(-(E_t - E_a16)/tau) sum_k V16[k] G H
                    const float dE = diff_f2(Et2, E_s[32 * kc + 15]);
#pragma unroll
                    for (int m = 0; m < KMAX; ++m)
                        if (m < K) dwr_i[m] = fmaf(ex2_approx(-dE * l2r[m]), a16[m], dwr_i[m]);
                } else {
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) {
                        gv[kk] = hv[kk] = 0.f;
                        XX[t * XS + k0 + kk] = 0.f;
                    }
                }
                store_item(gv, hv, mg, k0);
            };
#pragma unroll 1
            for (int it = grp; it < 16; it += 2) {
                const int kc = it >> 2, q8 = it & 3;
                if (kc == I) {
                    diag_item(kc, q8 == grp);
                    continue;
                }
                const int k0 = 32 * kc + 8 * q8;
                unsigned char *mg = sMG + (kc >> 1) * 16384 + t * 128 + ((((kc & 1) * 4 + q8) ^ (t & 7)) * 16);
                if (kc > I) {
                    *reinterpret_cast<uint4 *>(mg) = make_uint4(0, 0, 0, 0);
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) XX[t * XS + k0 + kk] = 0.f;  // rows are 129 floats apart
                    continue;
                }
                float gv[8], hv[8];
                tmem_ld8(lane_base + colG + k0, gv);
                tmem_ld8(lane_base + colH + k0, hv);
                {
                    float gm[8], gp[8];
                    tmem_ld8(lane_base + colGam + k0, gm);
                    tmem_ld8(lane_base + colGamP + k0, gp);
                    tmem_ld_wait();
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) {
                        const int k = k0 + kk;
                        const float gh = gv[kk] * hv[kk];
                        XX[t * XS + k] = gp[kk] * gh;
                        GHs[t * XS + k] = gh;
                        const float4 v0 = *reinterpret_cast<const float4 *>(Vs + k * KMAX);
                        const float4 v1 = *reinterpret_cast<const float4 *>(Vs + k * KMAX + 4);
                        const float vk[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
                        const float2 gh2 = make_float2(gh, gh);
#pragma unroll
                        for (int m = 0; m < KMAX; m += 2) {
                            const float2 s2 = __ffma2_rn(make_float2(vk[m], vk[m + 1]), gh2, make_float2(acc[m], acc[m + 1]));
                            acc[m] = s2.x;
                            acc[m + 1] = s2.y;
                        }
                        gv[kk] *= gm[kk];  // Gamma o G
                        hv[kk] *= gm[kk];  // Gamma o H
                    }
                }
                store_item(gv, hv, mg, k0);
                if (kc < I && q8 >= 2) {  // this thread's last item of the factored block kc
                    const float dE = diff_f2(Et2, E_s[32 * kc + 31]);
#pragma unroll
                    for (int m = 0; m < KMAX; ++m) {
                        if (m < K) dwr_i[m] = fmaf(ex2_approx(-dE * l2r[m]), acc[m], dwr_i[m]);
                        acc[m] = 0.f;
                    }
                }
            }
            if (grp == 1) {
#pragma unroll
                for (int m = 0; m < KMAX; ++m) part[t * KMAX + m] = dwr_i[m];
            }
        }
        fence_async_smem();
        tc_fence_before();
        mbar_arrive(&bars[5]);  // the Gamma o G tile written, G read: dx_intra may go
        sync_first256();
        tc_fence_after();
        if (!*abort_s && grp == 0 && t < n) {
            float4 *o = reinterpret_cast<float4 *>(a.dwr_acc + blh(d, b, c0 + t, h) * K);
#pragma unroll
            for (int q = 0; q < KMAX / 4; ++q) {
                if (4 * q < K) {
                    const float4 pq = *reinterpret_cast<const float4 *>(part + t * KMAX + 4 * q);
                    o[q] = make_float4(dwr_i[4 * q] + pq.x, dwr_i[4 * q + 1] + pq.y, dwr_i[4 * q + 2] + pq.z,
                                       dwr_i[4 * q + 3] + pq.w);
                }
            }
        }
        sync_first256();  // part[] is reused below
        // ---- column pass (group g takes the rows of parity g of column k): intra dkappa.  Rows of
        // later blocks use the factored form exp(-(E_a - E_k)/tau) sum_t U_J[t, m] G H[t, k]; rows of
        // the diagonal block (t >= k) sum directly.  Column block J has 128 - 32 J rows, so group 1's
        // warp w takes block 3 - w: every SM sub-partition gets blocks J and 3 - J.
        const int kcol = grp == 0 ? t : (((3 - (t >> 5)) << 5) | (t & 31));
        float dk[KMAX];
#pragma unroll
        for (int m = 0; m < KMAX; ++m) dk[m] = 0.f;
        if (!*abort_s) {
            const int k = kcol, J = k >> 5;
            const float2 Ek = E_s[k];
            float dk2[KMAX];
#pragma unroll
            for (int m = 0; m < KMAX; ++m) dk2[m] = 0.f;
            // direct rows: k's own 16-row quarter of the diagonal block (t >= k), rows of this
            // group's parity.  Every lane walks the eight rows of its quarter of that parity (the
            // same rows in a half-warp: broadcast reads); rows above the column (t < k) or past
            // the chunk run with a zero decay exponent and a zero G H
            const bool left = (k & 31) < 16;
            const int qs = 32 * J + (left ? 0 : 16) + grp;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int tt = qs + 2 * i;
                const bool valid = tt >= k && tt < n;
                const float dE = fmaxf(diff_f2(E_s[tt], Ek), 0.f);
                const float gh = valid ? GHs[tt * XS + k] : 0.f;
                const float4 w0 = *reinterpret_cast<const float4 *>(wr_s + tt * KMAX);
                const float4 w1 = *reinterpret_cast<const float4 *>(wr_s + tt * KMAX + 4);
                const float wv[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
                const float2 ndE = make_float2(-dE, -dE), gh2 = make_float2(gh, gh);
#pragma unroll
                for (int m = 0; m < KMAX; m += 2) {  // packed float32 pairs of modes (K is even)
                    if (m < K) {
                        const float2 x2 = __fmul2_rn(ndE, make_float2(l2r[m], l2r[m + 1]));
                        const float2 v = __fmul2_rn(make_float2(wv[m], wv[m + 1]),
                                                    make_float2(ex2_approx(x2.x), ex2_approx(x2.y)));
                        float *dst = (i & 1) ? dk2 : dk;
                        const float2 r2 = __ffma2_rn(v, gh2, make_float2(dst[m], dst[m + 1]));
                        dst[m] = r2.x;
                        dst[m + 1] = r2.y;
                    }
                }
            }
            if (left) {  // lower half of the diagonal block: factored through E at 32 J + 15
                float a16[KMAX];
#pragma unroll
                for (int m = 0; m < KMAX; ++m) a16[m] = 0.f;
                const int lend = min(n, 32 * J + 32);
                for (int tt = 32 * J + 16 + grp; tt < lend; tt += 2) {
                    const float gh = GHs[tt * XS + k];
                    const float *u16 = U16s + (16 * J + (tt & 15)) * KMAX;
                    const float4 u0 = *reinterpret_cast<const float4 *>(u16);
                    const float4 u1 = *reinterpret_cast<const float4 *>(u16 + 4);
                    const float uu[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
                    const float2 gh2 = make_float2(gh, gh);
#pragma unroll
                    for (int m = 0; m < KMAX; m += 2) {  // packed float32 pairs of modes
                        const float2 a2 = __ffma2_rn(make_float2(uu[m], uu[m + 1]), gh2, make_float2(a16[m], a16[m + 1]));
                        a16[m] = a2.x;
                        a16[m + 1] = a2.y;
                    }
                }
                const float dE16 = diff_f2(E_s[32 * J + 15], Ek);
#pragma unroll
                for (int m = 0; m < KMAX; ++m)
                    if (m < K) dk2[m] = fmaf(ex2_approx(-dE16 * l2r[m]), a16[m], dk2[m]);
            }
            float s0[KMAX], s1[KMAX];
#pragma unroll
            for (int m = 0; m < KMAX; ++m) s0[m] = s1[m] = 0.f;
            for (int tt0 = 32 * J + 32 + grp; tt0 < n; tt0 += 8) {
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int tt = tt0 + 2 * u;
                    if (tt < n) {
                        const float gh = GHs[tt * XS + k];
                        const float4 u0 = *reinterpret_cast<const float4 *>(Ufp + tt * 32 + 8 * J);
                        const float4 u1 = *reinterpret_cast<const float4 *>(Ufp + tt * 32 + 8 * J + 4);
                        const float uu[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
                        const float2 gh2 = make_float2(gh, gh);
                        float *sd = (u & 1) ? s1 : s0;
#pragma unroll
                        for (int m = 0; m < KMAX; m += 2) {  // packed float32 pairs of modes
                            const float2 r2 = __ffma2_rn(make_float2(uu[m], uu[m + 1]), gh2, make_float2(sd[m], sd[m + 1]));
                            sd[m] = r2.x;
                            sd[m + 1] = r2.y;
                        }
                    }
                }
            }
            const float dEa = diff_f2(E_s[32 * J + 31], Ek);
#pragma unroll
            for (int m = 0; m < KMAX; ++m) {
                dk[m] += dk2[m];
                if (m < K) dk[m] = fmaf(ex2_approx(-dEa * l2r[m]), s0[m] + s1[m], dk[m]);
            }
            if (grp == 1) {
#pragma unroll
                for (int m = 0; m < KMAX; ++m) part[k * KMAX + m] = dk[m];
            }
        }
        // exclusive row prefix of XX (row t): group 0 over j in [0, 64) (its total in xtot), group 1
        // over [64, 128) starting from 0; the column sums below add the suffix sum of xtot for the
        // columns j >= 64
        float *xtot = Vs;  // [128], free after the row pass
        if (!*abort_s) {
            float run = 0.f;
#pragma unroll 2
            for (int j0 = 64 * grp; j0 < 64 * grp + 64; j0 += 8) {
                float v[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) v[i] = XX[t * XS + j0 + i];
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    XX[t * XS + j0 + i] = run;
                    run += v[i];
                }
            }
            if (grp == 0) xtot[t] = run;
        }
        sync_first256();
        // rect[j] = sum_{t' >= j} sum_{k < j} X[t', k]: column j's suffix sum of the row prefixes,
        // rows of parity g in group g (column kcol, the column pass's balanced assignment)
        float *rpart = Vs + TQ;  // [128] group 1's partial rect
        float sr = 0.f;
        if (!*abort_s) {
            const int j = kcol;
            const bool upper = j >= 64;  // uniform in a warp
            float s4[4] = {0.f, 0.f, 0.f, 0.f};
            int tp = j + ((j + grp) & 1);
            for (; tp + 6 < n; tp += 8) {
                float v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) v[u] = XX[(tp + 2 * u) * XS + j];
                if (upper) {
#pragma unroll
                    for (int u = 0; u < 4; ++u) v[u] += xtot[tp + 2 * u];
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) s4[u] += v[u];
            }
            for (; tp < n; tp += 2) s4[0] += XX[tp * XS + j] + (upper ? xtot[tp] : 0.f);
            sr = (s4[0] + s4[1]) + (s4[2] + s4[3]);
        }
        if (grp == 1) rpart[kcol] = sr;
        sync_first256();  // G H (in the C / B region) and the U copy (in the x tile) are read
        mbar_arrive(&bars[6]);  // the next item's C, B, x may load
        if (!*abort_s && grp == 0 && t < n) {
            float4 *o = reinterpret_cast<float4 *>(a.dkap_acc + blh(d, b, c0 + t, h) * K);
#pragma unroll
            for (int q = 0; q < KMAX / 4; ++q) {
                if (4 * q < K) {
                    const float4 pq = *reinterpret_cast<const float4 *>(part + t * KMAX + 4 * q);
                    o[q] = make_float4(dk[4 * q] + pq.x, dk[4 * q + 1] + pq.y, dk[4 * q + 2] + pq.z,
                                       dk[4 * q + 3] + pq.w);
                }
            }
            a.rect[blh(d, b, c0 + t, h)] = sr + rpart[t];
        }
        if (!*abort_s && !mbar_wait(&bars[2], ph)) *abort_s = 1;
        sync_first256();
        tc_fence_after();
        {  // dx_intra row: group g takes columns [32 g, 32 g + 32) (nothing written after an abort)
            float v[32];
            tmem_ld32(lane_base + colX + grp * 32, v);
            tmem_ld_wait();
            uint4 e[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) e[q] = f4_bits(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
            const int t8 = t & ~7;
            put_rows<8, false>(e, reinterpret_cast<unsigned char *>(a.dx_acc + blh(d, b, c0 + t8, h) * P + grp * 32),
                               size_t(d.H) * P * 4, *abort_s ? 0 : n - t8);
        }
        tc_fence_before();
        mbar_arrive(&bars[7]);  // this item's TMEM reads are done: the next item's MMAs may go
        sync_first256();
        if (*abort_s) break;
    }  // items
    cp_async_wait_all();
    if (*abort_s && tid == 0) atomicExch(a.err, kTimeoutCode);
    tc_fence_before();
    __syncthreads();
    if (tid < 32) tmem_dealloc(tmem, 512);
}

// ============================================================================= state terms
// One CTA per (b, c, group of hg heads of one B/C group), 256 compute threads plus an issuing warp
// and three dot-product warps, software-pipelined over the (head, mode) steps.  Step i, with the
// mode's S_in and dS_out tiles [p][n] streamed in by TMA (two buffers):
//   Z_m = C S_in,m^T,  U_m = B dS_out,m^T                  (TMEM, one buffer of 2 x 64 columns)
//   dC += (f_m o dY) S_in,m,  dB += (s_m o X) dS_out,m       (TMEM, summed over modes and heads)
// The generated operands f_m o dY and s_m o X are written by the threads straight into TMEM (each
// thread owns the lane of its row; two buffers) and feed the dC / dB MMAs as the A operand, so
// they cost no shared-memory traffic.  Step i's Z / U MMAs start once step i - 1 has been read
// out; the threads read out step i - 1 after writing step i's operands: group 0 contracts Z_m with
// its dY row (dw_read, the a term), group 1 contracts U_m with its X row (dkappa, the b term) and
// accumulates dx = sum_m s_m U_m in registers.  Three more warps form <dS_out,m, S_in,m> from the
// two tiles in shared memory, and one of their lanes refills a tile buffer once its step's MMAs
// and the three warps are done with it.  The next head's dY, X and coefficient rows are staged by
// TMA a whole head ahead.  The head-summed intra tile Gamma o H adds M_H B to dC and M_H^T C to dB
// once per (b, c, B/C group).
constexpr int kStThreads = 256;  // compute threads (two warpgroups); a ninth warp issues the MMAs
                                 // (one thread)
constexpr int kCdThreads = 96;   // three more warps form <dS_out,m, S_in,m> from each step's tiles
constexpr int kStLaunch = kStThreads + 32 + kCdThreads;
constexpr int kStBuf = 2;   // S_in / dS_out tile buffers
constexpr int kCoefStride = 3 * KMAX + 1;  // per-thread coefficient row (odd: no bank conflicts)
// the next head's inputs staged by TMA in the generator region: dY [128 t][64 p] and X (bf16,
// 128-byte rows), then the coefficient rows [128 t][4 K] (fp32, 128- or 64-byte rows), each
// with the TMA swizzle so that eight threads reading the same chunk of their rows hit distinct
// banks
constexpr int kStageX = 16384, kStageCoef = 32768;

struct StSmem {
    int cb, tile, gen, total;
    __host__ __device__ explicit StSmem(int N) {
        cb = (N / 64) * 16384;   // one of C / B: [t][n]
        tile = (N / 64) * 8192;  // one S_in or dS_out mode tile: [p = 64][n], 64-wide n atoms
        gen = 2 * 16384;         // two units: M_H [t][k] at the start, dC staging at the end
        total = 2 * cb + kStBuf * 2 * tile + 2 * gen + kStThreads * kCoefStride * 4 + 1024;
    }
};

__device__ __forceinline__ float dot_bf16x8(uint4 a, uint4 b, float acc) {
    const uint32_t ra[4] = {a.x, a.y, a.z, a.w}, rb[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 fa = bf16x2_to_float2(ra[i]), fb = bf16x2_to_float2(rb[i]);
        acc = fmaf(fa.x, fb.x, fmaf(fa.y, fb.y, acc));
    }
    return acc;
}

// eight bf16 values times s, as packed bf16 products (s rounded to bf16 first)
__device__ __forceinline__ uint4 scale_bf16x8(uint4 a, float s) {
    const __nv_bfloat162 s2 = __float2bfloat162_rn(s);
    return make_uint4(bf16x2_mul(a.x, s2), bf16x2_mul(a.y, s2), bf16x2_mul(a.z, s2), bf16x2_mul(a.w, s2));
}

__global__ void __launch_bounds__(kStLaunch, 1)
    tc_bwd_state(const __grid_constant__ CUtensorMap mapC, const __grid_constant__ CUtensorMap mapB,
                 const __grid_constant__ CUtensorMap mapS, const __grid_constant__ CUtensorMap mapD,
                 const __grid_constant__ CUtensorMap mapdC, const __grid_constant__ CUtensorMap mapdB,
                 const __grid_constant__ CUtensorMap mapDY, const __grid_constant__ CUtensorMap mapX,
                 const __grid_constant__ CUtensorMap mapCf, BwdArgs a) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char *base = align1024(smem_raw);
    const ScanDims &d = a.d;
    const int K = d.K, N = d.N, P = d.P;
    const StSmem L(N);
    unsigned char *sC = base, *sB = sC + L.cb, *sT = sB + L.cb;
    unsigned char *sG = sT + kStBuf * 2 * L.tile;             // [buf][f o dY | s o X]
    // this thread's mode coefficients for the current head: cA (f or s), cB (exp(-E/tau) or u), s
    float *coef_s = reinterpret_cast<float *>(sG + 2 * L.gen);  // [256][kCoefStride]
    float *itau_s = coef_s + kStThreads * kCoefStride;         // [hg][K] 1 / tau (hg <= 16)
    double *wsum = reinterpret_cast<double *>(itau_s + 16 * KMAX);  // [8]
    double *Eend_s = wsum + 8;                                  // [1]
    // bars: 0..2 tile buffers | 3, 4 MMA of step parity | 5 C, B | 6 intra MMA |
    //       7, 8 generated operands of step parity written (all 256 threads arrive) |
    //       9, 10 tile buffer released: read by the <dS_out, S_in> warps (all 96 threads arrive)
    //             and by every MMA of its step (one arrival from the issuer's commit)
    uint64_t *bars = reinterpret_cast<uint64_t *>(Eend_s + 2);
    //       11 Z and U of the step written (their readout need not wait for dC / dB) |
    //       12 Z and U of the step read out (all 256 threads arrive) | 13 next head staged
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bars + 14);
    volatile int *abort_s = reinterpret_cast<volatile int *>(tslot + 1);

    const int tid = threadIdx.x, grp = tid >> 7, t = tid & 127, w = tid >> 5, w4 = w & 3;
    const int hgi = blockIdx.x, c = blockIdx.y, b = blockIdx.z;
    const int h_first = hgi * a.hg;
    const int g = h_first / (d.H / d.G);
    const int c0 = c * TQ, n = min(TQ, d.L - c0);
    const int nsteps = a.hg * K;
    const bool intra = (h_first % (d.H / d.G)) == 0;
    // TMEM columns: dC, dB accumulators; Z (+0) and U (+64); generated operands of buffer gb at
    // colG + 64 gb, f o dY (+0, group 0) and s o X (+32, group 1) as packed bf16 pairs
    constexpr uint32_t colC = 0, colB = 128, colZU = 256, colG = 384;

    if (tid == 0) {
        for (int i = 0; i < 7; ++i) mbar_init(&bars[i], 1);
        mbar_init(&bars[7], kStThreads);
        mbar_init(&bars[8], kStThreads);
        mbar_init(&bars[9], kCdThreads + 1);
        mbar_init(&bars[10], kCdThreads + 1);
        mbar_init(&bars[11], 1);
        mbar_init(&bars[12], kStThreads);
        mbar_init(&bars[13], 1);
        *abort_s = 0;
        fence_barrier_init();
    }
    if (w == 0) tmem_alloc_once(tslot, 512);
    for (int i = tid; i < a.hg * K; i += kStLaunch) itau_s[i] = 1.f / a.tau[h_first * K + i];
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    const uint32_t lane_base = tmem + (uint32_t(w4 * 32) << 16);

    const bool issuer = tid == kStThreads;  // lane 0 of the ninth warp
    auto issue_tiles = [&](int i) {  // S_in / dS_out tiles of step i into buffer i % kStBuf
        const int q = i % kStBuf;
        const int srow = int(((size_t(b) * d.H + h_first + i / K) * d.nc + c) * K + i % K);
        mbar_arrive_expect_tx(&bars[q], uint32_t(2 * L.tile));
        for (int jb = 0; jb < N / 64; ++jb) {
            tma_load_3d(sT + (2 * q) * L.tile + jb * 8192, &mapS, &bars[q], 64 * jb, 0, srow);
            tma_load_3d(sT + (2 * q + 1) * L.tile + jb * 8192, &mapD, &bars[q], 64 * jb, 0, srow);
        }
    };
    if (issuer) {
        mbar_arrive_expect_tx(&bars[5], uint32_t(2 * L.cb));
        for (int jb = 0; jb < N / 64; ++jb) {
            tma_load_3d(sC + jb * 16384, &mapC, &bars[5], g * N + 64 * jb, c0, b);
            tma_load_3d(sB + jb * 16384, &mapB, &bars[5], g * N + 64 * jb, c0, b);
        }
        for (int i = 0; i < min(kStBuf, nsteps); ++i) issue_tiles(i);
    }

    // head-summed intra term: dC = M_H B, dB = M_H^T C (M_H as bf16 [t][k] in generator buffer 0)
    if (intra) {
        if (tid < kStThreads) {  // row t, k in [64 grp, 64 grp + 64), read row-coalesced in two halves
            const float *mrow8 = a.mh_total + (((size_t(b) * d.nc + c) * d.G + g) * TQ + (t & ~7)) * TQ + grp * 64;
#pragma unroll
            for (int hf = 0; hf < 2; ++hf) {
                uint4 e[8];
                get_rows<8>(e, reinterpret_cast<const unsigned char *>(mrow8 + 32 * hf), TQ * 4, 8);
#pragma unroll
                for (int k8 = 0; k8 < 4; ++k8) {
                    const uint4 u0 = e[2 * k8], u1 = e[2 * k8 + 1];
                    const float v[8] = {__uint_as_float(u0.x), __uint_as_float(u0.y), __uint_as_float(u0.z),
                                        __uint_as_float(u0.w), __uint_as_float(u1.x), __uint_as_float(u1.y),
                                        __uint_as_float(u1.z), __uint_as_float(u1.w)};
                    const int kb = 4 * hf + k8;  // 8-column block within the group's 64
                    store_bf16x8(sG + grp * 16384 + t * 128 + ((kb ^ (t & 7)) * 16), v);
                }
            }
        }
        fence_async_smem();
        __syncthreads();
        if (issuer) {
            if (!mbar_wait(&bars[5], 0)) {
                *abort_s = 1;
            } else {
                tc_fence_after();
                const uint32_t idC = idesc_bf16(128, N, false, true);
                const uint32_t idB = idesc_bf16(128, N, true, true);
                for (int ks = 0; ks < TQ / 16; ++ks) {
                    mma_bf16(tmem + colC, desc_sw128(smem_u32(sG) + (ks / 4) * 16384 + (ks % 4) * 32, 16, 1024),
                             desc_sw128(smem_u32(sB) + ks * 2048, 16384, 1024), idC, ks > 0);
                    mma_bf16(tmem + colB, desc_sw128(smem_u32(sG) + ks * 2048, 16384, 1024),
                             desc_sw128(smem_u32(sC) + ks * 2048, 16384, 1024), idB, ks > 0);
                }
                mma_commit(&bars[6]);
            }
        }
        __syncthreads();
        if (!*abort_s && !mbar_wait(&bars[6], 0)) *abort_s = 1;  // generator buffer 0 is rewritten
    }
    if (!*abort_s && !mbar_wait(&bars[5], 0)) *abort_s = 1;      // C and B are read below

    // mode coefficients of row t: group 0 cA = f, cB = exp(-E/tau); group 1 cA = s, cB = u
    float *my_coef = coef_s + (tid < kStThreads ? tid : 0) * kCoefStride;  // cA [0, 8), cB [8, 16), s [16, 24)
    uint4 row[8];     // group 0: dY row (64 p), group 1: X row
    float dxr[32];    // inter-chunk dx of this row, p in [32 grp, 32 grp + 32), current head
    float acc_h[KMAX], ab_h = 0.f;  // group 0: dw_read and a; group 1: dkappa and b
#pragma unroll
    for (int m = 0; m < KMAX; ++m) acc_h[m] = 0.f;
#pragma unroll
    for (int q = 0; q < 8; ++q) row[q] = make_uint4(0, 0, 0, 0);
#pragma unroll
    for (int p = 0; p < 32; ++p) dxr[p] = 0.f;

    // read out step j (its MMAs complete): Z (group 0) or U (group 1) against this row, and
    // dx[t, p] += s_m U_m[t, p] with group g taking p in [32 g, 32 g + 32)
    auto readout = [&](int j) {
        if (!*abort_s && !mbar_wait(&bars[11], j & 1)) *abort_s = 1;
        tc_fence_after();
        const int mj = j % K, hj = h_first + j / K;
        if (!*abort_s) {
            const uint32_t zu = lane_base + colZU;  // Z at +0, U at +64
            const float sj = my_coef[2 * KMAX + mj], aj = my_coef[mj], bj = my_coef[KMAX + mj];
            float2 dp[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                            make_float2(0.f, 0.f)};  // independent partial sums (packed float32 pairs)
            const float2 sj2 = make_float2(sj, sj);
            // 16-column chunks, the next one loading while the current one is used: group 0 reads
            // Z (4 chunks, against dY) and U's first half (2, dx); group 1 reads U (4, against X,
            // the second half also for dx)
            const int nch = grp == 0 ? 6 : 4;
            auto col = [&](int ch) -> uint32_t {
                return grp == 0 ? (ch < 4 ? 16u * ch : 64u + 16u * (ch - 4)) : 64u + 16u * ch;
            };
            float za[16], zb[16];
            tmem_ld16(zu + col(0), za);
            tmem_ld_wait16(za);
#pragma unroll
            for (int ch = 0; ch < 6; ++ch) {
                if (ch < nch) {
                    float *cur = (ch & 1) ? zb : za, *nxt = (ch & 1) ? za : zb;
                    if (ch + 1 < nch) tmem_ld16(zu + col(ch + 1), nxt);
                    if (ch < 4) {
#pragma unroll
                        for (int q = 0; q < 2; ++q) {
                            const uint4 rv = row[2 * ch + q];
                            const uint32_t rr[4] = {rv.x, rv.y, rv.z, rv.w};
#pragma unroll
                            for (int k = 0; k < 4; ++k)
                                dp[k] = __ffma2_rn(bf16x2_to_float2(rr[k]),
                                                   make_float2(cur[8 * q + 2 * k], cur[8 * q + 2 * k + 1]), dp[k]);
                        }
                    }
                    if (ch >= 2 && (grp == 1 || ch >= 4)) {  // dx: U columns [0, 32) (group 0) / [32, 64)
                        const int o = 16 * ((ch - 2) & 1);
#pragma unroll
                        for (int i = 0; i < 16; i += 2) {
                            const float2 v = __ffma2_rn(sj2, make_float2(cur[i], cur[i + 1]),
                                                        make_float2(dxr[o + i], dxr[o + i + 1]));
                            dxr[o + i] = v.x;
                            dxr[o + i + 1] = v.y;
                        }
                    }
                    if (ch + 1 < nch) tmem_ld_wait16(nxt);
                }
            }
            tc_fence_before();
            mbar_arrive(&bars[12]);  // the Z / U columns may take step j + 1
            const float dotv = ((dp[0].x + dp[0].y) + (dp[1].x + dp[1].y)) + ((dp[2].x + dp[2].y) + (dp[3].x + dp[3].y));
#pragma unroll
            for (int m = 0; m < KMAX; ++m) {
                if (m == mj) acc_h[m] = bj * dotv;  // group 0: dw_read (inter); group 1: dkappa (inter)
            }
            ab_h = fmaf(aj * dotv, itau_s[(j / K) * K + mj], ab_h);  // group 0: a; group 1: b
        }
        if (mj == K - 1) {  // head hj complete: reductions, nothing waits
            if (!*abort_s && t < n) {
                const size_t i0 = blh(d, b, c0 + t, hj);
                float4 *acc_dst = reinterpret_cast<float4 *>((grp == 0 ? a.dwr_acc : a.dkap_acc) + i0 * K);
#pragma unroll
                for (int q = 0; q < KMAX / 4; ++q)
                    if (4 * q < K)
                        atomicAdd(acc_dst + q,
                                  make_float4(acc_h[4 * q], acc_h[4 * q + 1], acc_h[4 * q + 2], acc_h[4 * q + 3]));
                a.ab_acc[i0 * 2 + grp] = ab_h;
                if (a.inter_acc) {  // the inter-chunk parts kept apart (timescale gradient)
                    float4 *o = reinterpret_cast<float4 *>(a.inter_acc + (i0 * 2 + grp) * K);
#pragma unroll
                    for (int q = 0; q < KMAX / 4; ++q)
                        if (4 * q < K)
                            o[q] = make_float4(acc_h[4 * q], acc_h[4 * q + 1], acc_h[4 * q + 2], acc_h[4 * q + 3]);
                }
            }
            uint4 e[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) e[q] = f4_bits(dxr[4 * q], dxr[4 * q + 1], dxr[4 * q + 2], dxr[4 * q + 3]);
            const int t8 = t & ~7;
            put_rows<8, true>(e, reinterpret_cast<unsigned char *>(a.dx_acc + blh(d, b, c0 + t8, hj) * P + 32 * grp),
                              size_t(d.H) * P * 4, *abort_s ? 0 : n - t8);
        }
    };

    if (issuer) {
        // step i: Z / U once its tiles are in and step i - 1 has been read out, then dC / dB once
        // the threads have written step i's generated operands into TMEM; the descriptors of the
        // K slices are fixed offsets from those of the operands
        const uint32_t id64 = idesc_bf16(128, 64, false, false);
        const uint32_t idN = idesc_bf16(128, N, false, true);
        const uint64_t dC0 = desc_sw128(smem_u32(sC), 16, 1024), dB0 = desc_sw128(smem_u32(sB), 16, 1024);
        const int nks = N / 16;
        for (int i = 0; i < nsteps && !*abort_s; ++i) {
            const int gb = i & 1, q = i % kStBuf;
            if (!mbar_wait(&bars[q], (i / kStBuf) & 1) || (i >= 1 && !mbar_wait(&bars[12], (i - 1) & 1))) {
                *abort_s = 1;
                break;
            }
            tc_fence_after();
            const uint32_t sS = smem_u32(sT + (2 * q) * L.tile), sD = smem_u32(sT + (2 * q + 1) * L.tile);
            const uint64_t dS = desc_sw128(sS, 16, 1024), dD = desc_sw128(sD, 16, 1024);
#pragma unroll
            for (int ks = 0; ks < 8; ++ks) {
                if (ks < nks) {
                    const uint32_t ko = (ks / 4) * 16384 + (ks % 4) * 32, to = (ks / 4) * 8192 + (ks % 4) * 32;
                    mma_bf16(tmem + colZU, desc_add(dC0, ko), desc_add(dS, to), id64, ks > 0);
                    mma_bf16(tmem + colZU + 64, desc_add(dB0, ko), desc_add(dD, to), id64, ks > 0);
                }
            }
            mma_commit(&bars[11]);  // Z, U of step i: the readout may start
            if (!mbar_wait(&bars[7 + gb], (i >> 1) & 1)) {
                *abort_s = 1;
                break;
            }
            tc_fence_after();
            const uint32_t g1 = tmem + colG + 64 * gb, g2 = g1 + 32;
            const uint64_t dSn = desc_sw128(sS, 8192, 1024), dDn = desc_sw128(sD, 8192, 1024);
            const uint32_t acc0 = (intra || i > 0) ? 1u : 0u;
#pragma unroll
            for (int ks = 0; ks < 4; ++ks) {  // K = p, 16 per MMA: 8 columns of packed pairs
                mma_bf16_ts(tmem + colC, g1 + 8 * ks, desc_add(dSn, ks * 2048), idN, ks > 0 ? 1u : acc0);
                mma_bf16_ts(tmem + colB, g2 + 8 * ks, desc_add(dDn, ks * 2048), idN, ks > 0 ? 1u : acc0);
            }
            mma_commit(&bars[9 + q]);   // the tile buffer, once every MMA of step i has read it
            mma_commit(&bars[3 + gb]);  // the generated operands of buffer gb, and dC / dB
        }
        // the releases of the last tile buffers complete before the CTA ends (nothing else waits
        // for them)
        for (int i = max(0, nsteps - kStBuf); i < nsteps && !*abort_s; ++i)
            if (!mbar_wait(&bars[9 + i % kStBuf], (i / kStBuf) & 1)) *abort_s = 1;
    }
    if (tid >= kStThreads + 32) {
        // <dS_out,m, S_in,m> of every step from its two tiles (the same swizzle in both), then the
        // tile buffer is released to the issuer
        const int ct = tid - (kStThreads + 32);
        for (int i = 0; i < nsteps; ++i) {
            const int q = i % kStBuf;
            // the warp leaves together (its lanes meet in the shuffles below)
            if (!__all_sync(0xffffffffu, !*abort_s && mbar_wait(&bars[q], (i / kStBuf) & 1))) {
                *abort_s = 1;
                break;
            }
            const uint4 *ps = reinterpret_cast<const uint4 *>(sT + (2 * q) * L.tile);
            const uint4 *pd = reinterpret_cast<const uint4 *>(sT + (2 * q + 1) * L.tile);
            float acc0 = 0.f, acc1 = 0.f;
            int k = ct;
            for (; k + kCdThreads < L.tile / 16; k += 2 * kCdThreads) {
                acc0 = dot_bf16x8(ps[k], pd[k], acc0);
                acc1 = dot_bf16x8(ps[k + kCdThreads], pd[k + kCdThreads], acc1);
            }
            if (k < L.tile / 16) acc0 = dot_bf16x8(ps[k], pd[k], acc0);
            mbar_arrive(&bars[9 + q]);
            const float v = warp_sum(acc0 + acc1);
            if ((tid & 31) == 0)
                atomicAdd(a.cdot + ((size_t(b) * d.H + h_first + i / K) * d.nc + c) * K + i % K, v);
            // the tile buffer of step i takes the tiles of step i + kStBuf once it is released
            if (ct == 0 && i + kStBuf < nsteps) {
                if (*abort_s || !mbar_wait(&bars[9 + q], (i / kStBuf) & 1))
                    *abort_s = 1;
                else
                    issue_tiles(i + kStBuf);
            }
        }
    }
    for (int i = 0; i < nsteps && tid < kStThreads; ++i) {
        const int hh = i / K, m = i % K, h = h_first + hh, gb = i & 1;
        bool prev_done = i == 0;
        if (m == 0) {
            // a new head: step i - 1 (the previous head's last) is read out with that head's
            // coefficients first, then the coefficients of row t and its row of dY / X change
            if (i > 0) {
                readout(i - 1);
                prev_done = true;
            }
#pragma unroll
            for (int k = 0; k < KMAX; ++k) acc_h[k] = 0.f;
            if (hh > 0) {
                // from the staged tiles: this thread's row of dY / X and its coefficient pieces
                // (group 0: f, exp(-E/tau), s; group 1: s, u, s), unswizzled
                if (!*abort_s && !mbar_wait(&bars[13], (hh - 1) & 1)) *abort_s = 1;
                const unsigned char *ry = sG + (grp == 0 ? 0 : kStageX) + t * 128;
#pragma unroll
                for (int k = 0; k < 8; ++k) row[k] = *reinterpret_cast<const uint4 *>(ry + ((k ^ (t & 7)) * 16));
                const unsigned char *rc = sG + kStageCoef + t * (16 * K);
                const int kinds[3] = {grp == 0 ? 0 : 1, grp == 0 ? 3 : 2, 1};  // f s u exp(-E/tau) = 0 1 2 3
#pragma unroll
                for (int k = 0; k < 3; ++k)
                    for (int j = 0; j < K / 4; ++j) {
                        const int ch = kinds[k] * (K / 4) + j;
                        const int cs = K == 8 ? (ch ^ (t & 7)) : (ch ^ ((t >> 1) & 3));
                        const float4 v = *reinterpret_cast<const float4 *>(rc + cs * 16);
                        float *dst = my_coef + k * KMAX + 4 * j;
                        dst[0] = v.x; dst[1] = v.y; dst[2] = v.z; dst[3] = v.w;
                    }
                fence_async_smem();
                sync_first256();  // every row is out of the staged tiles
            } else {
            // coefficients of this row from tc_coef (group 0: f, exp(-E/tau); group 1: s, u;
            // both: s) and its row of dY / X, read row-coalesced across each 8-lane group
            const int t8 = t & ~7;
            const size_t r8 = blh(d, b, c0 + t8, h);
            float4 c4[6];
            {
                auto f4 = [](uint4 v) {
                    return make_float4(__uint_as_float(v.x), __uint_as_float(v.y), __uint_as_float(v.z),
                                       __uint_as_float(v.w));
                };
                if (K == 8) {  // pieces: f 0-1, s 2-3, u 4-5, exp(-E/tau) 6-7
                    uint4 cr[8];
                    get_rows<8>(cr, reinterpret_cast<const unsigned char *>(a.coef + r8 * 32), size_t(d.H) * 128,
                                n - t8);
#pragma unroll
                    for (int q = 0; q < 2; ++q) {
                        c4[q] = f4(grp == 0 ? cr[q] : cr[2 + q]);
                        c4[2 + q] = f4(grp == 0 ? cr[6 + q] : cr[4 + q]);
                        c4[4 + q] = f4(cr[2 + q]);
                    }
                } else {  // K == 4, 64-byte rows in 4-lane groups; pieces: f, s, u, exp(-E/tau)
                    const int t4 = t & ~3;
                    uint4 cr[4];
                    get_rows<4>(cr, reinterpret_cast<const unsigned char *>(a.coef + blh(d, b, c0 + t4, h) * 16),
                                size_t(d.H) * 64, n - t4);
                    const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
                    c4[0] = f4(grp == 0 ? cr[0] : cr[1]);
                    c4[2] = f4(grp == 0 ? cr[3] : cr[2]);
                    c4[4] = f4(cr[1]);
                    c4[1] = c4[3] = c4[5] = z;
                }
            }
            {
                uint4 rr[8];
                get_rows<8>(rr, reinterpret_cast<const unsigned char *>((grp == 0 ? a.dy : a.x) + r8 * P),
                            size_t(d.H) * P * 2, n - t8);
#pragma unroll
                for (int k = 0; k < 8; ++k) row[k] = rr[k];
            }
#pragma unroll
            for (int k = 0; k < 6; ++k) {  // this thread's row: scalar stores (the row stride is odd)
                float *dst = my_coef + (k >> 1) * KMAX + (k & 1) * 4;
                dst[0] = c4[k].x; dst[1] = c4[k].y; dst[2] = c4[k].z; dst[3] = c4[k].w;
            }
            }
            if (tid == 0 && hh + 1 < a.hg) {  // the next head's dY, X and coefficient tiles
                mbar_arrive_expect_tx(&bars[13], uint32_t(2 * 16384 + TQ * 16 * K));
                tma_load_3d(sG, &mapDY, &bars[13], (h + 1) * P, c0, b);
                tma_load_3d(sG + kStageX, &mapX, &bars[13], (h + 1) * P, c0, b);
                tma_load_3d(sG + kStageCoef, &mapCf, &bars[13], (h + 1) * 4 * K, c0, b);
            }
            ab_h = 0.f;
#pragma unroll
            for (int p = 0; p < 32; ++p) dxr[p] = 0.f;
        }
        // generated operands of step i into TMEM buffer gb (this thread's lane), once step i - 2's
        // MMAs have read it
        if (i >= 2 && !*abort_s && !mbar_wait(&bars[3 + gb], ((i - 2) >> 1) & 1)) *abort_s = 1;
        tc_fence_after();
        {
            const float sc = my_coef[m];
            const uint32_t dst = lane_base + colG + 64 * gb + 32 * grp;
#pragma unroll
            for (int hf = 0; hf < 2; ++hf) {
                uint32_t v[16];
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const uint4 g = scale_bf16x8(row[4 * hf + k], sc);
                    v[4 * k] = g.x; v[4 * k + 1] = g.y; v[4 * k + 2] = g.z; v[4 * k + 3] = g.w;
                }
                tmem_st16(dst + 16 * hf, v);
            }
            tmem_st_wait();
        }
        // hand the generated operands to the MMA issuer (no CTA-wide barrier in the loop)
        tc_fence_before();
        mbar_arrive(&bars[7 + gb]);
        // step i - 1 is read out while the tensor cores run step i
        if (!prev_done) readout(i - 1);
    }
    if (nsteps > 0 && tid < kStThreads) readout(nsteps - 1);
    // the group's dC / dB into the float32 accumulators (group g takes n in [64 g, 64 g + 64))
    tc_fence_after();
    // every MMA (dC, dB of the last step included) has completed before the accumulators are read
    if (tid < kStThreads && nsteps > 0 && !*abort_s &&
        !mbar_wait(&bars[3 + ((nsteps - 1) & 1)], ((nsteps - 1) >> 1) & 1))
        *abort_s = 1;
    tc_fence_after();
    // the group's dC / dB into the float32 accumulators by TMA reduce-add: every warp has left
    // the tiles and the generated operands, which now stage dC (generator buffers) and dB (tile
    // buffers) as [N / 32 boxes][128 t][32 n] float32 with the 128-byte swizzle
    __syncthreads();
    if (tid < kStThreads && grp < N / 64) {
        for (int n32 = 0; n32 < 64; n32 += 32) {
            float vc[32], vb[32];
            tmem_ld32(lane_base + colC + grp * 64 + n32, vc);
            tmem_ld32(lane_base + colB + grp * 64 + n32, vb);
            tmem_ld_wait();
            const int q = (grp * 64 + n32) / 32;
            unsigned char *rc = sG + q * 16384 + t * 128, *rb = sT + q * 16384 + t * 128;
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                *reinterpret_cast<float4 *>(rc + ((k ^ (t & 7)) * 16)) =
                    make_float4(vc[4 * k], vc[4 * k + 1], vc[4 * k + 2], vc[4 * k + 3]);
                *reinterpret_cast<float4 *>(rb + ((k ^ (t & 7)) * 16)) =
                    make_float4(vb[4 * k], vb[4 * k + 1], vb[4 * k + 2], vb[4 * k + 3]);
            }
        }
        fence_async_smem();
    }
    __syncthreads();
    if (tid == 0 && !*abort_s) {  // rows past the end of the sequence fall outside the map
        for (int q = 0; q < N / 32; ++q) {
            tma_reduce_add_4d(&mapdC, sG + q * 16384, 32 * q, g, c0, b);
            tma_reduce_add_4d(&mapdB, sT + q * 16384, 32 * q, g, c0, b);
        }
        bulk_commit();
        bulk_wait_all();
    }
    if (*abort_s && tid == 0) atomicExch(a.err, kTimeoutCode);
    tc_fence_before();
    __syncthreads();
    if (w == 0) tmem_dealloc(tmem, 512);
}

// ============================================================================= final
// Float block scans of one value per thread over 128 threads: inclusive prefix, inclusive suffix
// and total (no difference of two sums is ever formed).
__device__ __forceinline__ void block_scans128(float v, float *pre, float *suf, float *tot,
                                               float *sh /* [3][4] */) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    float p = v, q = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float up = __shfl_up_sync(0xffffffffu, p, o);
        const float dn = __shfl_down_sync(0xffffffffu, q, o);
        if (lane >= o) p += up;
        if (lane + o < 32) q += dn;
    }
    if (lane == 31) sh[w] = p;  // warp totals
    __syncthreads();
    float before = 0.f, after = 0.f;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        if (i < w) before += sh[i];
        if (i > w) after += sh[i];
    }
    *pre = p + before;
    *suf = q + after;
    *tot = (sh[0] + sh[1]) + (sh[2] + sh[3]);
    __syncthreads();
}

// One CTA per (b, h, chunk): per-position gradients of Delta, alpha, lambda, w_write, w_read
// (from the accumulated mode terms and rho <dS_t, S_{t-1}>), then dx = dx_acc + D dy as bf16 and
// the dD partial, one warp per row so that every access is a contiguous row segment.
__global__ void __launch_bounds__(kThreads) tc_bwd_final(BwdArgs a) {
    const ScanDims &d = a.d;
    const int K = d.K, P = d.P;
    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z, t = threadIdx.x;
    const int lane = t & 31, w = t >> 5;
    const int c0 = c * TQ, n = min(TQ, d.L - c0);
    __shared__ float itau[32], tau_sh[32];
    __shared__ float sh[4];
    __shared__ float red[4];
    __shared__ float tq_sh[4][KMAX];  // per warp and mode: sums of the timescale-gradient terms
    if (t < K) {
        const float tv = a.tau[h * K + t];
        tau_sh[t] = tv;
        itau[t] = 1.f / tv;
    }
    const size_t i = (t < n) ? blh(d, b, c0 + t, h) : 0;
    float dtv = 1.f, alv = 1.f, lmv = 1.f, av = 0.f, bv = 0.f, rc = 0.f;
    float ww[KMAX], dkv[KMAX], dwv[KMAX];
#pragma unroll
    for (int m = 0; m < KMAX; ++m) ww[m] = dkv[m] = dwv[m] = 0.f;
    if (t < n) {
        dtv = a.dt[i];
        alv = a.alpha[i];
        lmv = a.lam[i];
        const float2 ab = *reinterpret_cast<const float2 *>(a.ab_acc + i * 2);
        av = ab.x;
        bv = ab.y;
        rc = a.rect[i];
        load_weights(a.ww + i * K, K, ww);
#pragma unroll
        for (int q = 0; q < KMAX / 4; ++q) {
            if (4 * q < K) {
                const float4 u = *reinterpret_cast<const float4 *>(a.dkap_acc + i * K + 4 * q);
                const float4 v = *reinterpret_cast<const float4 *>(a.dwr_acc + i * K + 4 * q);
                dkv[4 * q] = u.x; dkv[4 * q + 1] = u.y; dkv[4 * q + 2] = u.z; dkv[4 * q + 3] = u.w;
                dwv[4 * q] = v.x; dwv[4 * q + 1] = v.y; dwv[4 * q + 2] = v.z; dwv[4 * q + 3] = v.w;
            }
        }
    }
    __syncthreads();
    float tmax = 0.f;
    for (int m = 0; m < K; ++m) tmax = fmaxf(tmax, tau_sh[m]);
    const float log_cap = logf(64.f * tmax);
    float e = 0.f;
    bool cl = false;
    if (t < n) e = token_rate(dtv, alv, lmv, log_cap, &cl);
    float pe, se, Eend;  // chunk total of e (the log-decay across the chunk)
    block_scans128(e, &pe, &se, &Eend, sh);
    float pa, suf_a, ta, pb, sb, tb;
    block_scans128(av, &pa, &suf_a, &ta, sh);  // suffix of a, inclusive
    block_scans128(bv, &pb, &sb, &tb, sh);     // prefix of b, exclusive = inclusive - own
    float cprime = 0.f;
    for (int m = 0; m < K; ++m)
        cprime = fmaf(expf(-Eend * itau[m]) * itau[m], a.cdot[((size_t(b) * d.H + h) * d.nc + c) * K + m], cprime);
    if (t < n) {
        const float pre_b = pb - bv;
        const float R = (suf_a + pre_b) + cprime + rc;
        float de = -R;
        float dww[KMAX];
#pragma unroll
        for (int m = 0; m < KMAX; ++m) {
            dww[m] = 0.f;
            if (m < K) {
                const float z = e * itau[m];
                const float rho = expf(-z), omr = -expm1f(-z);
                de = fmaf(dkv[m] * rho * ww[m], itau[m], de);
                dww[m] = dkv[m] * omr;
            }
        }
        if (K == 8) {
            *reinterpret_cast<uint4 *>(a.dwr + i * K) =
                make_uint4(pack_bf16x2(dwv[0], dwv[1]), pack_bf16x2(dwv[2], dwv[3]), pack_bf16x2(dwv[4], dwv[5]),
                           pack_bf16x2(dwv[6], dwv[7]));
            *reinterpret_cast<uint4 *>(a.dww + i * K) =
                make_uint4(pack_bf16x2(dww[0], dww[1]), pack_bf16x2(dww[2], dww[3]), pack_bf16x2(dww[4], dww[5]),
                           pack_bf16x2(dww[6], dww[7]));
        } else {
            *reinterpret_cast<uint2 *>(a.dwr + i * K) = make_uint2(pack_bf16x2(dwv[0], dwv[1]), pack_bf16x2(dwv[2], dwv[3]));
            *reinterpret_cast<uint2 *>(a.dww + i * K) = make_uint2(pack_bf16x2(dww[0], dww[1]), pack_bf16x2(dww[2], dww[3]));
        }
        const float ge = cl ? 0.f : de * e;
        a.ddt[i] = ge / dtv;
        a.dlam[i] = ge / (alv * lmv);
        a.dalpha[i] = -ge * logf(lmv) / (alv * alv);
    }
    if (a.dtau) {
        // Timescale gradient, the terms with S_in or dS_out: per mode, each weighted by the e_t
        // it spans (E_t from the chunk start, E_end - E_t to its end, E_end for the whole chunk):
        //   E_t w_read dw_read^inter + (E_end - E_t) kappa dkappa^inter - e_t dkappa rho w_write
        // plus E_end d_m <dS_out, S_in>_m once per chunk; the pairs inside the chunk come from
        // the dtau_pairs kernel.
        float wrv[KMAX], dwi[KMAX], dki[KMAX];
#pragma unroll
        for (int m = 0; m < KMAX; ++m) wrv[m] = dwi[m] = dki[m] = 0.f;
        if (t < n) {
            load_weights(a.wr + i * K, K, wrv);
#pragma unroll
            for (int q = 0; q < KMAX / 4; ++q)
                if (4 * q < K) {
                    const float4 u = *reinterpret_cast<const float4 *>(a.inter_acc + (i * 2) * K + 4 * q);
                    const float4 v = *reinterpret_cast<const float4 *>(a.inter_acc + (i * 2 + 1) * K + 4 * q);
                    dwi[4 * q] = u.x; dwi[4 * q + 1] = u.y; dwi[4 * q + 2] = u.z; dwi[4 * q + 3] = u.w;
                    dki[4 * q] = v.x; dki[4 * q + 1] = v.y; dki[4 * q + 2] = v.z; dki[4 * q + 3] = v.w;
                }
        }
#pragma unroll
        for (int m = 0; m < KMAX; ++m) {
            float v = 0.f;
            if (t < n && m < K) {
                const float z = e * itau[m];
                const float rho = expf(-z), kap = -expm1f(-z) * ww[m];
                // E_end - E_t as the exclusive suffix of e (scanned directly, no difference of sums)
                v = pe * wrv[m] * dwi[m] + (se - e) * kap * dki[m] - e * dkv[m] * rho * ww[m];
            }
            v = warp_sum(v);
            if (lane == 0) tq_sh[w][m] = v;
        }
        __syncthreads();
        if (t < K) {
            const float cd = a.cdot[((size_t(b) * d.H + h) * d.nc + c) * K + t];
            const float sum = (tq_sh[0][t] + tq_sh[1][t]) + (tq_sh[2][t] + tq_sh[3][t]) +
                              Eend * expf(-Eend * itau[t]) * cd;
            atomicAdd(a.dtau + h * K + t, sum * itau[t] * itau[t]);
        }
    }
    // dx = dx_acc + D dy (bf16) and sum dy x: each thread takes 8 p of 8 rows (rows r = 16 j + t / 8,
    // p in [8 (t % 8), 8 (t % 8) + 8)), all loads issued before any is used; every instruction
    // covers 16 whole 256-byte (or 128-byte) row segments
    const float Dh = a.D[h];
    float dd = 0.f;
    {
        const int p8 = 8 * (t & 7), r0 = t >> 3;
        float4 acc[8][2];
        uint4 dyv[8], xv[8];
#pragma unroll
        for (int jr = 0; jr < 8; ++jr) {
            const int r = 16 * jr + r0;
            if (r < n) {
                const size_t i0 = blh(d, b, c0 + r, h) * P + p8;
                acc[jr][0] = *reinterpret_cast<const float4 *>(a.dx_acc + i0);
                acc[jr][1] = *reinterpret_cast<const float4 *>(a.dx_acc + i0 + 4);
                dyv[jr] = *reinterpret_cast<const uint4 *>(a.dy + i0);
                xv[jr] = *reinterpret_cast<const uint4 *>(a.x + i0);
            }
        }
#pragma unroll
        for (int jr = 0; jr < 8; ++jr) {
            const int r = 16 * jr + r0;
            if (r < n) {
                const size_t i0 = blh(d, b, c0 + r, h) * P + p8;
                const float av8[8] = {acc[jr][0].x, acc[jr][0].y, acc[jr][0].z, acc[jr][0].w,
                                      acc[jr][1].x, acc[jr][1].y, acc[jr][1].z, acc[jr][1].w};
                const uint32_t dw[4] = {dyv[jr].x, dyv[jr].y, dyv[jr].z, dyv[jr].w};
                const uint32_t xw[4] = {xv[jr].x, xv[jr].y, xv[jr].z, xv[jr].w};
                uint32_t o[4];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float2 fy = bf16x2_to_float2(dw[q]), fx = bf16x2_to_float2(xw[q]);
                    o[q] = pack_bf16x2(fmaf(Dh, fy.x, av8[2 * q]), fmaf(Dh, fy.y, av8[2 * q + 1]));
                    dd = fmaf(fy.x, fx.x, fmaf(fy.y, fx.y, dd));
                }
                *reinterpret_cast<uint4 *>(a.dx + i0) = make_uint4(o[0], o[1], o[2], o[3]);
            }
        }
    }
    dd = warp_sum(dd);
    if (lane == 0) red[w] = dd;
    __syncthreads();
    if (t == 0) atomicAdd(a.dD + h, (red[0] + red[1]) + (red[2] + red[3]));
}

__global__ void f32_to_bf16_tc(const float *__restrict__ in, bf16 *__restrict__ out, size_t n) {
    for (size_t i = blockIdx.x * size_t(blockDim.x) + threadIdx.x; i < n; i += size_t(gridDim.x) * blockDim.x)
        out[i] = __float2bfloat16_rn(in[i]);
}

// Heads per CTA of tc_bwd_state: a divisor of the heads of one B/C group, at most 16 (more
// heads amortise the CTA's set-up and dC / dB epilogue), but no more than leaves two waves of
// CTAs on the SMs; when even one head per CTA leaves fewer, the largest divisor.
int pick_hg(const ScanDims &d, int sms) {
    const int hpg = d.H / d.G;
    const size_t per_head = size_t(d.nc) * d.B, want = 2 * size_t(sms);
    int largest = 1, fits = 0;
    for (int hg = 1; hg <= 16; ++hg) {
        if (hpg % hg) continue;
        largest = hg;
        if (size_t(d.H / hg) * per_head >= want) fits = hg;
    }
    return fits ? fits : largest;
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
    l->coef = (float *)take(tc_coef_elems(d) * 4);  // S_in, coef and ek as in the forward's workspace
    l->ek = (float *)take(tc_ek_elems(d) * 4);
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
    l->inter_acc = (float *)take(blh_ * 2 * d.K * 4);
    return off;
}

cudaError_t tc_scan_bwd(const ScanDims &d, const ScanPtrs &p, const TcBwdWorkspace &ws, int *err,
                        bool reuse_states, cudaStream_t st) {
    cudaError_t e;
    const size_t ngn = size_t(d.B) * d.L * d.G * d.N;
    if ((e = cudaMemsetAsync(p.dD, 0, sizeof(float) * d.H, st))) return e;
    if ((e = cudaMemsetAsync(ws.dB_acc, 0, sizeof(float) * ngn, st))) return e;
    if ((e = cudaMemsetAsync(ws.dC_acc, 0, sizeof(float) * ngn, st))) return e;
    if ((e = cudaMemsetAsync(ws.cdot, 0, sizeof(float) * d.B * d.H * d.nc * d.K, st))) return e;
    if ((e = cudaMemsetAsync(ws.mh_total, 0, sizeof(float) * d.B * d.nc * d.G * TQ * TQ, st))) return e;
    if (p.dtau && (e = cudaMemsetAsync(p.dtau, 0, sizeof(float) * d.H * d.K, st))) return e;
    if (!reuse_states &&
        ((e = tc_coef_launch(d, p, ws.coef, ws.ek, st)) ||
         (e = tc_state_pass_launch(d, false, p.x, p.Bm, ws.coef, p.h0, ws.S_in, nullptr, err, st))))
        return e;
    if ((e = tc_state_pass_launch(d, true, p.dy, p.Cm, ws.coef, p.dh_final, ws.dS_out, p.dh0, err, st)))
        return e;
    if (d.nc == 0) return cudaSuccess;
    const uint64_t GN = uint64_t(d.G) * d.N, HP = uint64_t(d.H) * d.P;
    CUtensorMap mapC, mapB, mapX, mapDY, mapS, mapD, mapdC, mapdB, mapCf;
    const uint64_t srows = uint64_t(d.B) * d.H * d.nc * d.K;
    if (!tc_make_map3(&mapC, p.Cm, GN, d.L, d.B, GN * 2, uint64_t(d.L) * GN * 2, 64, TQ, 1) ||
        !tc_make_map3(&mapB, p.Bm, GN, d.L, d.B, GN * 2, uint64_t(d.L) * GN * 2, 64, TQ, 1) ||
        !tc_make_map3(&mapX, p.x, HP, d.L, d.B, HP * 2, uint64_t(d.L) * HP * 2, 64, TQ, 1) ||
        !tc_make_map3(&mapDY, p.dy, HP, d.L, d.B, HP * 2, uint64_t(d.L) * HP * 2, 64, TQ, 1) ||
        !tc_make_map3(&mapS, ws.S_in, d.N, d.P, srows, uint64_t(d.N) * 2, uint64_t(d.P) * d.N * 2, 64,
                      64, 1) ||
        !tc_make_map3(&mapD, ws.dS_out, d.N, d.P, srows, uint64_t(d.N) * 2, uint64_t(d.P) * d.N * 2, 64,
                      64, 1) ||
        // per-position coefficients [B, L, H, 4 K] as (h 4K, l, b); a box is one head's 128 rows
        !tc_make_map3_f32(&mapCf, ws.coef, uint64_t(d.H) * 4 * d.K, d.L, d.B, uint64_t(d.H) * 4 * d.K * 4,
                          uint64_t(d.L) * d.H * 4 * d.K * 4, 4 * d.K, TQ, 1, d.K == 8 ? 128 : 64))
        return cudaErrorInvalidValue;
    {  // dC / dB float32 accumulators [B, L, G, N] as (n, g, l, b); a box is 32 n x 128 positions
        const uint64_t dims[4] = {uint64_t(d.N), uint64_t(d.G), uint64_t(d.L), uint64_t(d.B)};
        const uint64_t strides[3] = {uint64_t(d.N) * 4, uint64_t(d.G) * d.N * 4, uint64_t(d.L) * d.G * d.N * 4};
        const uint32_t box[4] = {32, 1, TQ, 1};
        if (!tc_make_map4_f32(&mapdC, ws.dC_acc, dims, strides, box) ||
            !tc_make_map4_f32(&mapdB, ws.dB_acc, dims, strides, box))
            return cudaErrorInvalidValue;
    }
    BwdArgs a;
    a.d = d;
    a.x = (const bf16 *)p.x; a.dy = (const bf16 *)p.dy;
    a.wr = (const bf16 *)p.wr; a.ww = (const bf16 *)p.ww;
    a.dt = p.dt; a.alpha = p.alpha; a.lam = p.lam; a.tau = p.tau; a.D = p.D;
    a.S_in = (const bf16 *)ws.S_in; a.dS_out = (const bf16 *)ws.dS_out;
    a.dx_acc = ws.dx_acc; a.dwr_acc = ws.dwr_acc; a.dkap_acc = ws.dkap_acc; a.ab_acc = ws.ab_acc;
    a.rect = ws.rect; a.cdot = ws.cdot; a.mh_total = ws.mh_total; a.coef = ws.coef; a.ek = ws.ek;
    a.dB_acc = ws.dB_acc; a.dC_acc = ws.dC_acc;
    a.dx = (bf16 *)p.dx; a.dwr = (bf16 *)p.dwr; a.dww = (bf16 *)p.dww;
    a.ddt = p.ddt; a.dalpha = p.dalpha; a.dlam = p.dlam; a.dD = p.dD;
    a.dtau = p.dtau;
    a.inter_acc = p.dtau ? ws.inter_acc : nullptr;
    a.err = err;
    {
        int dev = 0, nsm = 0;
        if ((e = cudaGetDevice(&dev)) || (e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)))
            return e;
        a.pf_sms = std::max(nsm, 1);
    }
    a.hg = pick_hg(d, a.pf_sms);

    {
        const size_t smem = IntraSmem().total + 1024;
        cudaFuncSetAttribute(tc_bwd_intra, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        trace_begin("bwd_intra_tc", st);
        // persistent: one CTA per SM (shared memory), items (h, c, b) strided by the grid
        const int items = d.H * d.nc * d.B;
        tc_bwd_intra<<<std::min(items, a.pf_sms), kIntraLaunch, smem, st>>>(mapC, mapB, mapX, mapDY, a);
        trace_end(st);
        if ((e = cudaGetLastError())) return e;
    }
    {
        const size_t smem = StSmem(d.N).total + 1024;
        cudaFuncSetAttribute(tc_bwd_state, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        trace_begin("bwd_state_tc", st);
        tc_bwd_state<<<dim3(d.H / a.hg, d.nc, d.B), kStLaunch, smem, st>>>(mapC, mapB, mapS, mapD, mapdC, mapdB,
                                                                              mapDY, mapX, mapCf, a);
        trace_end(st);
        if ((e = cudaGetLastError())) return e;
    }
    trace_begin("bwd_final_tc", st);
    tc_bwd_final<<<dim3(d.nc, d.H, d.B), kThreads, 0, st>>>(a);
    trace_end(st);
    if ((e = cudaGetLastError())) return e;
    if ((e = dtau_pairs_launch(d, 1, p, st))) return e;
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
