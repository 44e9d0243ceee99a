// Tensor-core (tcgen05 / TMEM / TMA) chunked Frac scan for bf16 inputs, sm_103a.
//
// Same chunked evaluation order as the CUDA-core kernels (App. F of the paper), with chunk
// Q = 128 and the two state contractions of every chunk on the tensor cores:
//
//   tc_coef        (one CTA per (b, h, chunk)): the per-position mode coefficients of the
//        chunk (f, s = kappa u, u, exp(-E/tau) from the float-pair cumulative log-decay E), read
//        by the state passes and the backward instead of being recomputed per P-slice.
//   tc_state_pass  (chunk-serial; one CTA of 256 threads per (b, h, 128/K-wide slice of P)):
//        the P-slice of every mode's state lives in tensor memory as fp32, lanes = (mode, p),
//        columns = n.  Per chunk: emit the entering state (bf16) for the output kernel, scale
//        it by d_m = exp(-E_end/tau_m) in place, then accumulate
//        S_m += sum_k s_{k,m} x_k B_k^T  as  D[(m,p), n] += A[(m,p), k] * B[k, n]
//        (A = s o x generated in shared memory, B = the chunk of B loaded by TMA).
//        Run over the chunks in reverse with (dy, C, f) it carries dS for the backward.
//   tc_chunk_fwd   (chunk-parallel; one CTA per (b, c, h), headdim 64):
//        G = C B^T and the factored Gamma blocks on the tensor cores, Gamma o G -> bf16 tile,
//        Y = (Gamma o G) X in TMEM; then Z_m = C S_in,m^T, two modes per product (S_in tiles
//        streamed by TMA by a loading warp, MMAs issued by an issuing warp), which the threads
//        fold into their rows with f_m[t]: y = Y + sum_m f_m o Z_m + D x.
//
// All mbarrier waits are bounded (a few seconds); on a timeout the kernel records
// FRAC_ERR_TIMEOUT in the error word, stops issuing work, frees its tensor memory and exits.
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


struct StateArgs {
    ScanDims d;
    const bf16 *U;      // x or dy      [B, L, H, P]
    const float *coef;  // per-position mode coefficients [B, L, H, 4, K] (tc_coef)
    const float *init;  // h0 or dh_final [B, H, K, P, N] or null
    bf16 *emit;         // per-chunk entering states [B, H, nc, K, P, N]
    float *fin;         // h_final or dh0, or null
    int *err;
};

// ---------------------------------------------------------------------------------------------
// Per-position mode coefficients of every chunk, computed once for all kernels that need them:
// with E_t the in-chunk cumulative log-decay (float-pair scan of the token rates, Sec. 3.2) and
// kappa = (1 - exp(-e_t/tau)) w_write,
//   f = w_read exp(-E_t/tau)   s = kappa u   u = exp(-(E_end - E_t)/tau)   d = exp(-E_t/tau)
// stored as coef[b, t, h, {f, s, u, d}, K].  d at the chunk's last position is the chunk decay.
// E_t (as the float pair hi + lo) and kappa go to a second array ek[b, t, h, :] for the kernels
// that evaluate pairwise decays (the forward output and the intra-chunk backward).
struct CoefArgs {
    ScanDims d;
    const bf16 *wr, *ww;
    const float *dt, *alpha, *lam, *tau;
    float *coef;
    float *ek;  // per position {E hi, E lo, 0, 0, kappa[K], 0 ...}: tc_ek_width(K) floats
};

template <int KK>
__global__ void __launch_bounds__(TQ) tc_coef(CoefArgs a) {
    __shared__ float2 wsum[4];
    __shared__ float2 Eend_s;
    const ScanDims &d = a.d;
    const int t = threadIdx.x, h = blockIdx.x, c = blockIdx.y, b = blockIdx.z;
    const int c0 = c * TQ, n = min(TQ, d.L - c0);
    float itau[KK], l2t[KK], tmax = 0.f;
#pragma unroll
    for (int m = 0; m < KK; ++m) {
        const float tv = a.tau[h * KK + m];
        itau[m] = 1.f / tv;
        l2t[m] = kLog2e / tv;
        tmax = fmaxf(tmax, tv);
    }
    float e = 0.f, wr[KMAX], ww[KMAX];
#pragma unroll
    for (int m = 0; m < KMAX; ++m) wr[m] = ww[m] = 0.f;
    if (t < n) {
        const size_t i = blh(d, b, c0 + t, h);
        bool cl;
        e = token_rate(a.dt[i], a.alpha[i], a.lam[i], logf(64.f * tmax), &cl);
        load_weights(a.wr + i * KK, KK, wr);
        load_weights(a.ww + i * KK, KK, ww);
    }
    const float2 Et = group_scan128_f2(e, wsum);
    if (t == n - 1) Eend_s = Et;
    __syncthreads();
    const float dEnd = diff_f2(Eend_s, Et);  // E_end - E_t >= 0
    float f[KK], s[KK], u[KK], dv[KK], kp[KK];
#pragma unroll
    for (int m = 0; m < KK; ++m) {
        dv[m] = ex2_approx(-Et.x * l2t[m]);
        u[m] = ex2_approx(-dEnd * l2t[m]);
        f[m] = wr[m] * dv[m];
        kp[m] = -expm1f(-e * itau[m]) * ww[m];
        s[m] = kp[m] * u[m];
    }
    // row t: KK / 4 pieces of each kind, written row-coalesced across KK-lane groups
    uint4 pc[KK];
#pragma unroll
    for (int q = 0; q < KK / 4; ++q) {
        pc[q] = f4_bits(f[4 * q], f[4 * q + 1], f[4 * q + 2], f[4 * q + 3]);
        pc[KK / 4 + q] = f4_bits(s[4 * q], s[4 * q + 1], s[4 * q + 2], s[4 * q + 3]);
        pc[KK / 2 + q] = f4_bits(u[4 * q], u[4 * q + 1], u[4 * q + 2], u[4 * q + 3]);
        pc[3 * KK / 4 + q] = f4_bits(dv[4 * q], dv[4 * q + 1], dv[4 * q + 2], dv[4 * q + 3]);
    }
    const int tg = t & ~(KK - 1);
    put_rows<KK, false>(pc, reinterpret_cast<unsigned char *>(a.coef + blh(d, b, c0 + tg, h) * 4 * KK),
                        size_t(d.H) * 4 * KK * 4, n - tg);
    // ek row: {E hi, E lo, 0, 0}, kappa in KK / 4 pieces, zero padding (EK / 4 pieces in all)
    constexpr int EK = KK == 8 ? 16 : 8;
    uint4 pe[EK / 4];
    pe[0] = f4_bits(Et.x, Et.y, 0.f, 0.f);
#pragma unroll
    for (int q = 0; q < KK / 4; ++q) pe[1 + q] = f4_bits(kp[4 * q], kp[4 * q + 1], kp[4 * q + 2], kp[4 * q + 3]);
#pragma unroll
    for (int q = 1 + KK / 4; q < EK / 4; ++q) pe[q] = make_uint4(0, 0, 0, 0);
    const int te = t & ~(EK / 4 - 1);
    put_rows<EK / 4, false>(pe, reinterpret_cast<unsigned char *>(a.ek + blh(d, b, c0 + te, h) * EK),
                            size_t(d.H) * EK * 4, n - te);
}

// Shared-memory plan of tc_state_pass (offsets from a 1024-aligned base): about 83 KB at N = 128
// (two CTAs share an SM).
struct StateSmem {
    int a_bytes, v_bytes, total;
    __host__ __device__ explicit StateSmem(int N) {
        a_bytes = 2 * 16384;         // 2 M-atoms x (128 k rows x 128 B), MN-major
        v_bytes = (N / 64) * 16384;  // N/64 boxes of [128 t][64 n]
        total = a_bytes + v_bytes + 8 * 2048 /*emit staging, one 2 KB tile per warp*/ + 32 * 4 /*dec*/ +
                64 /*bars*/;
    }
};

// P-slice of one state-pass CTA: the 128 TMEM lanes hold (mode, p) for all KK modes.
template <int KK>
__host__ __device__ constexpr int state_tps() {
    return TQ / KK;
}

// Two groups of four warps share the 128 TMEM lanes: group g writes M-atom g of the A tile and
// emits / decays the state columns [g N / 2, (g + 1) N / 2).
constexpr int kSPThreads = 256;

template <bool REV, int KK>
__global__ void __launch_bounds__(kSPThreads, 2)
    tc_state_pass(const __grid_constant__ CUtensorMap mapV, const __grid_constant__ CUtensorMap mapE, StateArgs a) {
    constexpr int TPSK = state_tps<KK>();  // 16 (KK = 8) or 32 (KK = 4)
    constexpr int NX = TPSK / 8;           // 16-byte pieces of one position's x slice
    extern __shared__ unsigned char smem_raw[];
    unsigned char *base =
        reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const ScanDims &d = a.d;
    const int N = d.N, P = d.P;
    const StateSmem plan(N);
    unsigned char *sA = base;
    unsigned char *sV = sA + plan.a_bytes;
    unsigned char *sE = sV + plan.v_bytes;                          // [8 warps][32 rows x 64 B] emit staging
    float *dec = reinterpret_cast<float *>(sE + 8 * 2048);          // [32] this chunk's decay per mode
    uint64_t *bars = reinterpret_cast<uint64_t *>(dec + 32);        // tma, mma
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bars + 2);
    volatile int *abort_s = reinterpret_cast<volatile int *>(tslot + 1);

    const int tid = threadIdx.x, w = tid >> 5, j = tid & 31, grp = tid >> 7, t = tid & 127, w4 = w & 3;
    const int h = blockIdx.y, b = blockIdx.z, p0 = blockIdx.x * TPSK;
    const int g = h / (d.H / d.G);
    const uint32_t ncols = uint32_t(N);  // 64 or 128
    const size_t PN = size_t(P) * N;
    const size_t bh = size_t(b) * d.H + h;
    // this thread's TMEM lane: mode lm, row p0 + lp of the slice; its column half
    const int lm = t / TPSK, lp = t % TPSK;
    const int nblk = N / 32, hb0 = grp * (nblk / 2);  // 32-column blocks [hb0, hb0 + nblk / 2)

    if (tid == 0) {
        mbar_init(&bars[0], 1);
        mbar_init(&bars[1], 1);
        *abort_s = 0;
        fence_barrier_init();
    }
    if (w == 0) tmem_alloc_once(tslot, ncols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    const uint32_t lane_base = tmem + (uint32_t(w4 * 32) << 16);

    // initial state into tensor memory: lane (mode, p), columns n (this group's half)
    {
        const float *src = a.init ? a.init + (bh * KK + lm) * PN + size_t(p0 + lp) * N : nullptr;
        for (int c8 = 32 * hb0; c8 < 32 * hb0 + N / 2; c8 += 8) {
            float v[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) v[i] = src ? src[c8 + i] : 0.f;
            tmem_st8(lane_base + c8, v);
        }
    }
    tmem_st_wait();
    if (!REV && d.expire_ns) {
        // Test hook of the bounded waits: the MMA barrier has not been signalled (nothing is
        // issued yet), so this wait runs out, and the CTA leaves through the timeout path below
        // with no TMA load, bulk store or MMA of its own in flight.
        __syncthreads();
        if (tid == 0 && !mbar_wait(&bars[1], 0, d.expire_ns)) *abort_s = 1;
        __syncthreads();
    }

    // Thread t of each group owns chunk position t: its slice of x (or dy) and its coefficient
    // per mode (s = kappa exp(-(E_end - E_t)/tau) forward, f = w_read exp(-E_t/tau) reverse) stay
    // in registers, and the inputs of chunk ci + 1 are fetched while chunk ci is processed.
    constexpr int NC = KK / 4;  // 16-byte pieces of one coefficient kind
    uint4 nx[NX], ncv[NC];
    float ndec = 0.f;
    auto fetch = [&](int ci_) {
        const int c_ = REV ? d.nc - 1 - ci_ : ci_;
        const int c0_ = c_ * TQ, n_ = min(TQ, d.L - c0_);
        {  // the slice's TPSK x values and the coefficient row, read row-coalesced (the lane
           // transposes that complete them wait until the chunk that uses them)
            const int tg = t & ~(NX - 1);
            load_rows<NX>(nx, reinterpret_cast<const unsigned char *>(a.U + blh(d, b, c0_ + tg, h) * P + p0),
                          size_t(d.H) * P * 2, n_ - tg);
            const int tc = t & ~(NC - 1);
            load_rows<NC>(ncv,
                          reinterpret_cast<const unsigned char *>(a.coef + blh(d, b, c0_ + tc, h) * 4 * KK +
                                                                  (REV ? 0 : KK)),
                          size_t(d.H) * 4 * KK * 4, n_ - tc);
        }
        if (tid < KK) ndec = a.coef[blh(d, b, c0_ + n_ - 1, h) * 4 * KK + 3 * KK + tid];
    };
    if (d.nc > 0) fetch(0);

    int phase = 0;
    for (int ci = 0; ci < d.nc; ++ci, phase ^= 1) {
        const int c = REV ? d.nc - 1 - ci : ci;
        const int c0 = c * TQ;
        uint4 xr[NX];
        float cv[KK];
#pragma unroll
        for (int q = 0; q < NX; ++q) xr[q] = nx[q];
        lane_transpose<NX>(xr, j);
        lane_transpose<NC>(ncv, j);
#pragma unroll
        for (int q = 0; q < NC; ++q) {
            cv[4 * q] = __uint_as_float(ncv[q].x);
            cv[4 * q + 1] = __uint_as_float(ncv[q].y);
            cv[4 * q + 2] = __uint_as_float(ncv[q].z);
            cv[4 * q + 3] = __uint_as_float(ncv[q].w);
        }
        if (tid < KK) dec[tid] = ndec;  // the previous chunk's emit has passed the barrier before its MMAs
        if (ci + 1 < d.nc) fetch(ci + 1);
        if (ci > 0) {  // previous chunk's MMAs done: tensor memory, sA and sV are free
            if (!mbar_wait(&bars[1], phase ^ 1)) *abort_s = 1;
        }
        __syncthreads();
        if (*abort_s) break;
        tc_fence_after();
        if (tid == 0) {
            mbar_arrive_expect_tx(&bars[0], uint32_t(N * TQ * 2));
            for (int jb = 0; jb < N / 64; ++jb)
                tma_load_3d(sV + jb * 16384, &mapV, &bars[0], g * N + 64 * jb, c0, b);
        }
        // A[(m, p), k] = s_{k,m} x_{k,p} as bf16, MN-major: row k = this thread's position,
        // 64-element M-atoms (64 / TPSK modes x TPSK p each), 128-byte swizzle; group g writes atom g.
        // Packed bf16 products (one instruction per two elements; s rounded to bf16 first)
        {
            unsigned char *row = sA + grp * 16384 + t * 128;
#pragma unroll
            for (int c8 = 0; c8 < 8; ++c8) {  // elements M = 64 grp + 8 c8 ..: mode M / TPSK
                const float s = grp == 0 ? cv[(8 * c8) / TPSK] : cv[(64 + 8 * c8) / TPSK];
                const __nv_bfloat162 s2 = __float2bfloat162_rn(s);
                const uint4 xv = xr[c8 % NX];
                *reinterpret_cast<uint4 *>(row + ((c8 ^ (t & 7)) * 16)) =
                    make_uint4(bf16x2_mul(xv.x, s2), bf16x2_mul(xv.y, s2), bf16x2_mul(xv.z, s2), bf16x2_mul(xv.w, s2));
            }
        }
        // emit the entering state (bf16) and apply the chunk's decay in place (the TMEM load of
        // the next 32 columns is in flight while the current ones are processed).  Each warp's 32
        // rows x 32 columns go through a 2 KB staging tile (64-byte swizzle) and one TMA store:
        // rows (mode, p) of the warp are (32 w4 / TPSK + lane / TPSK, p0 + lane % TPSK).
        {
            const float dm = dec[lm];
            unsigned char *stg = sE + w * 2048;
            const int rowE = int((bh * d.nc + c) * KK + (32 * w4) / TPSK);
            auto process = [&](float *v, int blk) {
                if (j == 0) bulk_wait_read();  // the previous store has read the staging tile
                __syncwarp();
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    *reinterpret_cast<uint4 *>(stg + j * 64 + ((q ^ ((j >> 1) & 3)) * 16)) =
                        make_uint4(pack_bf16x2(v[8 * q], v[8 * q + 1]), pack_bf16x2(v[8 * q + 2], v[8 * q + 3]),
                                   pack_bf16x2(v[8 * q + 4], v[8 * q + 5]), pack_bf16x2(v[8 * q + 6], v[8 * q + 7]));
                fence_async_smem();
                __syncwarp();
                if (j == 0) {
                    tma_store_3d(&mapE, stg, 32 * blk, p0, rowE);
                    bulk_commit();
                }
#pragma unroll
                for (int i = 0; i < 32; ++i) v[i] *= dm;
#pragma unroll
                for (int q = 0; q < 4; ++q) tmem_st8(lane_base + 32 * blk + 8 * q, v + 8 * q);
            };
            float v0[32], v1[32];
            tmem_ld32(lane_base + 32 * hb0, v0);
            if (nblk == 4) {
                tmem_ld_wait();
                tmem_ld32(lane_base + 32 * (hb0 + 1), v1);
                process(v0, hb0);
                tmem_ld_wait();
                process(v1, hb0 + 1);
            } else {  // N = 64: one block per group
                tmem_ld_wait();
                process(v0, hb0);
            }
        }
        tmem_st_wait();
        fence_async_smem();
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
        if (tid == 0) {
            if (!mbar_wait(&bars[0], phase)) {
                *abort_s = 1;
            } else {
                const uint32_t idesc = idesc_bf16(128, N, true, true);
                // descriptors advance by (byte offset >> 4) in their start-address field
                const uint64_t ad0 = desc_sw128(smem_u32(sA), 16384, 1024);
                const uint64_t bd0 = desc_sw128(smem_u32(sV), 16384, 1024);
#pragma unroll
                for (int ks = 0; ks < TQ / 16; ++ks)
                    mma_bf16(tmem, ad0 + uint64_t((ks * 2048) >> 4), bd0 + uint64_t((ks * 2048) >> 4), idesc, 1);
                mma_commit(&bars[1]);
            }
        }
    }
    // drain: last chunk's MMAs
    __syncthreads();
    if (!*abort_s && d.nc > 0) {
        if (!mbar_wait(&bars[1], phase ^ 1)) *abort_s = 1;
    }
    __syncthreads();
    tc_fence_after();
    if (!*abort_s && a.fin) {
        float *dst = a.fin + (bh * KK + lm) * PN + size_t(p0 + lp) * N;
        for (int c32 = 32 * hb0; c32 < 32 * hb0 + N / 2; c32 += 32) {
            float v[32];
            tmem_ld32(lane_base + c32, v);
            tmem_ld_wait();
            float4 *o = reinterpret_cast<float4 *>(dst + c32);
#pragma unroll
            for (int q = 0; q < 8; ++q) o[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        }
    }
    if (j == 0) bulk_wait_all();  // this warp's emit stores are complete
    if (*abort_s && tid == 0) atomicExch(a.err, kTimeoutCode);
    tc_fence_before();
    __syncthreads();
    if (w == 0) tmem_dealloc(tmem, ncols);
}

// ---------------------------------------------------------------------------------------------
struct OutArgs {
    ScanDims d;
    const float *coef, *ek;  // tc_coef's per-position coefficients and {E, kappa}
    const bf16 *wr, *ww;
    const float *dt, *alpha, *lam, *tau, *D;
    bf16 *y;
    int *err;
};

constexpr int kOutThreads = 256;  // two groups of four warps share the 128 TMEM lanes
constexpr int kOutLaunch = kOutThreads + 64;  // a ninth warp issues the entering-state MMAs, a
                                              // tenth loads their S_in tiles
constexpr int kSBuf = 3;          // 8 KB units of the S ring (the Gamma operands, then one S_in pair slot)

// Shared-memory plan of tc_chunk_fwd (offsets from a 1024-aligned base): about 110 KB at
// N = 128, so that two CTAs share an SM.
struct OutSmem {
    int c, m, x, s, total;
    __host__ __device__ explicit OutSmem(int N) {
        c = (N / 64) * 16384;  // C chunk [t][n], K-major, 64-wide n atoms
        m = 2 * 16384;         // B chunk, then Gamma o G [t][k]
        x = 16384;             // x chunk [t][p]: the MN-major operand of the intra MMA
        s = kSBuf * 8192;      // U / V tf32 tiles of Gamma, then one S_in pair slot: [2 x 64 p][64 n]
        total = c + m + x + s + TQ * KMAX * 4 /*kappa*/ + TQ * 8 /*E*/ + 64 * 4 /*tau, l2t*/ +
                64 /*wsum*/ + 24 * 8 /*bars*/ + 16 + 64 * KMAX * 4 /*V16*/;
    }
};


// The entering-state MMAs of tc_chunk_fwd (one thread of the ninth warp).  Two modes go
// together: pair tile j = (mode pair j / nhalf, 64-wide n half j % nhalf) stacks the [64 p][64 n]
// S_in tiles of modes 2 mp and 2 mp + 1 into one 16 KB slot, the B operand of one N = 128
// product, so Z_{2mp}, Z_{2mp+1} = C S_in^T land side by side in TMEM buffer mp % 2 (128
// columns) once the compute threads have read its previous contents.  Slots: the first 16 KB
// of the S ring, then the two halves of the Gamma o G tile once the intra MMA has read it.
// bars: 3 + s slot s loaded | 6 + s slot s read by its MMAs | 9 + zb Z buffer written |
//       13 + zb Z buffer read by all compute threads (buffer 1: first the intra Y)
constexpr int kZSlots = 3;
__device__ __forceinline__ void chunk_fwd_issuer(const ScanDims &d, unsigned char *sC, unsigned char *sS,
                                                 unsigned char *sM, uint64_t *bars, volatile int *abort_s,
                                                 uint32_t tmem) {
    const int nhalf = d.N / 64, npair = d.K / 2, ntile = npair * nhalf;
    auto slot = [&](int s) { return s == 0 ? sS : sM + (s - 1) * 16384; };
    // the intra Y MMA (issued after the Gamma o G pass) frees the G and Gamma columns
    if (!mbar_wait(&bars[2], 0)) {
        *abort_s = 1;
        return;
    }
    tc_fence_after();
    const uint32_t idZ = idesc_bf16(128, 128, false, false);
    for (int j = 0; j < ntile && !*abort_s; ++j) {
        const int mp = j / nhalf, hn = j % nhalf, zb = mp & 1, s = j % kZSlots;
        if (hn == 0) {  // buffer zb read by all compute threads (buffer 1: first the intra Y)
            const int k = mp >> 1;
            if ((zb == 1 || k > 0) && !mbar_wait(&bars[13 + zb], (zb == 1 ? k : k - 1) & 1)) {
                *abort_s = 1;
                break;
            }
        }
        if (!mbar_wait(&bars[3 + s], (j / kZSlots) & 1)) {
            *abort_s = 1;
            break;
        }
        tc_fence_after();
        const uint64_t da = desc_sw128(smem_u32(sC) + hn * 16384, 16, 1024), db = desc_sw128(smem_u32(slot(s)), 16, 1024);
#pragma unroll
        for (int ks = 0; ks < 4; ++ks)
            mma_bf16(tmem + 128 * zb, desc_add(da, ks * 32), desc_add(db, ks * 32), idZ, (hn > 0 || ks > 0) ? 1u : 0u);
        mma_commit(&bars[6 + s]);  // the slot, once its MMAs have read it
        if (hn == nhalf - 1) mma_commit(&bars[9 + zb]);
    }
}

// The S_in pair tiles of tc_chunk_fwd (one thread of the tenth warp): slot s of the ring takes
// tile j + kZSlots once the MMAs of tile j have read it.  The first slot waits for the Gamma
// MMAs (it held their operands), the other two for the intra Y MMA (the Gamma o G tile).
__device__ __forceinline__ void chunk_fwd_loader(const ScanDims &d, unsigned char *sS, unsigned char *sM,
                                                 uint64_t *bars, volatile int *abort_s, const CUtensorMap &mapS,
                                                 int srow) {
    const int nhalf = d.N / 64, npair = d.K / 2, ntile = npair * nhalf;
    auto slot = [&](int s) { return s == 0 ? sS : sM + (s - 1) * 16384; };
    auto load = [&](int j) {
        const int s = j % kZSlots, mp = j / nhalf, hn = j % nhalf;
        mbar_arrive_expect_tx(&bars[3 + s], 16384u);
        tma_load_3d(slot(s), &mapS, &bars[3 + s], hn * 64, 0, srow + 2 * mp);
        tma_load_3d(slot(s) + 8192, &mapS, &bars[3 + s], hn * 64, 0, srow + 2 * mp + 1);
    };
    if (!mbar_wait(&bars[1], 0)) {
        *abort_s = 1;
        return;
    }
    if (ntile > 0) load(0);
    if (!mbar_wait(&bars[2], 0)) {
        *abort_s = 1;
        return;
    }
    for (int j = 1; j < min(kZSlots, ntile); ++j) load(j);
    for (int j = 0; j + kZSlots < ntile && !*abort_s; ++j) {
        if (!mbar_wait(&bars[6 + j % kZSlots], (j / kZSlots) & 1)) {
            *abort_s = 1;
            break;
        }
        load(j + kZSlots);
    }
}

// One CTA per (b, h, chunk), headdim 64:
//   Y  = (Gamma o C B^T) X                      (intra-chunk pairs, K = t; tensor memory)
//   y  = Y + sum_m f_m o (C S_in,m^T) + D x     (entering state)
// G = C B^T comes from the tensor cores; Gamma is formed per position pair.  A ninth warp
// streams Z_m = C S_in,m^T, two modes per N = 128 product, through two 128-column TMEM buffers
// (S_in tiles by TMA, two pair tiles ahead) while the 256 compute threads fold each Z_m into
// their rows of y with the weight f_m[t]: no per-mode scaled operand and no CTA-wide barrier.
__global__ void __launch_bounds__(kOutLaunch, 2)
    tc_chunk_fwd(const __grid_constant__ CUtensorMap mapC, const __grid_constant__ CUtensorMap mapB,
                 const __grid_constant__ CUtensorMap mapX, const __grid_constant__ CUtensorMap mapS,
                 OutArgs a) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char *base =
        reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const ScanDims &d = a.d;
    const int K = d.K, N = d.N, P = d.P;
    const OutSmem plan(N);
    unsigned char *sC = base;
    unsigned char *sM = sC + plan.c;
    unsigned char *sX = sM + plan.m;
    unsigned char *sS = sX + plan.x;
    float *kap_s = reinterpret_cast<float *>(sS + plan.s);      // [128][KMAX]
    float2 *E_s = reinterpret_cast<float2 *>(kap_s + TQ * KMAX);  // [128] hi / lo pairs
    float *tau_s = reinterpret_cast<float *>(E_s + TQ);           // [32]
    float *l2t = tau_s + 32;                                      // [32] log2(e) / tau
    float2 *wsum = reinterpret_cast<float2 *>(l2t + 32);          // [8]
    // bars: 0 C, B, x loaded | 1 G done | 2 intra Y done | 3..5 S tile loaded | 6..8 S tile read
    //       by its MMAs | 9..12 Z buffer written | 13..16 Z buffer read (all compute threads)
    uint64_t *bars = reinterpret_cast<uint64_t *>(wsum + 8);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bars + 17);
    volatile int *abort_s = reinterpret_cast<volatile int *>(tslot + 1);
    // the lower-left 16 x 16 quarter of each diagonal 32 x 32 block, factored through E at the
    // block's 16th position: V16 [64 (block, k mod 16)][KMAX] = kappa exp(-(E_a16 - E_k)/tau)
    float *V16s = reinterpret_cast<float *>(bars + 24);

    const int tid = threadIdx.x, grp = tid >> 7, t = tid & 127, w4 = (tid >> 5) & 3;
    const int h = blockIdx.x, c = blockIdx.y, b = blockIdx.z;
    const int g = h / (d.H / d.G);
    const int c0 = c * TQ, n = min(TQ, d.L - c0);
    const int nhalf = N / 64;
    const int srow = int(((size_t(b) * d.H + h) * d.nc + c) * K);

    if (tid == kOutThreads + 32) {  // the loading warp: barriers, then C, B and x at once
        for (int i = 0; i < 13; ++i) mbar_init(&bars[i], 1);
        for (int i = 13; i < 15; ++i) mbar_init(&bars[i], kOutThreads);
        *abort_s = 0;
        fence_barrier_init();
        mbar_arrive_expect_tx(&bars[0], uint32_t(2 * plan.c + plan.x));
        for (int jb = 0; jb < nhalf; ++jb) {
            tma_load_3d(sC + jb * 16384, &mapC, &bars[0], g * N + 64 * jb, c0, b);
            tma_load_3d(sM + jb * 16384, &mapB, &bars[0], g * N + 64 * jb, c0, b);
        }
        tma_load_3d(sX, &mapX, &bars[0], h * P, c0, b);
    }
    if (tid < K) {
        const float tv = a.tau[h * K + tid];
        tau_s[tid] = tv;
        l2t[tid] = kLog2e / tv;
    }
    if (tid < 32) tmem_alloc_once(tslot, 256);
    // per-position inputs of row t, all loads issued before anything waits on them: w_read, and
    // from tc_coef the cumulative log-decay E (hi, lo), kappa and f = w_read exp(-E/tau) (rows
    // read row-coalesced; rows t >= n read as zero)
    float wr_t[KMAX], kap_t[KMAX], f_t[KMAX];
    float2 Et2;
    {
        if (t < n)
            load_weights(a.wr + blh(d, b, c0 + t, h) * K, K, wr_t);
        else
#pragma unroll
            for (int m = 0; m < KMAX; ++m) wr_t[m] = 0.f;
        auto fl = [](uint4 v, float *o) {
            o[0] = __uint_as_float(v.x);
            o[1] = __uint_as_float(v.y);
            o[2] = __uint_as_float(v.z);
            o[3] = __uint_as_float(v.w);
        };
        if (K == 8) {
            uint4 pe[4], pf[2];
            get_rows<4>(pe, reinterpret_cast<const unsigned char *>(a.ek + blh(d, b, c0 + (t & ~3), h) * 16),
                        size_t(d.H) * 64, n - (t & ~3));
            get_rows<2>(pf, reinterpret_cast<const unsigned char *>(a.coef + blh(d, b, c0 + (t & ~1), h) * 32),
                        size_t(d.H) * 128, n - (t & ~1));
            Et2 = make_float2(__uint_as_float(pe[0].x), __uint_as_float(pe[0].y));
            fl(pe[1], kap_t);
            fl(pe[2], kap_t + 4);
            // past the end of a ragged chunk E stays at its last value (zero token rates)
            if (t >= n) Et2 = *reinterpret_cast<const float2 *>(a.ek + blh(d, b, c0 + n - 1, h) * 16);
            fl(pf[0], f_t);
            fl(pf[1], f_t + 4);
        } else {  // K == 4
            uint4 pe[2], pf[1];
            get_rows<2>(pe, reinterpret_cast<const unsigned char *>(a.ek + blh(d, b, c0 + (t & ~1), h) * 8),
                        size_t(d.H) * 32, n - (t & ~1));
            get_rows<1>(pf, reinterpret_cast<const unsigned char *>(a.coef + blh(d, b, c0 + t, h) * 16),
                        size_t(d.H) * 64, n - t);
            Et2 = make_float2(__uint_as_float(pe[0].x), __uint_as_float(pe[0].y));
            fl(pe[1], kap_t);
            fl(pf[0], f_t);
            if (t >= n) Et2 = *reinterpret_cast<const float2 *>(a.ek + blh(d, b, c0 + n - 1, h) * 8);
#pragma unroll
            for (int m = 4; m < KMAX; ++m) kap_t[m] = f_t[m] = 0.f;
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    const uint32_t lane_base = tmem + (uint32_t(w4 * 32) << 16);
    // TMEM: G = C B^T at [0, 128), the factored Gamma blocks at [128, 256); then the intra Y at
    // [192, 256) and the Z buffers of mode pairs at 128 (pair % 2) (buffer 1 once Y has been read)
    constexpr uint32_t colG = 0, colGam = 128, colY = 192;
    if (tid >= kOutThreads) {
        if (tid == kOutThreads) chunk_fwd_issuer(a.d, sC, sS, sM, bars, abort_s, tmem);
        if (tid == kOutThreads + 32) chunk_fwd_loader(a.d, sS, sM, bars, abort_s, mapS, srow);
    } else {

    if (grp == 0) {
        E_s[t] = Et2;
#pragma unroll
        for (int m = 0; m < KMAX; ++m) kap_s[t * KMAX + m] = kap_t[m];
    }
    sync_first256();
    // Gamma below the diagonal 32 x 32 blocks, factored through the log-decay E_a at the end of
    // the column block J: exp(-(E_t - E_k)/tau) = exp(-(E_t - E_a)/tau) exp(-(E_a - E_k)/tau),
    // both factors <= 1, so Gamma[t, k in J] = sum_m U_J[t, m] V[k, m] (a K = 8 tf32 product):
    //   U_J[t, m] = w_read[t, m] exp(-(E_t - E_a)/tau_m)   (rows t of later blocks, else 0)
    //   V[k, m]   = kappa[k, m] exp(-(E_a - E_k)/tau_m)
    // U: [128 t][4 J x 8 m] and V: [32 k mod 32][4 J x 8 m], 128-byte swizzled, in the S ring.
    unsigned char *sU = sS, *sVt = sS + 16384;
    if (grp == 0) {
        const int I = t >> 5;
        unsigned char *row = sU + t * 128;
#pragma unroll
        for (int J = 0; J < 4; ++J) {
            uint32_t u[8];
            const float dE = diff_f2(Et2, E_s[32 * J + 31]);
#pragma unroll
            for (int m = 0; m < KMAX; ++m)
                u[m] = (J < I && m < K && t < n) ? to_tf32(wr_t[m] * ex2_approx(-dE * l2t[m])) : 0u;
            *reinterpret_cast<uint4 *>(row + (((2 * J) ^ (t & 7)) * 16)) = make_uint4(u[0], u[1], u[2], u[3]);
            *reinterpret_cast<uint4 *>(row + (((2 * J + 1) ^ (t & 7)) * 16)) = make_uint4(u[4], u[5], u[6], u[7]);
        }
    } else {
        const int J = t >> 5, r = t & 31;
        const float dE = diff_f2(E_s[32 * J + 31], Et2);
        uint32_t v[8];
#pragma unroll
        for (int m = 0; m < KMAX; ++m) v[m] = m < K ? to_tf32(kap_t[m] * ex2_approx(-dE * l2t[m])) : 0u;
        unsigned char *row = sVt + r * 128;
        *reinterpret_cast<uint4 *>(row + (((2 * J) ^ (r & 7)) * 16)) = make_uint4(v[0], v[1], v[2], v[3]);
        *reinterpret_cast<uint4 *>(row + (((2 * J + 1) ^ (r & 7)) * 16)) = make_uint4(v[4], v[5], v[6], v[7]);
        if (r < 16) {  // left half of its block: V16 against the anchor 32 J + 15
            const float dE16 = diff_f2(E_s[32 * J + 15], Et2);
#pragma unroll
            for (int m = 0; m < KMAX; ++m)
                V16s[(16 * J + r) * KMAX + m] = m < K ? kap_t[m] * ex2_approx(-dE16 * l2t[m]) : 0.f;
        }
    }
    fence_async_smem();
    sync_first256();
    // G = C B^T (bf16) and the four Gamma column blocks (tf32)
    if (tid == 0) {
        if (!mbar_wait(&bars[0], 0)) {
            *abort_s = 1;
        } else {
            tc_fence_after();
            const uint32_t idG = idesc_bf16(128, 128, false, false);
            for (int ks = 0; ks < N / 16; ++ks) {
                const uint32_t koff = (ks / 4) * 16384 + (ks % 4) * 32;
                mma_bf16(tmem + colG, desc_sw128(smem_u32(sC) + koff, 16, 1024),
                         desc_sw128(smem_u32(sM) + koff, 16, 1024), idG, ks > 0);
            }
            const uint32_t idT = idesc_tf32(128, 32);
            for (int J = 0; J < 4; ++J)
                mma_tf32(tmem + colGam + 32 * J, desc_sw128(smem_u32(sU) + 32 * J, 16, 1024),
                         desc_sw128(smem_u32(sVt) + 32 * J, 16, 1024), idT, 0);
            mma_commit(&bars[1]);
        }
    }
    sync_first256();
    if (!*abort_s && !mbar_wait(&bars[1], 0)) *abort_s = 1;
    sync_first256();
    tc_fence_after();
    if (!*abort_s) {
        // row t of Gamma o G -> bf16, K-major [t][k] over the B tile.  Warp rows are one 32-block
        // I; column block kc < I takes the factored Gamma, kc == I the direct sum (pairs k <= t),
        // kc > I is zero.  The 8-column items (kc, q8) alternate between the two groups, so both
        // take half of every block (the diagonal one included); loops stay rolled (compact code)
        const int I = t >> 5;
#pragma unroll 1
        for (int it = grp; it < 16; it += 2) {
            const int kc = it >> 2;
            int q8 = it & 3;
            float gv[8];
            if (kc == I) {
                // the diagonal block in 16 x 16 quarters: the two on the diagonal sum their pairs
                // k <= t directly, the lower-left one is factored through E at 32 I + 15 (both
                // factors <= 1), the upper-right one is zero.  The direct step gives every lane
                // its own diagonal quarter (upper rows: left half, lower rows: right half), the
                // other step the rest (lower rows: factored, upper rows: zero).
                const bool upper = (t & 31) < 16, dstep = q8 == grp;
                q8 = (dstep == upper) ? grp : grp + 2;  // this lane's 8 columns
                const int k0 = 32 * kc + 8 * q8;
                {
                    float ga[8], gb[8];
                    tmem_ld8(lane_base + colG + 32 * kc + 8 * grp, ga);
                    tmem_ld8(lane_base + colG + 32 * kc + 8 * grp + 16, gb);
                    tmem_ld_wait();
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) gv[kk] = q8 == grp ? ga[kk] : gb[kk];
                }
                if (dstep) {
                    // branch-free over the eight columns (a pair above the diagonal runs with its
                    // decay exponent clamped to zero and is masked after), modes in packed float32
                    // pairs (K is even)
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) {
                        const int k = k0 + kk;
                        const bool valid = k <= t && t < n;
                        const float dE = fmaxf(diff_f2(Et2, E_s[k]), 0.f);
                        const float4 ka = *reinterpret_cast<const float4 *>(kap_s + k * KMAX);
                        const float4 kb = *reinterpret_cast<const float4 *>(kap_s + k * KMAX + 4);
                        const float kpv[8] = {ka.x, ka.y, ka.z, ka.w, kb.x, kb.y, kb.z, kb.w};
                        const float2 ndE = make_float2(-dE, -dE);
                        float2 g2 = make_float2(0.f, 0.f);
#pragma unroll
                        for (int m = 0; m < KMAX; m += 2) {
                            if (m < K) {
                                const float2 x2 = __fmul2_rn(ndE, make_float2(l2t[m], l2t[m + 1]));
                                g2 = __ffma2_rn(__fmul2_rn(make_float2(wr_t[m], wr_t[m + 1]), make_float2(kpv[m], kpv[m + 1])),
                                                make_float2(ex2_approx(x2.x), ex2_approx(x2.y)), g2);
                            }
                        }
                        gv[kk] = valid ? (g2.x + g2.y) * gv[kk] : 0.f;
                    }
                } else if (!upper) {
                    const float dE = diff_f2(Et2, E_s[32 * kc + 15]);
                    float u16[KMAX];
#pragma unroll
                    for (int m = 0; m < KMAX; ++m) u16[m] = m < K ? wr_t[m] * ex2_approx(-dE * l2t[m]) : 0.f;
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) {  // the K = 8 mode sum in packed float32 pairs
                        const float *v16 = V16s + (16 * kc + ((k0 + kk) & 15)) * KMAX;
                        const float4 v0 = *reinterpret_cast<const float4 *>(v16);
                        const float4 v1 = *reinterpret_cast<const float4 *>(v16 + 4);
                        float2 g2 = __fmul2_rn(make_float2(u16[0], u16[1]), make_float2(v0.x, v0.y));
                        g2 = __ffma2_rn(make_float2(u16[2], u16[3]), make_float2(v0.z, v0.w), g2);
                        g2 = __ffma2_rn(make_float2(u16[4], u16[5]), make_float2(v1.x, v1.y), g2);
                        g2 = __ffma2_rn(make_float2(u16[6], u16[7]), make_float2(v1.z, v1.w), g2);
                        gv[kk] = t < n ? (g2.x + g2.y) * gv[kk] : 0.f;
                    }
                } else {
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) gv[kk] = 0.f;
                }
            } else if (kc < I) {
                const int k0 = 32 * kc + 8 * q8;
                float gm[8];
                tmem_ld8(lane_base + colG + k0, gv);
                tmem_ld8(lane_base + colGam + k0, gm);
                tmem_ld_wait();
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) gv[kk] *= gm[kk];
            } else {
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) gv[kk] = 0.f;
            }
            *reinterpret_cast<uint4 *>(sM + (kc >> 1) * 16384 + t * 128 + ((((kc & 1) * 4 + q8) ^ (t & 7)) * 16)) =
                make_uint4(pack_bf16x2(gv[0], gv[1]), pack_bf16x2(gv[2], gv[3]), pack_bf16x2(gv[4], gv[5]),
                           pack_bf16x2(gv[6], gv[7]));
        }
    }
    fence_async_smem();
    tc_fence_before();
    sync_first256();
    tc_fence_after();
    if (tid == 0 && !*abort_s) {  // Y = (Gamma o G) X: M = t, N = p, K = k (over G's columns)
        const uint32_t idY = idesc_bf16(128, 64, false, true);
        for (int ks = 0; ks < TQ / 16; ++ks)
            mma_bf16(tmem + colY, desc_sw128(smem_u32(sM) + (ks / 4) * 16384 + (ks % 4) * 32, 16, 1024),
                     desc_sw128(smem_u32(sX) + ks * 2048, 16384, 1024), idY, ks > 0);
        mma_commit(&bars[2]);
    }
    // y row t (group g: p in [32 g, 32 g + 32)): the intra Y from tensor memory, then every
    // mode's Z_m = C S_in,m^T weighted by f_m[t]; each buffer read is handed back to the issuer
    float yv[32];
    if (!*abort_s && !mbar_wait(&bars[2], 0)) *abort_s = 1;
    tc_fence_after();
    tmem_ld32(lane_base + colY + grp * 32, yv);
    tmem_ld_wait();
    tc_fence_before();
    mbar_arrive(&bars[13 + 1]);
#pragma unroll
    for (int mp = 0; mp < KMAX / 2; ++mp) {
        if (2 * mp < K) {
            const int zb = mp & 1;
            if (!*abort_s && !mbar_wait(&bars[9 + zb], (mp >> 1) & 1)) *abort_s = 1;
            tc_fence_after();
            float z0[32], z1[32];
            tmem_ld32(lane_base + 128 * zb + grp * 32, z0);
            tmem_ld32(lane_base + 128 * zb + 64 + grp * 32, z1);
            tmem_ld_wait();
            tc_fence_before();
            mbar_arrive(&bars[13 + zb]);
            const float f0 = f_t[2 * mp], f1 = f_t[2 * mp + 1];
#pragma unroll
            for (int i = 0; i < 32; ++i) yv[i] = fmaf(f1, z1[i], fmaf(f0, z0[i], yv[i]));
        }
    }
    {  // y = Y + sum_m f_m Z_m + D x (rows t >= n and aborted CTAs write nothing)
        const float Dh = a.D[h];
        const unsigned char *xrow = sX + t * 128;
        uint4 e[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const uint4 u = *reinterpret_cast<const uint4 *>(xrow + (((grp * 4 + q) ^ (t & 7)) * 16));
            const uint32_t xw[4] = {u.x, u.y, u.z, u.w};
            uint32_t r[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float2 f = bf16x2_to_float2(xw[i]);
                r[i] = pack_bf16x2(fmaf(Dh, f.x, yv[8 * q + 2 * i]), fmaf(Dh, f.y, yv[8 * q + 2 * i + 1]));
            }
            e[q] = make_uint4(r[0], r[1], r[2], r[3]);
        }
        const int t4 = t & ~3;
        put_rows<4, false>(e, reinterpret_cast<unsigned char *>(a.y + blh(d, b, c0 + t4, h) * P + grp * 32),
                           size_t(d.H) * P * 2, *abort_s ? 0 : n - t4);
    }
    }  // compute threads
    if (*abort_s && tid == 0) atomicExch(a.err, kTimeoutCode);
    tc_fence_before();
    __syncthreads();
    if (tid < 32) tmem_dealloc(tmem, 256);
}

// ------------------------------------------------------------------------------------- host
typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    }
    return fn;
}

}  // namespace

// 3-D bf16 tensor map, innermost dimension first; 128-byte swizzle.
bool tc_make_map3(CUtensorMap *m, const void *ptr, uint64_t d0, uint64_t d1, uint64_t d2,
               uint64_t stride1_bytes, uint64_t stride2_bytes, uint32_t b0, uint32_t b1,
               uint32_t b2, int swizzle_bytes) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[3] = {d0, d1, d2};
    const cuuint64_t strides[2] = {stride1_bytes, stride2_bytes};
    const cuuint32_t box[3] = {b0, b1, b2};
    const cuuint32_t es[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(ptr), dims, strides, box,
              es, CU_TENSOR_MAP_INTERLEAVE_NONE,
              swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 3-D float32 tensor map, innermost dimension first; 128- or 64-byte swizzle (inner box of 32 or
// 16 floats).
bool tc_make_map3_f32(CUtensorMap *m, const void *ptr, uint64_t d0, uint64_t d1, uint64_t d2,
                      uint64_t stride1_bytes, uint64_t stride2_bytes, uint32_t b0, uint32_t b1,
                      uint32_t b2, int swizzle_bytes) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[3] = {d0, d1, d2};
    const cuuint64_t strides[2] = {stride1_bytes, stride2_bytes};
    const cuuint32_t box[3] = {b0, b1, b2};
    const cuuint32_t es[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<void *>(ptr), dims, strides, box,
              es, CU_TENSOR_MAP_INTERLEAVE_NONE,
              swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 4-D float32 tensor map, innermost dimension first; 128-byte swizzle (inner box of 32 floats).
bool tc_make_map4_f32(CUtensorMap *m, const void *ptr, const uint64_t dims[4], const uint64_t strides_bytes[3],
                      const uint32_t box[4]) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dd[4] = {dims[0], dims[1], dims[2], dims[3]};
    const cuuint64_t ss[3] = {strides_bytes[0], strides_bytes[1], strides_bytes[2]};
    const cuuint32_t bb[4] = {box[0], box[1], box[2], box[3]};
    const cuuint32_t es[4] = {1, 1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, const_cast<void *>(ptr), dd, ss, bb, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool tc_supported(const ScanDims &d, int dtype) {
    if (dtype != 1) return false;
    if (d.P != 64 || (d.N != 64 && d.N != 128) || (d.K != 4 && d.K != 8)) return false;
    return true;
}

size_t tc_state_elems(const ScanDims &d) {
    return size_t(d.B) * d.H * d.nc * d.K * d.P * d.N;
}

size_t tc_coef_elems(const ScanDims &d) { return size_t(d.B) * d.L * d.H * 4 * d.K; }

size_t tc_ek_elems(const ScanDims &d) { return size_t(d.B) * d.L * d.H * tc_ek_width(d.K); }

cudaError_t tc_coef_launch(const ScanDims &d, const ScanPtrs &p, float *coef, float *ek, cudaStream_t st) {
    if (d.nc == 0) return cudaSuccess;
    CoefArgs a;
    a.d = d;
    a.wr = (const bf16 *)p.wr;
    a.ww = (const bf16 *)p.ww;
    a.dt = p.dt; a.alpha = p.alpha; a.lam = p.lam; a.tau = p.tau;
    a.coef = coef;
    a.ek = ek;
    trace_begin("coef_tc", st);
    if (d.K == 8)
        tc_coef<8><<<dim3(d.H, d.nc, d.B), TQ, 0, st>>>(a);
    else
        tc_coef<4><<<dim3(d.H, d.nc, d.B), TQ, 0, st>>>(a);
    trace_end(st);
    return cudaGetLastError();
}

cudaError_t tc_state_pass_launch(const ScanDims &d, bool rev, const void *U, const void *V,
                                 const float *coef, const float *init, void *emit, float *fin,
                                 int *err, cudaStream_t st) {
    CUtensorMap mapV;
    if (!tc_make_map3(&mapV, V, uint64_t(d.G) * d.N, d.L, d.B, uint64_t(d.G) * d.N * 2,
                   uint64_t(d.L) * d.G * d.N * 2, 64, TQ, 1))
        return cudaErrorInvalidValue;
    // per-chunk states [B, H, nc, K, P, N] as (n, p, (b, h, c, m)) rows; a box is one warp's
    // 32 columns x 32 TMEM lanes = 128 / K ... modes x P-slice rows
    CUtensorMap mapE;
    const int tps = 128 / d.K;
    if (!tc_make_map3(&mapE, emit, d.N, d.P, uint64_t(d.B) * d.H * d.nc * d.K, uint64_t(d.N) * 2,
                      uint64_t(d.P) * d.N * 2, 32, uint32_t(tps), uint32_t(32 / tps), 64))
        return cudaErrorInvalidValue;
    StateArgs a;
    a.d = d;
    a.U = (const bf16 *)U;
    a.coef = coef;
    a.init = init;
    a.emit = (bf16 *)emit;
    a.fin = fin;
    a.err = err;
    const size_t smem = StateSmem(d.N).total + 1024;
    auto launch = [&](auto kern, int tps, const char *name) {
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        trace_begin(name, st);
        kern<<<dim3(d.P / tps, d.H, d.B), kSPThreads, smem, st>>>(mapV, mapE, a);
        trace_end(st);
    };
    if (d.K == 8) {
        if (rev)
            launch(tc_state_pass<true, 8>, state_tps<8>(), "state_pass_rev_tc");
        else
            launch(tc_state_pass<false, 8>, state_tps<8>(), "state_pass_fwd_tc");
    } else {
        if (rev)
            launch(tc_state_pass<true, 4>, state_tps<4>(), "state_pass_rev_tc");
        else
            launch(tc_state_pass<false, 4>, state_tps<4>(), "state_pass_fwd_tc");
    }
    return cudaGetLastError();
}

cudaError_t tc_scan_fwd(const ScanDims &d, const ScanPtrs &p, void *S_in, float *coef, float *ek,
                        int *err, cudaStream_t st) {
    cudaError_t e = tc_coef_launch(d, p, coef, ek, st);
    if (e == cudaSuccess) e = tc_state_pass_launch(d, false, p.x, p.Bm, coef, p.h0, S_in, p.h_final, err, st);
    if (e != cudaSuccess || d.nc == 0) return e;
    CUtensorMap mapC, mapB, mapX, mapS;
    const uint64_t GN = uint64_t(d.G) * d.N, HP = uint64_t(d.H) * d.P;
    if (!tc_make_map3(&mapC, p.Cm, GN, d.L, d.B, GN * 2, uint64_t(d.L) * GN * 2, 64, TQ, 1) ||
        !tc_make_map3(&mapB, p.Bm, GN, d.L, d.B, GN * 2, uint64_t(d.L) * GN * 2, 64, TQ, 1) ||
        !tc_make_map3(&mapX, p.x, HP, d.L, d.B, HP * 2, uint64_t(d.L) * HP * 2, 64, TQ, 1) ||
        !tc_make_map3(&mapS, S_in, d.N, d.P, uint64_t(d.B) * d.H * d.nc * d.K, uint64_t(d.N) * 2,
                      uint64_t(d.P) * d.N * 2, 64, 64, 1))
        return cudaErrorInvalidValue;
    OutArgs a;
    a.d = d;
    a.coef = coef;
    a.ek = ek;
    a.wr = (const bf16 *)p.wr;
    a.ww = (const bf16 *)p.ww;
    a.dt = p.dt; a.alpha = p.alpha; a.lam = p.lam; a.tau = p.tau; a.D = p.D;
    a.y = (bf16 *)p.y;
    a.err = err;
    const size_t smem = OutSmem(d.N).total + 1024;
    cudaFuncSetAttribute(tc_chunk_fwd, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    dim3 grid(d.H, d.nc, d.B);
    trace_begin("chunk_fwd_tc", st);
    tc_chunk_fwd<<<grid, kOutLaunch, smem, st>>>(mapC, mapB, mapX, mapS, a);
    trace_end(st);
    return cudaGetLastError();
}

}  // namespace frac
