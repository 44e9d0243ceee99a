// Intra-chunk part of the timescale gradient (the learned-timescale variant, App. G), on the
// CUDA cores, run only when frac_scan_bwd is asked for dtau.
//
// dtau_m = tau_m^-2 sum_t e_t (rho_t <dS_t, S_{t-1}>_m - dkappa_{t,m} rho_{t,m} w_write_{t,m}).
// The backward kernels add the terms that involve the entering state S_in or the leaving
// adjoint dS_out (each weighted by the e_t it spans: E_t, E_end - E_t or E_end); this kernel adds
// the pairs of positions inside a chunk, whose span is (k, t]:
//     sum_{k < t} (E_t - E_k) w_read_{t,m} kappa_{k,m} exp(-(E_t - E_k)/tau_m) G_{t,k} H_{t,k}
// with G = C B^T, H = dy x^T of the chunk and E the in-chunk cumulative log-decay.  The weight
// E_t - E_k is formed per pair: splitting the sum into E_t- and E_k-weighted totals cancels
// badly (the fp64 chunked model measures a condition number ~1e4 for that split).
//
// One CTA per (chunk, head, batch): the chunk's rates and cumulative log-decay (double), then G
// and H as register-tiled products over 32-column slices of C, B and dy, x staged in shared
// memory (float32), then one thread per row t sums its pairs for every mode.
#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace frac {
namespace {

constexpr int kDtThreads = 256;
constexpr int kSlice = 32;     // columns of C, B (or dy, x) staged per step
constexpr int kQ = 128;        // largest chunk

struct DtauSmem {
    size_t E, kap, wr, gh, a, b, total;
    __host__ __device__ DtauSmem(int Q, int K) {
        E = 0;                                          // double [Q]
        kap = E + sizeof(double) * kQ;                  // float [Q][K]
        wr = kap + sizeof(float) * kQ * K;              // float [Q][K]
        gh = wr + sizeof(float) * kQ * K;               // float [Q][Q + 1]: G, then G o H
        a = gh + sizeof(float) * kQ * (kQ + 1);         // float [Q][kSlice + 1]: C or dy slice
        b = a + sizeof(float) * kQ * (kSlice + 1);      // float [Q][kSlice + 1]: B or x slice
        total = b + sizeof(float) * kQ * (kSlice + 1) + sizeof(float) * 32;
        (void)Q;
    }
};

// acc[8][8] += A[rows r0..r0+7][:] . Bt[cols c0..c0+7][:] over the staged slice
__device__ __forceinline__ void tile_mac(const float *A, const float *Bt, int r0, int c0, int w,
                                         float acc[8][8]) {
    for (int j = 0; j < w; ++j) {
        float av[8], bv[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            av[i] = A[(r0 + i) * (kSlice + 1) + j];
            bv[i] = Bt[(c0 + i) * (kSlice + 1) + j];
        }
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
            for (int k = 0; k < 8; ++k) acc[i][k] = fmaf(av[i], bv[k], acc[i][k]);
    }
}

// stage columns [j0, j0 + w) of rows [c0, c0 + n) of a [B, L, rows_per_pos, cols] tensor (row
// index `sel` at each position) into dst[Q][kSlice + 1] as float; rows >= n read as zero
template <typename T>
__device__ __forceinline__ void stage(float *dst, const T *src, int b, int c0, int n, int L, int rows_per_pos,
                                      int sel, int cols, int j0, int w) {
    for (int idx = threadIdx.x; idx < kQ * kSlice; idx += blockDim.x) {
        const int t = idx / kSlice, j = idx % kSlice;
        float v = 0.f;
        if (t < n && j < w) v = to_f(src[((size_t(b) * L + c0 + t) * rows_per_pos + sel) * cols + j0 + j]);
        dst[t * (kSlice + 1) + j] = v;
    }
}

template <typename T>
__global__ void __launch_bounds__(kDtThreads) dtau_pairs(ScanDims d, const T *__restrict__ x,
                                                           const T *__restrict__ dy, const T *__restrict__ Bm,
                                                           const T *__restrict__ Cm, const T *__restrict__ wr,
                                                           const T *__restrict__ ww, const float *__restrict__ dt,
                                                           const float *__restrict__ alpha,
                                                           const float *__restrict__ lam,
                                                           const float *__restrict__ tau, float *__restrict__ dtau) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int K = d.K, Q = d.Q;
    const int c0 = c * Q, n = min(Q, d.L - c0);
    const int g = h / (d.H / d.G);
    const int tid = threadIdx.x;
    const DtauSmem L_(Q, K);
    double *E = reinterpret_cast<double *>(smem_raw + L_.E);
    float *kap = reinterpret_cast<float *>(smem_raw + L_.kap);
    float *wrs = reinterpret_cast<float *>(smem_raw + L_.wr);
    float *GH = reinterpret_cast<float *>(smem_raw + L_.gh);
    float *sa = reinterpret_cast<float *>(smem_raw + L_.a);
    float *sb = reinterpret_cast<float *>(smem_raw + L_.b);
    float *red = reinterpret_cast<float *>(smem_raw + L_.b + sizeof(float) * kQ * (kSlice + 1));

    // rates, cumulative log-decay (double, serial over <= 128 positions), kappa, read weights
    float tmax = 0.f;
    for (int m = 0; m < K; ++m) tmax = fmaxf(tmax, tau[h * K + m]);
    const float log_cap = logf(64.f * tmax);
    if (tid < 32) red[tid] = 0.f;
    if (tid < n) {
        const size_t i = (size_t(b) * d.L + c0 + tid) * d.H + h;
        bool cl;
        const float e = token_rate(dt[i], alpha[i], lam[i], log_cap, &cl);
        E[tid] = double(e);  // prefix-summed below
        for (int m = 0; m < K; ++m) {
            kap[tid * K + m] = -expm1f(-e / tau[h * K + m]) * to_f(ww[i * K + m]);
            wrs[tid * K + m] = to_f(wr[i * K + m]);
        }
    }
    __syncthreads();
    if (tid == 0)
        for (int t = 1; t < n; ++t) E[t] += E[t - 1];

    // G = C B^T and H = dy x^T, 8 x 8 outputs per thread
    const int r0 = 8 * (tid / 16), q0 = 8 * (tid % 16);
    float G[8][8], Hm[8][8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int k = 0; k < 8; ++k) G[i][k] = Hm[i][k] = 0.f;
    for (int j0 = 0; j0 < d.N; j0 += kSlice) {
        const int w = min(kSlice, d.N - j0);
        __syncthreads();
        stage<T>(sa, Cm, b, c0, n, d.L, d.G, g, d.N, j0, w);
        stage<T>(sb, Bm, b, c0, n, d.L, d.G, g, d.N, j0, w);
        __syncthreads();
        tile_mac(sa, sb, r0, q0, w, G);
    }
    for (int j0 = 0; j0 < d.P; j0 += kSlice) {
        const int w = min(kSlice, d.P - j0);
        __syncthreads();
        stage<T>(sa, dy, b, c0, n, d.L, d.H, h, d.P, j0, w);
        stage<T>(sb, x, b, c0, n, d.L, d.H, h, d.P, j0, w);
        __syncthreads();
        tile_mac(sa, sb, r0, q0, w, Hm);
    }
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int k = 0; k < 8; ++k) GH[(r0 + i) * (kQ + 1) + q0 + k] = G[i][k] * Hm[i][k];
    __syncthreads();

    // per row t: sum over k < t of (E_t - E_k) kappa_k exp(-(E_t - E_k)/tau) GH, per mode
    float part[32];
    for (int m = 0; m < 32; ++m) part[m] = 0.f;
    if (tid < n) {
        const int t = tid;
        float itau[32];
        for (int m = 0; m < K; ++m) itau[m] = 1.f / tau[h * K + m];
        float acc[32];
        for (int m = 0; m < K; ++m) acc[m] = 0.f;
        for (int k = 0; k < t; ++k) {
            const float dE = float(E[t] - E[k]);
            const float gh = GH[t * (kQ + 1) + k];
            for (int m = 0; m < K; ++m) acc[m] = fmaf(dE * kap[k * K + m] * expf(-dE * itau[m]), gh, acc[m]);
        }
        for (int m = 0; m < K; ++m) part[m] = acc[m] * wrs[t * K + m];
    }
    for (int m = 0; m < K; ++m) {
        const float v = warp_sum(part[m]);
        if ((tid & 31) == 0 && v != 0.f) atomicAdd(&red[m], v);
    }
    __syncthreads();
    if (tid < K) {
        const float it = 1.f / tau[h * K + tid];
        atomicAdd(dtau + h * K + tid, red[tid] * it * it);
    }
}

}  // namespace

cudaError_t dtau_pairs_launch(const ScanDims &d, int dtype, const ScanPtrs &p, cudaStream_t st) {
    if (!p.dtau || d.nc == 0) return cudaSuccess;
    if (d.Q > kQ || d.K > 32) return cudaErrorInvalidValue;
    const size_t smem = DtauSmem(d.Q, d.K).total;
    dim3 grid(d.nc, d.H, d.B);
    trace_begin("dtau_pairs", st);
    if (dtype == 1) {
        auto k = dtau_pairs<__nv_bfloat16>;
        cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        using bf = __nv_bfloat16;
        k<<<grid, kDtThreads, smem, st>>>(d, (const bf *)p.x, (const bf *)p.dy, (const bf *)p.Bm,
                                          (const bf *)p.Cm, (const bf *)p.wr, (const bf *)p.ww, p.dt,
                                          p.alpha, p.lam, p.tau, p.dtau);
    } else {
        auto k = dtau_pairs<float>;
        cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        k<<<grid, kDtThreads, smem, st>>>(d, (const float *)p.x, (const float *)p.dy, (const float *)p.Bm,
                                          (const float *)p.Cm, (const float *)p.wr, (const float *)p.ww,
                                          p.dt, p.alpha, p.lam, p.tau, p.dtau);
    }
    trace_end(st);
    return cudaGetLastError();
}

}  // namespace frac
