// One decode step of the Frac scan (Algorithm 1 of App. D, one token, recurrent form).
//
// HBM-bound: every call streams the whole float32 mode state once (read + write).
// One warp owns one (b, h, p) row and all K modes of it: lanes cover the N state
// columns in float4 pieces, all K loads of a group of modes are issued before any
// arithmetic (memory-level parallelism), the state is read and written with
// streaming (evict-first) hints, and the readout sum over n is one warp reduction
// per row after the K modes have been folded in registers.
#include "common.cuh"
#include "kernels.h"

namespace frac {

template <typename T> struct Vec4;
template <> struct Vec4<float> {
    static __device__ __forceinline__ float4 load(const float *p) {
        return *reinterpret_cast<const float4 *>(p);
    }
};
template <> struct Vec4<__nv_bfloat16> {
    static __device__ __forceinline__ float4 load(const __nv_bfloat16 *p) {
        const uint2 u = *reinterpret_cast<const uint2 *>(p);
        const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162 *>(&u.x);
        const __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162 *>(&u.y);
        const float2 fa = __bfloat1622float2(a), fb = __bfloat1622float2(b);
        return make_float4(fa.x, fa.y, fb.x, fb.y);
    }
};

constexpr int kDecodeModeGroup = 8;

template <typename T, bool VEC>
__global__ void __launch_bounds__(256, 4) decode_step_kernel(
    DecodeArgs a, const T *__restrict__ x, const T *__restrict__ Bt, const T *__restrict__ Ct,
    const T *__restrict__ wr, const T *__restrict__ ww, T *__restrict__ y) {
    const int64_t row = (int64_t(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    const int64_t rows = int64_t(a.B) * a.H * a.P;
    if (row >= rows) return;  // warp-uniform
    const int p = int(row % a.P);
    const int64_t bh = row / a.P;
    const int h = int(bh % a.H);
    const int b = int(bh / a.H);
    const int g = h / (a.H / a.G);
    const int K = a.K, N = a.N;

    // per-(b,h) mode parameters: lane m < K owns mode m
    const float tl = lane < K ? a.tau[h * K + lane] : 0.f;
    float tmax = tl;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, o));
    bool clamped;
    const float e = token_rate(a.dt[bh], a.alpha[bh], a.lam[bh], logf(64.f * tmax), &clamped);
    float rho_l = 0.f, kap_l = 0.f, wr_l = 0.f;
    if (lane < K) {
        const float z = e / tl;
        rho_l = expf(-z);
        kap_l = -expm1f(-z) * to_f(ww[bh * K + lane]);
        wr_l = to_f(wr[bh * K + lane]);
    }
    const float xp = to_f(x[bh * a.P + p]);
    const T *Bg = Bt + (int64_t(b) * a.G + g) * N;
    const T *Cg = Ct + (int64_t(b) * a.G + g) * N;
    const int64_t PN = int64_t(a.P) * N;
    float *srow = a.state + (bh * K) * PN + int64_t(p) * N;
    float acc = 0.f;

    if (VEC) {
        const int N4 = N >> 2;
        for (int q = lane; q < N4; q += 32) {
            const float4 bv = Vec4<T>::load(Bg + 4 * q);
            const float4 cv = Vec4<T>::load(Cg + 4 * q);
            for (int m0 = 0; m0 < K; m0 += kDecodeModeGroup) {
                float4 s[kDecodeModeGroup];
#pragma unroll
                for (int j = 0; j < kDecodeModeGroup; ++j)
                    if (m0 + j < K)
                        s[j] = __ldcs(reinterpret_cast<const float4 *>(srow + (m0 + j) * PN) + q);
#pragma unroll
                for (int j = 0; j < kDecodeModeGroup; ++j) {
                    if (m0 + j < K) {
                        const float r = __shfl_sync(0xffffffffu, rho_l, m0 + j);
                        const float kx = __shfl_sync(0xffffffffu, kap_l, m0 + j) * xp;
                        const float w = __shfl_sync(0xffffffffu, wr_l, m0 + j);
                        float4 v = s[j];
                        v.x = fmaf(r, v.x, kx * bv.x);
                        v.y = fmaf(r, v.y, kx * bv.y);
                        v.z = fmaf(r, v.z, kx * bv.z);
                        v.w = fmaf(r, v.w, kx * bv.w);
                        acc = fmaf(w, v.x * cv.x + v.y * cv.y + v.z * cv.z + v.w * cv.w, acc);
                        __stcs(reinterpret_cast<float4 *>(srow + (m0 + j) * PN) + q, v);
                    }
                }
            }
        }
    } else {
        for (int m = 0; m < K; ++m) {
            const float r = __shfl_sync(0xffffffffu, rho_l, m);
            const float kx = __shfl_sync(0xffffffffu, kap_l, m) * xp;
            const float w = __shfl_sync(0xffffffffu, wr_l, m);
            float part = 0.f;
            for (int n = lane; n < N; n += 32) {
                float v = srow[m * PN + n];
                v = fmaf(r, v, kx * to_f(Bg[n]));
                part = fmaf(v, to_f(Cg[n]), part);
                srow[m * PN + n] = v;
            }
            acc = fmaf(w, part, acc);
        }
    }
    acc = warp_sum(acc);
    if (lane == 0) y[bh * a.P + p] = from_f<T>(acc + a.D[h] * xp);
}

// N = 1 (the paper's own layer: scalar B, C per position): one thread per (b, h, p), all K mode
// states of the row loaded before any arithmetic (for each mode a warp reads 32 consecutive p: one
// 128-byte line), then S_m <- rho_m S_m + kappa_m x B and y = sum_m w_read,m C S_m + D x with no
// cross-lane reduction.
constexpr int kDecodeN1Modes = 32;  // nmodes <= 32 (checked at the boundary)

template <typename T>
__global__ void __launch_bounds__(256) decode_step_n1_kernel(
    DecodeArgs a, const T *__restrict__ x, const T *__restrict__ Bt, const T *__restrict__ Ct,
    const T *__restrict__ wr, const T *__restrict__ ww, T *__restrict__ y) {
    const int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i >= int64_t(a.B) * a.H * a.P) return;
    const int p = int(i % a.P);
    const int64_t bh = i / a.P;
    const int h = int(bh % a.H), b = int(bh / a.H), g = h / (a.H / a.G);
    const int K = a.K;
    float *srow = a.state + bh * K * a.P + p;  // mode m at srow[m P]
    float sv[kDecodeN1Modes];
#pragma unroll
    for (int m = 0; m < kDecodeN1Modes; ++m)
        if (m < K) sv[m] = __ldcs(srow + int64_t(m) * a.P);
    float tmax = 0.f;
    for (int m = 0; m < K; ++m) tmax = fmaxf(tmax, a.tau[h * K + m]);
    bool clamped;
    const float e = token_rate(a.dt[bh], a.alpha[bh], a.lam[bh], logf(64.f * tmax), &clamped);
    const float xp = to_f(x[bh * a.P + p]);
    const float kb = xp * to_f(Bt[int64_t(b) * a.G + g]), cv = to_f(Ct[int64_t(b) * a.G + g]);
    float acc = 0.f;
#pragma unroll
    for (int m = 0; m < kDecodeN1Modes; ++m) {
        if (m < K) {
            const float z = e / a.tau[h * K + m];
            const float kap = -expm1f(-z) * to_f(ww[bh * K + m]);
            const float v = fmaf(expf(-z), sv[m], kap * kb);
            acc = fmaf(to_f(wr[bh * K + m]), v * cv, acc);
            __stcs(srow + int64_t(m) * a.P, v);
        }
    }
    y[bh * a.P + p] = from_f<T>(acc + a.D[h] * xp);
}

template <typename T>
cudaError_t launch_decode_t(const DecodeArgs &a, const void *x, const void *Bt, const void *Ct,
                            const void *wr, const void *ww, void *y, cudaStream_t st) {
    const int64_t rows = int64_t(a.B) * a.H * a.P;
    const int64_t blocks = (rows * 32 + 255) / 256;
    // vector path: N a multiple of 128 so that every lane runs the same number of iterations
    // (the mode broadcasts use full-warp shuffles), the state 16-byte aligned and B/C aligned
    // to four elements
    const bool vec = a.N % 128 == 0 && (reinterpret_cast<uintptr_t>(a.state) & 15u) == 0 &&
                     (reinterpret_cast<uintptr_t>(Bt) % (4 * sizeof(T))) == 0 &&
                     (reinterpret_cast<uintptr_t>(Ct) % (4 * sizeof(T))) == 0;
    trace_begin("decode_step", st);
    if (a.N == 1) {
        const int64_t nthreads = rows;
        decode_step_n1_kernel<T><<<dim3(unsigned((nthreads + 255) / 256)), 256, 0, st>>>(
            a, (const T *)x, (const T *)Bt, (const T *)Ct, (const T *)wr, (const T *)ww, (T *)y);
    } else if (vec)
        decode_step_kernel<T, true><<<dim3(unsigned(blocks)), 256, 0, st>>>(
            a, (const T *)x, (const T *)Bt, (const T *)Ct, (const T *)wr, (const T *)ww, (T *)y);
    else
        decode_step_kernel<T, false><<<dim3(unsigned(blocks)), 256, 0, st>>>(
            a, (const T *)x, (const T *)Bt, (const T *)Ct, (const T *)wr, (const T *)ww, (T *)y);
    trace_end(st);
    return cudaGetLastError();
}

cudaError_t launch_decode(const DecodeArgs &a, int dtype, const void *x, const void *Bt,
                          const void *Ct, const void *wr, const void *ww, void *y,
                          cudaStream_t st) {
    if (dtype == 0) return launch_decode_t<float>(a, x, Bt, Ct, wr, ww, y, st);
    return launch_decode_t<__nv_bfloat16>(a, x, Bt, Ct, wr, ww, y, st);
}

}  // namespace frac
