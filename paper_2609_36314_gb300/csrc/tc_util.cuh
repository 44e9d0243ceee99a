// Small device helpers shared by the tensor-core kernels.
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

#include "common.cuh"
#include "kernels.h"

namespace frac {

constexpr int TQ = 128;          // chunk length on the tensor path
constexpr int TPS = 32;          // P-slice of the state pass / output kernels
constexpr int KMAX = 8;          // modes handled by the tensor path (4 or 8)
constexpr int kTimeoutCode = 4;  // FRAC_ERR_TIMEOUT

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<const uint32_t *>(&v);
}

// The two bf16 halves of a 32-bit word as floats (low half first); exact.
__device__ __forceinline__ float2 bf16x2_to_float2(uint32_t v) {
    return make_float2(__uint_as_float(v << 16), __uint_as_float(v & 0xffff0000u));
}

__device__ __forceinline__ size_t blh(const ScanDims &d, int b, int t, int h) {
    return (size_t(b) * d.L + t) * d.H + h;
}

// The K (4 or 8) bf16 mode weights of one position as floats (16- or 8-byte load); modes
// beyond K are zero.
__device__ __forceinline__ void load_weights(const __nv_bfloat16 *src, int K, float *w) {
    if (K == 8) {
        const uint4 v = *reinterpret_cast<const uint4 *>(src);
        const uint32_t r[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float2 f = bf16x2_to_float2(r[q]);
            w[2 * q] = f.x;
            w[2 * q + 1] = f.y;
        }
    } else {  // K == 4
        const uint2 v = *reinterpret_cast<const uint2 *>(src);
        const uint32_t r[2] = {v.x, v.y};
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            const float2 f = bf16x2_to_float2(r[q]);
            w[2 * q] = f.x;
            w[2 * q + 1] = f.y;
        }
#pragma unroll
        for (int m = 4; m < KMAX; ++m) w[m] = 0.f;
    }
}

// Inclusive prefix sum (double) of one value per thread over a 128-thread block.
__device__ __forceinline__ double block_scan128(double v, double *wsum) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    v = warp_inclusive_scan_d(v);
    if (lane == 31) wsum[w] = v;
    __syncthreads();
    double off = 0.0;
    for (int i = 0; i < w; ++i) off += wsum[i];
    __syncthreads();
    return v + off;
}

// 2^x with the hardware approximation (relative error ~2^-22); exp(-d / tau) is evaluated as
// 2^(-d * l2t) with l2t = log2(e) / tau precomputed.
__device__ __forceinline__ float ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
constexpr float kLog2e = 1.4426950408889634f;

// A cumulative log-decay kept as an unevaluated float pair hi + lo (hi = E rounded to float):
// the difference of two such values is accurate to float precision of the difference itself,
// without a double-precision subtraction per pair.
__device__ __forceinline__ float2 split_f2(double E) {
    const float hi = float(E);
    return make_float2(hi, float(E - double(hi)));
}
__device__ __forceinline__ float diff_f2(float2 a, float2 b) { return (a.x - b.x) + (a.y - b.y); }

// Float-pair (hi + lo) arithmetic for the cumulative log-decay: Knuth's TwoSum keeps the
// rounding error of every addition, so a prefix sum of 128 values carries ~48 significant bits
// (the difference of two prefixes stays accurate to float precision of the difference).
__device__ __forceinline__ float2 f2_add(float2 a, float2 b) {
    const float s = a.x + b.x;
    const float bb = s - a.x;
    const float err = (a.x - (s - bb)) + (b.x - bb);
    const float lo = err + a.y + b.y;
    const float hi = s + lo;
    return make_float2(hi, lo - (hi - s));
}

// Inclusive prefix sum of one value per thread within groups of four warps (threads
// 128 g .. 128 g + 127 scan independently), as a float pair; wsum holds one pair per warp.
__device__ __forceinline__ float2 group_scan128_f2(float v, float2 *wsum) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    float2 p = make_float2(v, 0.f);
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float2 u = make_float2(__shfl_up_sync(0xffffffffu, p.x, o), __shfl_up_sync(0xffffffffu, p.y, o));
        if (lane >= o) p = f2_add(p, u);
    }
    if (lane == 31) wsum[w] = p;
    __syncthreads();
    float2 off = make_float2(0.f, 0.f);
    const int g0 = w & ~3;
    for (int i = g0; i < w; ++i) off = f2_add(off, wsum[i]);
    __syncthreads();
    return f2_add(p, off);
}

// Inclusive prefix sum (double) of one value per thread within groups of four warps (threads
// 128 g .. 128 g + 127 scan independently); wsum holds one slot per warp.
__device__ __forceinline__ double group_scan128(double v, double *wsum) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    v = warp_inclusive_scan_d(v);
    if (lane == 31) wsum[w] = v;
    __syncthreads();
    double off = 0.0;
    const int g0 = w & ~3;
    for (int i = g0; i < w; ++i) off += wsum[i];
    __syncthreads();
    return v + off;
}

}  // namespace frac
