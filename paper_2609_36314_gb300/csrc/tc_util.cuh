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
// (x.lo * s.lo, x.hi * s.hi) in one packed bf16 multiply (round to nearest); x as raw bits
__device__ __forceinline__ uint32_t bf16x2_mul(uint32_t x, __nv_bfloat162 s) {
    __nv_bfloat162 v = *reinterpret_cast<const __nv_bfloat162 *>(&x);
    v = __hmul2(v, s);
    return *reinterpret_cast<const uint32_t *>(&v);
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

// NL x NL transpose (NL = 4 or 8) of 16-byte pieces within each group of NL lanes: on return lane
// NL a + i holds in e[q] the piece that lane NL a + q held in e[i].  Butterfly: at stage k every
// piece whose index differs from the lane in bit k trades places with piece q ^ k of lane ^ k.
__device__ __forceinline__ void shfl_xor_u4(uint4 &v, int o) {
    v.x = __shfl_xor_sync(0xffffffffu, v.x, o);
    v.y = __shfl_xor_sync(0xffffffffu, v.y, o);
    v.z = __shfl_xor_sync(0xffffffffu, v.z, o);
    v.w = __shfl_xor_sync(0xffffffffu, v.w, o);
}
template <int NL>
__device__ __forceinline__ void lane_transpose(uint4 (&e)[NL], int lane) {
#pragma unroll
    for (int k = 1; k < NL; k <<= 1) {
        const bool b = lane & k;
#pragma unroll
        for (int q0 = 0; q0 < NL; ++q0) {
            if (q0 & k) continue;
            uint4 s = b ? e[q0] : e[q0 | k];
            shfl_xor_u4(s, k);
            if (b)
                e[q0] = s;
            else
                e[q0 | k] = s;
        }
    }
}

__device__ __forceinline__ uint4 f4_bits(float a, float b, float c, float d) {
    return make_uint4(__float_as_uint(a), __float_as_uint(b), __float_as_uint(c), __float_as_uint(d));
}

// Every lane holds NL 16-byte pieces of its own row (lane l: row l of its NL-lane group, the
// rows `stride` bytes apart from row0 = the group's first row).  After lane_transpose each
// instruction writes 32 / NL whole row segments of 16 NL contiguous bytes instead of 32
// scattered pieces; rows >= nvalid of the group are skipped.  ADD: float4 atomic add (the
// pieces are float4), else a plain 16-byte store.  Every lane of the warp must call it.
template <int NL, bool ADD>
__device__ __forceinline__ void put_rows(uint4 (&e)[NL], unsigned char *row0, size_t stride, int nvalid) {
    const int lane = threadIdx.x & 31, i = lane & (NL - 1);
    lane_transpose<NL>(e, lane);
#pragma unroll
    for (int q = 0; q < NL; ++q) {
        if (q < nvalid) {
            unsigned char *p = row0 + size_t(q) * stride + 16 * i;
            if (ADD)
                atomicAdd(reinterpret_cast<float4 *>(p), make_float4(__uint_as_float(e[q].x), __uint_as_float(e[q].y),
                                                                     __uint_as_float(e[q].z), __uint_as_float(e[q].w)));
            else
                *reinterpret_cast<uint4 *>(p) = e[q];
        }
    }
}

// The converse of put_rows: lane l of each NL-lane group receives in e[0 .. NL) the NL 16-byte
// pieces of row l of the group (rows `stride` bytes apart from row0), loaded so that each
// instruction reads 32 / NL whole row segments; rows >= nvalid read as zero.  Every lane of the
// warp must call it.  load_rows issues the loads alone (lane_transpose<NL> completes them
// later), so that their latency can overlap other work.
template <int NL>
__device__ __forceinline__ void load_rows(uint4 (&e)[NL], const unsigned char *row0, size_t stride, int nvalid) {
    const int i = threadIdx.x & (NL - 1);
#pragma unroll
    for (int q = 0; q < NL; ++q)
        e[q] = q < nvalid ? *reinterpret_cast<const uint4 *>(row0 + size_t(q) * stride + 16 * i)
                          : make_uint4(0, 0, 0, 0);
}
template <int NL>
__device__ __forceinline__ void get_rows(uint4 (&e)[NL], const unsigned char *row0, size_t stride, int nvalid) {
    load_rows<NL>(e, row0, stride, nvalid);
    lane_transpose<NL>(e, threadIdx.x & 31);
}

// Asynchronous global -> shared copy (cp.async, no register round trip) of 4, 8 or 16 bytes,
// both addresses aligned to the size; completed by cp_async_wait_all.
__device__ __forceinline__ void cp_async_bytes(void *dst, const void *src, int bytes) {
    const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst));
    if (bytes == 16)
        asm volatile("cp.async.ca.shared.global [%0], [%1], 16;" ::"r"(d), "l"(src) : "memory");
    else if (bytes == 8)
        asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(d), "l"(src) : "memory");
    else
        asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(d), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }

// Hint: bring the 128-byte line holding p into L2 (no register result, nothing waits on it).
__device__ __forceinline__ void prefetch_l2(const void *p) {
    asm volatile("prefetch.global.L2 [%0];" ::"l"(reinterpret_cast<uint64_t>(p)));
}

// 2^x with the hardware approximation (relative error ~2^-22); exp(-d / tau) is evaluated as
// 2^(-d * l2t) with l2t = log2(e) / tau precomputed.
__device__ __forceinline__ float ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
constexpr float kLog2e = 1.4426950408889634f;

// A cumulative log-decay kept as an unevaluated float pair hi + lo: the difference of two such
// values is accurate to float precision of the difference itself.
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

// Barrier over the first 256 threads of the block only (named barrier 1), for kernels whose
// extra warps take no part in the per-position work.
__device__ __forceinline__ void sync_first256() { asm volatile("bar.sync 1, 256;" ::: "memory"); }

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

}  // namespace frac
