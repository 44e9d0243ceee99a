// Device helpers shared by the Frac kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace frac {

// ------------------------------------------------------------------ element I/O
template <typename T> __device__ __forceinline__ float to_f(T v);
template <> __device__ __forceinline__ float to_f<float>(float v) { return v; }
template <> __device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 v) {
    return __bfloat162float(v);
}
template <typename T> __device__ __forceinline__ T from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float v) {
    return __float2bfloat16_rn(v);
}

// ------------------------------------------------------------------ mode parameters
// e = Delta * lambda^(1/alpha) evaluated as exp(ln Delta + ln lambda / alpha) so that
// lambda^(1/alpha) never overflows; clamped to `cap` (64 * max_m tau_m).  Returns whether
// the clamp was active (then the gradient of e is zero).
__device__ __forceinline__ float token_rate(float dt, float alpha, float lam, float log_cap,
                                            bool *clamped) {
    const float le = logf(dt) + logf(lam) / alpha;
    if (!(le < log_cap)) {  // also catches NaN from invalid controls
        *clamped = true;
        return expf(log_cap);
    }
    *clamped = false;
    return expf(le);
}

// ------------------------------------------------------------------ warp reductions
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Inclusive prefix sum over the 32 lanes of a warp, in double.
__device__ __forceinline__ double warp_inclusive_scan_d(double v) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const double u = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += u;
    }
    return v;
}

}  // namespace frac
