// The FracMixer operations around the scan (Sec. 3.3), HBM-bound:
//
//   depthwise causal conv1d   u[b,t,c] = act(bias_c + sum_j w[c,j] x[b, t-(W-1)+j, c])
//        (the content branch; width d_conv, 4 in App. E.2 / E.4; act = identity or SiLU; the
//        W-1 inputs before the sequence come from a carried state, zeros by default), its
//        backward, and one decode step that shifts the carried state;
//   gated RMS normalisation   out = v / sqrt(mean_group(v^2) + eps) * weight,  v = y * silu(z)
//        (before the output projection), and its backward.
//
// conv1d, bf16 with channel counts a multiple of 8: a block stages a tile of 64 positions (plus
// the filter's halo) x 256 channels in shared memory with cp.async, every piece in flight at once,
// and convolves from there (kernels *_tile_kernel below).  Other shapes: a thread owns four
// adjacent channels (a multiple of 4; else two, else one) and a run of kRun consecutive positions
// read from global memory.  The filter window of the last W-1 inputs stays in registers.  The
// backward streams g = du * act'(pre) through a register ring of the last W values (dx_t needs g
// at t .. t+W-1), and reduces dw / dbias in shared memory before one atomic per channel, tap and
// block.
// RMSNorm (dim <= 8192 forward, <= 4096 backward): a CTA per row holds the row in registers (or,
// bf16 backward, in a ring of shared-memory row buffers filled by cp.async), 8-element vectors
// per thread, so each row is read from HBM once; per-group sums by shared-memory atomics.  The
// backward is persistent over rows, loads the next rows while it processes the current one, and
// keeps each thread's dweight partials in registers until one global atomic per feature and CTA.
// Wider rows take streaming kernels that re-read the row.
#include <algorithm>
#include <cstdio>

#include "../../include/frac.h"
#include "common.cuh"
#include "kernels.h"

namespace frac {
namespace {

constexpr int kRun = 32;      // positions per thread (conv1d)
constexpr int kRows = 8;      // runs per block (threadIdx.y)
constexpr int kMaxW = 8;      // largest conv width

// logistic sigmoid 1 / (1 + 2^(-a log2 e)) from the approximate hardware exp2 and reciprocal
// (relative error ~1e-6 for |a| <= 20, well inside the float32 tolerance of the glue); for
// a < -88 the exponential is +inf and its reciprocal 0, for large a the exponential is 0
__device__ __forceinline__ float sigm(float a) {
    float e, r;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(e) : "f"(-1.4426950408889634f * a));
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(1.f + e));
    return r;
}
__device__ __forceinline__ float silu_f(float a) { return a * sigm(a); }
__device__ __forceinline__ float silu_grad_f(float a) {
    const float s = sigm(a);
    return s * (1.f + a * (1.f - s));
}

// two adjacent channels (c, c + 1) of one position; VEC2: one 2-element access (C even, aligned)
template <typename T, bool VEC2>
__device__ __forceinline__ float2 ld2(const T *p, bool has1) {
    if constexpr (VEC2) {
        if constexpr (sizeof(T) == 2) {
            const __nv_bfloat162 v = *reinterpret_cast<const __nv_bfloat162 *>(p);
            return __bfloat1622float2(v);
        } else {
            return *reinterpret_cast<const float2 *>(p);
        }
    } else {
        return make_float2(to_f(p[0]), has1 ? to_f(p[1]) : 0.f);
    }
}
template <typename T, bool VEC2>
__device__ __forceinline__ void st2(T *p, float2 v, bool has1) {
    if constexpr (VEC2) {
        if constexpr (sizeof(T) == 2)
            *reinterpret_cast<__nv_bfloat162 *>(p) = __floats2bfloat162_rn(v.x, v.y);
        else
            *reinterpret_cast<float2 *>(p) = v;
    } else {
        p[0] = from_f<T>(v.x);
        if (has1) p[1] = from_f<T>(v.y);
    }
}

struct ConvArgs {
    int B, L, C, W;
    bool silu;
    const void *x, *state_in, *du;
    const float *w, *bias;
    void *u, *state_out, *dx, *dstate;
    float *dw, *dbias;
};

// input at position t (t < 0 reads the carried state: index W-1+t, oldest first) for channel c
template <typename T>
__device__ __forceinline__ float x_at(const ConvArgs &a, int b, int t, int c) {
    if (t >= 0) return to_f(static_cast<const T *>(a.x)[(size_t(b) * a.L + t) * a.C + c]);
    if (!a.state_in) return 0.f;
    return to_f(static_cast<const T *>(a.state_in)[(size_t(b) * a.C + c) * (a.W - 1) + (a.W - 1 + t)]);
}

template <typename T, int W, bool VEC2>
__global__ void __launch_bounds__(32 * kRows) conv1d_fwd_kernel(ConvArgs a) {
    const int c = 2 * (blockIdx.x * 32 + threadIdx.x);
    const int t0 = (blockIdx.y * kRows + threadIdx.y) * kRun;
    const int b = blockIdx.z;
    if (c >= a.C || t0 >= a.L) return;
    const bool has1 = c + 1 < a.C;
    float w0[W], w1[W];
#pragma unroll
    for (int j = 0; j < W; ++j) {
        w0[j] = a.w[c * W + j];
        w1[j] = has1 ? a.w[(c + 1) * W + j] : 0.f;
    }
    const float b0 = a.bias ? a.bias[c] : 0.f, b1 = (a.bias && has1) ? a.bias[c + 1] : 0.f;
    float win0[W], win1[W];  // win[j] = input at t - (W-1) + j
#pragma unroll
    for (int j = 0; j < W - 1; ++j) {
        const int t = t0 - (W - 1) + j;
        if (t >= 0) {
            const float2 v = ld2<T, VEC2>(static_cast<const T *>(a.x) + (size_t(b) * a.L + t) * a.C + c, has1);
            win0[j] = v.x;
            win1[j] = v.y;
        } else {
            win0[j] = x_at<T>(a, b, t, c);
            win1[j] = has1 ? x_at<T>(a, b, t, c + 1) : 0.f;
        }
    }
    const int t1 = min(t0 + kRun, a.L);
    constexpr int kB = 8;  // positions whose inputs are loaded together (all in flight at once)
    float2 xb[kB];
    for (int t = t0; t < t1; ++t) {
        if ((t - t0) % kB == 0) {
#pragma unroll
            for (int j = 0; j < kB; ++j)
                xb[j] = t + j < t1 ? ld2<T, VEC2>(static_cast<const T *>(a.x) + (size_t(b) * a.L + t + j) * a.C + c, has1)
                                   : make_float2(0.f, 0.f);
        }
        const size_t off = (size_t(b) * a.L + t) * a.C + c;
        const float2 xv = xb[(t - t0) % kB];
        win0[W - 1] = xv.x;
        win1[W - 1] = xv.y;
        float p0 = b0, p1 = b1;
#pragma unroll
        for (int j = 0; j < W; ++j) {
            p0 = fmaf(w0[j], win0[j], p0);
            p1 = fmaf(w1[j], win1[j], p1);
        }
        if (a.silu) {
            p0 = silu_f(p0);
            p1 = silu_f(p1);
        }
        st2<T, VEC2>(static_cast<T *>(a.u) + off, make_float2(p0, p1), has1);
        if (a.state_out && t >= a.L - (W - 1)) {  // the last W-1 inputs become the carried state
            T *so = static_cast<T *>(a.state_out);
            const int k = t - (a.L - (W - 1));
            so[(size_t(b) * a.C + c) * (W - 1) + k] = from_f<T>(xv.x);
            if (has1) so[(size_t(b) * a.C + c + 1) * (W - 1) + k] = from_f<T>(xv.y);
        }
#pragma unroll
        for (int j = 0; j < W - 1; ++j) {
            win0[j] = win0[j + 1];
            win1[j] = win1[j + 1];
        }
    }
    if (a.state_out && t0 == 0 && a.L < W - 1) {  // short sequence: part of the old state stays
        T *so = static_cast<T *>(a.state_out);
        for (int k = 0; k < W - 1 - a.L; ++k) {
            so[(size_t(b) * a.C + c) * (W - 1) + k] = from_f<T>(x_at<T>(a, b, k + a.L - (W - 1), c));
            if (has1)
                so[(size_t(b) * a.C + c + 1) * (W - 1) + k] = from_f<T>(x_at<T>(a, b, k + a.L - (W - 1), c + 1));
        }
    }
}

template <typename T, int W, bool VEC2>
__global__ void __launch_bounds__(32 * kRows) conv1d_bwd_kernel(ConvArgs a) {
    __shared__ float red[kRows][W + 1][64];  // per run row: dw taps and dbias of the 64 channels
    const int lane = threadIdx.x, ry = threadIdx.y;
    const int c = 2 * (blockIdx.x * 32 + lane);
    const int t0 = (blockIdx.y * kRows + ry) * kRun;
    const int b = blockIdx.z;
    const bool active = c < a.C && t0 < a.L;
    const bool has1 = c + 1 < a.C;
    float acc0[W + 1], acc1[W + 1];  // dw taps, then dbias
#pragma unroll
    for (int j = 0; j <= W; ++j) acc0[j] = acc1[j] = 0.f;
    if (active) {
        float w0[W], w1[W];
#pragma unroll
        for (int j = 0; j < W; ++j) {
            w0[j] = a.w[c * W + j];
            w1[j] = has1 ? a.w[(c + 1) * W + j] : 0.f;
        }
        const float b0 = a.bias ? a.bias[c] : 0.f, b1 = (a.bias && has1) ? a.bias[c + 1] : 0.f;
        float win0[W], win1[W], g0[W], g1[W];  // inputs t-(W-1) .. t; g at t-(W-1) .. t
#pragma unroll
        for (int j = 0; j < W; ++j) g0[j] = g1[j] = 0.f;
#pragma unroll
        for (int j = 0; j < W - 1; ++j) {
            const int t = t0 - (W - 1) + j;
            win0[j] = x_at<T>(a, b, t, c);
            win1[j] = has1 ? x_at<T>(a, b, t, c + 1) : 0.f;
        }
        const int tr = min(t0 + kRun, a.L);          // this run's positions: [t0, tr)
        const int tg = min(tr + W - 1, a.L);         // g is needed up to tg - 1 for dx of the run
        constexpr int kB = 8;  // positions whose inputs are loaded together
        float2 xb[kB], db[kB];
        for (int t = t0; t < tg; ++t) {
            if ((t - t0) % kB == 0) {
#pragma unroll
                for (int j = 0; j < kB; ++j) {
                    const bool in = t + j < tg;
                    const size_t o = (size_t(b) * a.L + t + j) * a.C + c;
                    xb[j] = in ? ld2<T, VEC2>(static_cast<const T *>(a.x) + o, has1) : make_float2(0.f, 0.f);
                    db[j] = in ? ld2<T, VEC2>(static_cast<const T *>(a.du) + o, has1) : make_float2(0.f, 0.f);
                }
            }
            const float2 xv = xb[(t - t0) % kB];
            const float2 dv = db[(t - t0) % kB];
            win0[W - 1] = xv.x;
            win1[W - 1] = xv.y;
            float p0 = b0, p1 = b1;
#pragma unroll
            for (int j = 0; j < W; ++j) {
                p0 = fmaf(w0[j], win0[j], p0);
                p1 = fmaf(w1[j], win1[j], p1);
            }
            const float gg0 = a.silu ? dv.x * silu_grad_f(p0) : dv.x;
            const float gg1 = a.silu ? dv.y * silu_grad_f(p1) : dv.y;
#pragma unroll
            for (int j = 0; j < W - 1; ++j) {
                g0[j] = g0[j + 1];
                g1[j] = g1[j + 1];
            }
            g0[W - 1] = gg0;
            g1[W - 1] = gg1;
            if (t < tr) {  // this run's own positions: dw and dbias terms
#pragma unroll
                for (int j = 0; j < W; ++j) {
                    acc0[j] = fmaf(gg0, win0[j], acc0[j]);
                    acc1[j] = fmaf(gg1, win1[j], acc1[j]);
                }
                acc0[W] += gg0;
                acc1[W] += gg1;
            }
            // dx at s = t - (W-1) (all of its g are in the ring once t = s + W - 1 or t = L - 1)
            const int s = t - (W - 1);
            if (s >= t0) {
                float d0 = 0.f, d1 = 0.f;
#pragma unroll
                for (int j = 0; j < W; ++j) {  // g at s + (W-1) - j = ring slot W-1-j
                    d0 = fmaf(w0[j], g0[W - 1 - j], d0);
                    d1 = fmaf(w1[j], g1[W - 1 - j], d1);
                }
                st2<T, VEC2>(static_cast<T *>(a.dx) + (size_t(b) * a.L + s) * a.C + c, make_float2(d0, d1), has1);
            }
            if (a.dstate && t0 == 0 && t == min(W - 2, a.L - 1)) {
                // gradient of the carried inputs i = 0 .. W-2 (position i - (W-1)):
                // sum over taps j <= i of w_j g[i - j], g[t] at ring slot W-1-(tcur-t)
                for (int i = 0; i < W - 1; ++i) {
                    float d0 = 0.f, d1 = 0.f;
                    for (int j = 0; j <= i && j < W; ++j) {
                        const int tt = i - j;
                        if (tt <= t) {
                            d0 = fmaf(w0[j], g0[W - 1 - (t - tt)], d0);
                            d1 = fmaf(w1[j], g1[W - 1 - (t - tt)], d1);
                        }
                    }
                    T *ds = static_cast<T *>(a.dstate);
                    ds[(size_t(b) * a.C + c) * (W - 1) + i] = from_f<T>(d0);
                    if (has1) ds[(size_t(b) * a.C + c + 1) * (W - 1) + i] = from_f<T>(d1);
                }
            }
#pragma unroll
            for (int j = 0; j < W - 1; ++j) {
                win0[j] = win0[j + 1];
                win1[j] = win1[j + 1];
            }
        }
        // the run's tail positions s in [max(t0, tg - (W-1)), tr): the g beyond the end are 0
        for (int s = max(t0, tg - (W - 1)); s < tr; ++s) {
            const int sh = (tg - 1) - s;  // g at s + k sits at ring slot W-1-(tg-1-(s+k))
            float d0 = 0.f, d1 = 0.f;
            for (int j = 0; j < W; ++j) {
                const int k = (W - 1) - j;  // tap j reads g at s + k
                if (k <= sh) {
                    d0 = fmaf(w0[j], g0[W - 1 - (sh - k)], d0);
                    d1 = fmaf(w1[j], g1[W - 1 - (sh - k)], d1);
                }
            }
            st2<T, VEC2>(static_cast<T *>(a.dx) + (size_t(b) * a.L + s) * a.C + c, make_float2(d0, d1), has1);
        }
    }
#pragma unroll
    for (int j = 0; j <= W; ++j) {
        red[ry][j][2 * lane] = acc0[j];
        red[ry][j][2 * lane + 1] = acc1[j];
    }
    __syncthreads();
    // one atomic per channel and tap: threads (lane, ry) split the (W + 1) x 64 sums
    for (int q = ry * 32 + lane; q < (W + 1) * 64; q += 32 * kRows) {
        const int j = q / 64, cc = q % 64;
        const int ch = blockIdx.x * 64 + cc;
        if (ch >= a.C) continue;
        float s = 0.f;
#pragma unroll
        for (int r = 0; r < kRows; ++r) s += red[r][j][cc];
        if (j < W)
            atomicAdd(a.dw + ch * W + j, s);
        else if (a.dbias)
            atomicAdd(a.dbias + ch, s);
    }
}

// Four adjacent channels of one position as loaded (bf16: 8 bytes, float32: 16 bytes).
template <typename T> struct Raw4;
template <> struct Raw4<__nv_bfloat16> {
    uint2 u;
    __device__ __forceinline__ void load(const __nv_bfloat16 *p) { u = *reinterpret_cast<const uint2 *>(p); }
    __device__ __forceinline__ void get(float *v) const {
        const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&u);
        const float2 a = __bfloat1622float2(h[0]), b = __bfloat1622float2(h[1]);
        v[0] = a.x; v[1] = a.y; v[2] = b.x; v[3] = b.y;
    }
    __device__ __forceinline__ void zero() { u = make_uint2(0u, 0u); }
};
template <> struct Raw4<float> {
    float4 u;
    __device__ __forceinline__ void load(const float *p) { u = *reinterpret_cast<const float4 *>(p); }
    __device__ __forceinline__ void get(float *v) const { v[0] = u.x; v[1] = u.y; v[2] = u.z; v[3] = u.w; }
    __device__ __forceinline__ void zero() { u = make_float4(0.f, 0.f, 0.f, 0.f); }
};
template <typename T> __device__ __forceinline__ void st4(T *p, const float *v);
template <> __device__ __forceinline__ void st4<__nv_bfloat16>(__nv_bfloat16 *p, const float *v) {
    uint2 u;
    __nv_bfloat162 *h = reinterpret_cast<__nv_bfloat162 *>(&u);
    h[0] = __floats2bfloat162_rn(v[0], v[1]);
    h[1] = __floats2bfloat162_rn(v[2], v[3]);
    *reinterpret_cast<uint2 *>(p) = u;
}
template <> __device__ __forceinline__ void st4<float>(float *p, const float *v) {
    *reinterpret_cast<float4 *>(p) = make_float4(v[0], v[1], v[2], v[3]);
}

// The same convolution with four channels per thread (channels a multiple of 4, 4-element aligned
// rows): a warp covers 128 contiguous channels of one position per access, and the inputs of the
// next kB4 positions are loaded while the current ones are convolved, so every thread keeps two
// batches of loads in flight.
constexpr int kB4 = 8;

template <typename T, int W>
__global__ void __launch_bounds__(32 * kRows) conv1d_fwd4_kernel(ConvArgs a) {
    const int c = 4 * (blockIdx.x * 32 + threadIdx.x);
    const int t0 = (blockIdx.y * kRows + threadIdx.y) * kRun;
    const int b = blockIdx.z;
    if (c >= a.C || t0 >= a.L) return;
    const T *xb = static_cast<const T *>(a.x) + size_t(b) * a.L * a.C + c;
    float w[4][W], bs[4], win[4][W];  // win[k][j] = input at t - (W-1) + j, channel c + k
#pragma unroll
    for (int k = 0; k < 4; ++k) {
#pragma unroll
        for (int j = 0; j < W; ++j) w[k][j] = a.w[(c + k) * W + j];
        bs[k] = a.bias ? a.bias[c + k] : 0.f;
    }
#pragma unroll
    for (int j = 0; j < W - 1; ++j) {
        const int t = t0 - (W - 1) + j;
        if (t >= 0) {
            Raw4<T> r;
            r.load(xb + size_t(t) * a.C);
            float v[4];
            r.get(v);
#pragma unroll
            for (int k = 0; k < 4; ++k) win[k][j] = v[k];
        } else {
#pragma unroll
            for (int k = 0; k < 4; ++k) win[k][j] = x_at<T>(a, b, t, c + k);
        }
    }
    const int t1 = min(t0 + kRun, a.L);
    Raw4<T> cur[kB4], nxt[kB4];
#pragma unroll
    for (int i = 0; i < kB4; ++i) {
        if (t0 + i < t1) cur[i].load(xb + size_t(t0 + i) * a.C);
        else cur[i].zero();
    }
    for (int tb = t0; tb < t1; tb += kB4) {
#pragma unroll
        for (int i = 0; i < kB4; ++i) {  // the next batch, in flight while this one is convolved
            const int t = tb + kB4 + i;
            if (t < t1) nxt[i].load(xb + size_t(t) * a.C);
            else nxt[i].zero();
        }
#pragma unroll
        for (int i = 0; i < kB4; ++i) {
            const int t = tb + i;
            if (t < t1) {
                float xv[4], p[4];
                cur[i].get(xv);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    win[k][W - 1] = xv[k];
                    p[k] = bs[k];
#pragma unroll
                    for (int j = 0; j < W; ++j) p[k] = fmaf(w[k][j], win[k][j], p[k]);
                    if (a.silu) p[k] = silu_f(p[k]);
                }
                st4<T>(static_cast<T *>(a.u) + (size_t(b) * a.L + t) * a.C + c, p);
                if (a.state_out && t >= a.L - (W - 1)) {  // the last W-1 inputs become the carried state
                    T *so = static_cast<T *>(a.state_out);
                    const int ks = t - (a.L - (W - 1));
#pragma unroll
                    for (int k = 0; k < 4; ++k) so[(size_t(b) * a.C + c + k) * (W - 1) + ks] = from_f<T>(xv[k]);
                }
#pragma unroll
                for (int k = 0; k < 4; ++k)
#pragma unroll
                    for (int j = 0; j < W - 1; ++j) win[k][j] = win[k][j + 1];
            }
        }
#pragma unroll
        for (int i = 0; i < kB4; ++i) cur[i] = nxt[i];
    }
    if (a.state_out && t0 == 0 && a.L < W - 1) {  // short sequence: part of the old state stays
        T *so = static_cast<T *>(a.state_out);
        for (int ks = 0; ks < W - 1 - a.L; ++ks)
#pragma unroll
            for (int k = 0; k < 4; ++k)
                so[(size_t(b) * a.C + c + k) * (W - 1) + ks] = from_f<T>(x_at<T>(a, b, ks + a.L - (W - 1), c + k));
    }
}

constexpr int kB4b = 4;  // positions per batch of the backward (two streams in flight)

// r[idx] for a run-time idx by unrolled selects, so that the ring stays in registers
template <int W>
__device__ __forceinline__ float ring_at(const float (&r)[W], int idx) {
    float v = 0.f;
#pragma unroll
    for (int i = 0; i < W; ++i) v = i == idx ? r[i] : v;
    return v;
}

template <typename T, int W>
__global__ void __launch_bounds__(32 * kRows, 2) conv1d_bwd4_kernel(ConvArgs a) {
    __shared__ float red[kRows][W + 1][128];  // per run row: dw taps and dbias of the 128 channels
    const int lane = threadIdx.x, ry = threadIdx.y;
    const int c = 4 * (blockIdx.x * 32 + lane);
    const int t0 = (blockIdx.y * kRows + ry) * kRun;
    const int b = blockIdx.z;
    const bool active = c < a.C && t0 < a.L;
    float acc[4][W + 1];  // dw taps, then dbias
#pragma unroll
    for (int k = 0; k < 4; ++k)
#pragma unroll
        for (int j = 0; j <= W; ++j) acc[k][j] = 0.f;
    if (active) {
        const size_t rowb = size_t(b) * a.L * a.C + c;
        const T *xb = static_cast<const T *>(a.x) + rowb;
        const T *db = static_cast<const T *>(a.du) + rowb;
        T *dxb = static_cast<T *>(a.dx) + rowb;
        float w[4][W], bs[4], win[4][W], g[4][W];  // inputs t-(W-1) .. t; g at t-(W-1) .. t
#pragma unroll
        for (int k = 0; k < 4; ++k) {
#pragma unroll
            for (int j = 0; j < W; ++j) {
                w[k][j] = a.w[(c + k) * W + j];
                g[k][j] = 0.f;
            }
            bs[k] = a.bias ? a.bias[c + k] : 0.f;
        }
#pragma unroll
        for (int j = 0; j < W - 1; ++j)
#pragma unroll
            for (int k = 0; k < 4; ++k) win[k][j] = x_at<T>(a, b, t0 - (W - 1) + j, c + k);
        const int tr = min(t0 + kRun, a.L);   // this run's positions: [t0, tr)
        const int tg = min(tr + W - 1, a.L);  // g is needed up to tg - 1 for dx of the run
        Raw4<T> cx[kB4b], cd[kB4b], nx[kB4b], nd[kB4b];
#pragma unroll
        for (int i = 0; i < kB4b; ++i) {
            if (t0 + i < tg) {
                cx[i].load(xb + size_t(t0 + i) * a.C);
                cd[i].load(db + size_t(t0 + i) * a.C);
            } else {
                cx[i].zero();
                cd[i].zero();
            }
        }
        for (int tb = t0; tb < tg; tb += kB4b) {
#pragma unroll
            for (int i = 0; i < kB4b; ++i) {
                const int t = tb + kB4b + i;
                if (t < tg) {
                    nx[i].load(xb + size_t(t) * a.C);
                    nd[i].load(db + size_t(t) * a.C);
                } else {
                    nx[i].zero();
                    nd[i].zero();
                }
            }
#pragma unroll
            for (int i = 0; i < kB4b; ++i) {
                const int t = tb + i;
                if (t < tg) {
                    float xv[4], dv[4];
                    cx[i].get(xv);
                    cd[i].get(dv);
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        win[k][W - 1] = xv[k];
                        float p = bs[k];
#pragma unroll
                        for (int j = 0; j < W; ++j) p = fmaf(w[k][j], win[k][j], p);
                        const float gg = a.silu ? dv[k] * silu_grad_f(p) : dv[k];
#pragma unroll
                        for (int j = 0; j < W - 1; ++j) g[k][j] = g[k][j + 1];
                        g[k][W - 1] = gg;
                        if (t < tr) {  // this run's own positions: dw and dbias terms
#pragma unroll
                            for (int j = 0; j < W; ++j) acc[k][j] = fmaf(gg, win[k][j], acc[k][j]);
                            acc[k][W] += gg;
                        }
                    }
                    // dx at s = t - (W-1) (all of its g are in the ring once t = s + W - 1)
                    const int s = t - (W - 1);
                    if (s >= t0) {
                        float dx[4];
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            dx[k] = 0.f;
#pragma unroll
                            for (int j = 0; j < W; ++j) dx[k] = fmaf(w[k][j], g[k][W - 1 - j], dx[k]);
                        }
                        st4<T>(dxb + size_t(s) * a.C, dx);
                    }
                    if (a.dstate && t0 == 0 && t == min(W - 2, a.L - 1)) {
                        // gradient of the carried inputs i = 0 .. W-2 (position i - (W-1)):
                        // sum over taps j <= i of w_j g[i - j], g[tt] at ring slot W-1-(t-tt)
                        T *ds = static_cast<T *>(a.dstate);
                        for (int ii = 0; ii < W - 1; ++ii) {
#pragma unroll
                            for (int k = 0; k < 4; ++k) {
                                float d = 0.f;
#pragma unroll
                                for (int j = 0; j < W; ++j) {
                                    const int tt = ii - j;
                                    if (j <= ii && tt <= t) d = fmaf(w[k][j], ring_at<W>(g[k], W - 1 - (t - tt)), d);
                                }
                                ds[(size_t(b) * a.C + c + k) * (W - 1) + ii] = from_f<T>(d);
                            }
                        }
                    }
#pragma unroll
                    for (int k = 0; k < 4; ++k)
#pragma unroll
                        for (int j = 0; j < W - 1; ++j) win[k][j] = win[k][j + 1];
                }
            }
#pragma unroll
            for (int i = 0; i < kB4b; ++i) {
                cx[i] = nx[i];
                cd[i] = nd[i];
            }
        }
        // the run's tail positions s in [max(t0, tg - (W-1)), tr): the g beyond the end are 0
        for (int s = max(t0, tg - (W - 1)); s < tr; ++s) {
            const int sh = (tg - 1) - s;  // g at s + kk sits at ring slot W-1-(tg-1-(s+kk))
            float dx[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                dx[k] = 0.f;
#pragma unroll
                for (int j = 0; j < W; ++j) {
                    const int kk = (W - 1) - j;  // tap j reads g at s + kk
                    if (kk <= sh) dx[k] = fmaf(w[k][j], ring_at<W>(g[k], W - 1 - (sh - kk)), dx[k]);
                }
            }
            st4<T>(dxb + size_t(s) * a.C, dx);
        }
    }
#pragma unroll
    for (int k = 0; k < 4; ++k)
#pragma unroll
        for (int j = 0; j <= W; ++j) red[ry][j][4 * lane + k] = acc[k][j];
    __syncthreads();
    // one atomic per channel and tap: threads (lane, ry) split the (W + 1) x 128 sums
    for (int q = ry * 32 + lane; q < (W + 1) * 128; q += 32 * kRows) {
        const int j = q / 128, cc = q % 128;
        const int ch = blockIdx.x * 128 + cc;
        if (ch >= a.C) continue;
        float sum = 0.f;
#pragma unroll
        for (int r = 0; r < kRows; ++r) sum += red[r][j][cc];
        if (j < W)
            atomicAdd(a.dw + ch * W + j, sum);
        else if (a.dbias)
            atomicAdd(a.dbias + ch, sum);
    }
}

// Tile path of the forward (bf16, channels a multiple of 8, 16-byte aligned rows): a block stages
// positions [t0 - kHalo, t0 + kTileT) x channels [c0, c0 + kTileC) in shared memory by cp.async
// (every 16-byte piece of the tile in flight at once; zeros outside the sequence, the carried
// state patched in before position 0), then convolves from shared memory: thread i owns the
// channel pair c0 + 2 (i mod 128) and the 32 positions of half i / 128, a warp stores 128
// contiguous bytes per position.  36 KB of shared memory per block, six blocks per SM.
constexpr int kTileT = 64, kTileC = 256, kHalo = 8;  // kHalo >= W - 1 for every width

__device__ __forceinline__ void cp_async16_zfill(void *dst, const void *src, bool in) {
    const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(src), "r"(in ? 16 : 0) : "memory");
}

template <int W>
__global__ void __launch_bounds__(256) conv1d_fwd_tile_kernel(ConvArgs a) {
    using T = __nv_bfloat16;
    __shared__ __align__(16) T tile[kTileT + kHalo][kTileC];
    const int c0 = blockIdx.x * kTileC, t0 = blockIdx.y * kTileT, b = blockIdx.z;
    const T *x = static_cast<const T *>(a.x);
    for (int i = threadIdx.x; i < (kTileT + kHalo) * (kTileC / 8); i += blockDim.x) {
        const int r = i / (kTileC / 8), q = i % (kTileC / 8);
        const int t = t0 - kHalo + r, c = c0 + 8 * q;
        const bool in = t >= 0 && t < a.L && c < a.C;
        cp_async16_zfill(&tile[r][8 * q], in ? x + (size_t(b) * a.L + t) * a.C + c : x, in);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
    asm volatile("cp.async.wait_all;" ::: "memory");
    if (t0 == 0 && a.state_in && W > 1) {  // positions -(W-1) .. -1 from the carried state
        __syncthreads();
        const T *si = static_cast<const T *>(a.state_in);
        for (int i = threadIdx.x; i < (W - 1) * kTileC; i += blockDim.x) {
            const int j = i / kTileC, cc = i % kTileC, c = c0 + cc;
            if (c < a.C) tile[kHalo - (W - 1) + j][cc] = si[(size_t(b) * a.C + c) * (W - 1) + j];
        }
    }
    __syncthreads();
    const int cp = threadIdx.x & 127, half = threadIdx.x >> 7;
    const int c = c0 + 2 * cp;
    if (c >= a.C) return;  // C is a multiple of 8: the pair is whole
    float w0[W], w1[W], win0[W], win1[W];
#pragma unroll
    for (int j = 0; j < W; ++j) {
        w0[j] = a.w[c * W + j];
        w1[j] = a.w[(c + 1) * W + j];
    }
    const float b0 = a.bias ? a.bias[c] : 0.f, b1 = a.bias ? a.bias[c + 1] : 0.f;
    const int r0 = kHalo + 32 * half;  // tile row of this thread's first position
#pragma unroll
    for (int j = 0; j < W - 1; ++j) {
        const float2 v = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&tile[r0 - (W - 1) + j][2 * cp]));
        win0[j] = v.x;
        win1[j] = v.y;
    }
    T *u = static_cast<T *>(a.u);
#pragma unroll 4
    for (int i = 0; i < 32; ++i) {
        const int t = t0 + 32 * half + i;
        if (t >= a.L) break;
        const float2 v = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&tile[r0 + i][2 * cp]));
        win0[W - 1] = v.x;
        win1[W - 1] = v.y;
        float p0 = b0, p1 = b1;
#pragma unroll
        for (int j = 0; j < W; ++j) {
            p0 = fmaf(w0[j], win0[j], p0);
            p1 = fmaf(w1[j], win1[j], p1);
        }
        if (a.silu) {
            p0 = silu_f(p0);
            p1 = silu_f(p1);
        }
        *reinterpret_cast<__nv_bfloat162 *>(u + (size_t(b) * a.L + t) * a.C + c) = __floats2bfloat162_rn(p0, p1);
        if (a.state_out && t >= a.L - (W - 1)) {  // the last W-1 inputs become the carried state
            T *so = static_cast<T *>(a.state_out);
            const int ks = t - (a.L - (W - 1));
            so[(size_t(b) * a.C + c) * (W - 1) + ks] = __float2bfloat16_rn(v.x);
            so[(size_t(b) * a.C + c + 1) * (W - 1) + ks] = __float2bfloat16_rn(v.y);
        }
#pragma unroll
        for (int j = 0; j < W - 1; ++j) {
            win0[j] = win0[j + 1];
            win1[j] = win1[j + 1];
        }
    }
    if (a.state_out && t0 == 0 && half == 0 && a.L < W - 1) {  // short sequence: part of the old state stays
        T *so = static_cast<T *>(a.state_out);
        for (int ks = 0; ks < W - 1 - a.L; ++ks) {
            const int row = kHalo - (W - 1) + ks + a.L;  // position ks + L - (W-1) < 0: a state row
            so[(size_t(b) * a.C + c) * (W - 1) + ks] = tile[row][2 * cp];
            so[(size_t(b) * a.C + c + 1) * (W - 1) + ks] = tile[row][2 * cp + 1];
        }
    }
}

// Tile path of the backward (same conditions): a block stages x at positions [t0 - kHalo,
// t0 + kTileT + kHalo) and du at [t0, t0 + kTileT + kHalo) (76 KB, two blocks per SM); thread i
// owns the channel pair c0 + 2 (i mod 128) and the 32 positions s of half i / 128: it walks
// tt = s .. s + 31 + W - 1, forming g = du act'(pre) into a register ring of the last W values
// (dx_s needs g at s .. s + W - 1), accumulating dw and dbias over its own positions, and writing
// dx_s once the ring holds g at s .. s + W - 1.  dw, dbias: both halves' partials summed in shared
// memory, one atomic per (channel, tap) and block.
constexpr int kXRows = kTileT + 2 * kHalo, kDRows = kTileT + kHalo;

template <int W>
__global__ void __launch_bounds__(256, 2) conv1d_bwd_tile_kernel(ConvArgs a) {
    using T = __nv_bfloat16;
    extern __shared__ __align__(16) unsigned char tile_raw[];
    T (*xt)[kTileC] = reinterpret_cast<T (*)[kTileC]>(tile_raw);                          // [kXRows]
    T (*dt)[kTileC] = reinterpret_cast<T (*)[kTileC]>(tile_raw + kXRows * kTileC * 2);  // [kDRows]
    const int c0 = blockIdx.x * kTileC, t0 = blockIdx.y * kTileT, b = blockIdx.z;
    const T *x = static_cast<const T *>(a.x), *du = static_cast<const T *>(a.du);
    for (int i = threadIdx.x; i < (kXRows + kDRows) * (kTileC / 8); i += blockDim.x) {
        const bool isx = i < kXRows * (kTileC / 8);
        const int ii = isx ? i : i - kXRows * (kTileC / 8);
        const int r = ii / (kTileC / 8), q = ii % (kTileC / 8);
        const int t = isx ? t0 - kHalo + r : t0 + r, c = c0 + 8 * q;
        const bool in = t >= 0 && t < a.L && c < a.C;
        const T *src = isx ? x : du;
        cp_async16_zfill(isx ? &xt[r][8 * q] : &dt[r][8 * q], in ? src + (size_t(b) * a.L + t) * a.C + c : src, in);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
    asm volatile("cp.async.wait_all;" ::: "memory");
    if (t0 == 0 && a.state_in && W > 1) {  // positions -(W-1) .. -1 from the carried state
        __syncthreads();
        const T *si = static_cast<const T *>(a.state_in);
        for (int i = threadIdx.x; i < (W - 1) * kTileC; i += blockDim.x) {
            const int j = i / kTileC, cc = i % kTileC, c = c0 + cc;
            if (c < a.C) xt[kHalo - (W - 1) + j][cc] = si[(size_t(b) * a.C + c) * (W - 1) + j];
        }
    }
    __syncthreads();
    const int cp = threadIdx.x & 127, half = threadIdx.x >> 7;
    const int c = c0 + 2 * cp;
    const bool active = c < a.C;
    float acc0[W + 1], acc1[W + 1];  // dw taps, then dbias
#pragma unroll
    for (int j = 0; j <= W; ++j) acc0[j] = acc1[j] = 0.f;
    if (active) {
        float w0[W], w1[W], win0[W], win1[W], g0[W], g1[W], gf0[kMaxW], gf1[kMaxW];
#pragma unroll
        for (int j = 0; j < W; ++j) {
            w0[j] = a.w[c * W + j];
            w1[j] = a.w[(c + 1) * W + j];
            g0[j] = g1[j] = 0.f;
        }
        const float b0 = a.bias ? a.bias[c] : 0.f, b1 = a.bias ? a.bias[c + 1] : 0.f;
        const int s0 = t0 + 32 * half;  // this thread's first own position
        // x window before s0: positions s0 - (W-1) .. s0 - 1 at rows s0 - t0 + kHalo - (W-1) ..
#pragma unroll
        for (int j = 0; j < W - 1; ++j) {
            const float2 v = __bfloat1622float2(
                *reinterpret_cast<const __nv_bfloat162 *>(&xt[s0 - t0 + kHalo - (W - 1) + j][2 * cp]));
            win0[j] = v.x;
            win1[j] = v.y;
        }
        T *dx = static_cast<T *>(a.dx);
#pragma unroll 4
        for (int i = 0; i < 32 + W - 1; ++i) {
            const int tt = s0 + i;
            const float2 xv = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&xt[tt - t0 + kHalo][2 * cp]));
            const float2 dv = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&dt[tt - t0][2 * cp]));
            win0[W - 1] = xv.x;
            win1[W - 1] = xv.y;
            float p0 = b0, p1 = b1;
#pragma unroll
            for (int j = 0; j < W; ++j) {
                p0 = fmaf(w0[j], win0[j], p0);
                p1 = fmaf(w1[j], win1[j], p1);
            }
            const float gg0 = a.silu ? dv.x * silu_grad_f(p0) : dv.x;  // du is 0 past the end
            const float gg1 = a.silu ? dv.y * silu_grad_f(p1) : dv.y;
#pragma unroll
            for (int j = 0; j < W - 1; ++j) {
                g0[j] = g0[j + 1];
                g1[j] = g1[j + 1];
            }
            g0[W - 1] = gg0;
            g1[W - 1] = gg1;
            if (i < 32 && tt < a.L) {  // own positions: dw and dbias terms
#pragma unroll
                for (int j = 0; j < W; ++j) {
                    acc0[j] = fmaf(gg0, win0[j], acc0[j]);
                    acc1[j] = fmaf(gg1, win1[j], acc1[j]);
                }
                acc0[W] += gg0;
                acc1[W] += gg1;
            }
#pragma unroll
            for (int j = 0; j < W - 1; ++j)  // g at positions 0 .. W-2, for the carried-state gradient
                if (tt == j) {
                    gf0[j] = gg0;
                    gf1[j] = gg1;
                }
            const int s = tt - (W - 1);  // the ring now holds g at s .. s + W - 1
            if (i >= W - 1 && s < a.L) {
                float d0 = 0.f, d1 = 0.f;
#pragma unroll
                for (int j = 0; j < W; ++j) {
                    d0 = fmaf(w0[j], g0[W - 1 - j], d0);
                    d1 = fmaf(w1[j], g1[W - 1 - j], d1);
                }
                *reinterpret_cast<__nv_bfloat162 *>(dx + (size_t(b) * a.L + s) * a.C + c) = __floats2bfloat162_rn(d0, d1);
            }
#pragma unroll
            for (int j = 0; j < W - 1; ++j) {
                win0[j] = win0[j + 1];
                win1[j] = win1[j + 1];
            }
        }
        if (a.dstate && t0 == 0 && half == 0) {
            // gradient of the carried inputs i = 0 .. W-2 (position i - (W-1)): taps j <= i of
            // w_j g[i - j] over the positions that exist
            T *ds = static_cast<T *>(a.dstate);
#pragma unroll
            for (int ii = 0; ii < W - 1; ++ii) {
                float d0 = 0.f, d1 = 0.f;
#pragma unroll
                for (int j = 0; j < W; ++j) {
                    const int tt = ii - j;
                    if (j <= ii && tt < a.L) {
                        d0 = fmaf(w0[j], gf0[tt], d0);
                        d1 = fmaf(w1[j], gf1[tt], d1);
                    }
                }
                ds[(size_t(b) * a.C + c) * (W - 1) + ii] = __float2bfloat16_rn(d0);
                ds[(size_t(b) * a.C + c + 1) * (W - 1) + ii] = __float2bfloat16_rn(d1);
            }
        }
    }
    __syncthreads();  // the tiles are dead: their space sums dw, dbias
    float *red = reinterpret_cast<float *>(tile_raw);  // [2 halves][W + 1][kTileC]
#pragma unroll
    for (int j = 0; j <= W; ++j) {
        red[(half * (W + 1) + j) * kTileC + 2 * cp] = acc0[j];
        red[(half * (W + 1) + j) * kTileC + 2 * cp + 1] = acc1[j];
    }
    __syncthreads();
    for (int q = threadIdx.x; q < (W + 1) * kTileC; q += blockDim.x) {
        const int j = q / kTileC, cc = q % kTileC, ch = c0 + cc;
        if (ch >= a.C) continue;
        const float sum = red[j * kTileC + cc] + red[((W + 1) + j) * kTileC + cc];
        if (j < W)
            atomicAdd(a.dw + ch * W + j, sum);
        else if (a.dbias)
            atomicAdd(a.dbias + ch, sum);
    }
}
constexpr size_t kConvBwdTileSmem = size_t(kXRows + kDRows) * kTileC * 2;

// one decode step: window = carried state (W-1 inputs) then x_t; the state shifts by one
template <typename T>
__global__ void __launch_bounds__(256) conv1d_step_kernel(ConvArgs a, const T *__restrict__ xt, T *__restrict__ ut) {
    const int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i >= int64_t(a.B) * a.C) return;
    const int c = int(i % a.C);
    const int W = a.W;
    T *st = W > 1 ? static_cast<T *>(a.state_out) + i * (W - 1) : nullptr;
    float p = a.bias ? a.bias[c] : 0.f;
    float prev[kMaxW];
    for (int j = 0; j < W - 1; ++j) prev[j] = to_f(st[j]);
    const float x = to_f(xt[i]);
    for (int j = 0; j < W - 1; ++j) p = fmaf(a.w[c * W + j], prev[j], p);
    p = fmaf(a.w[c * W + W - 1], x, p);
    ut[i] = from_f<T>(a.silu ? silu_f(p) : p);
    for (int j = 0; j + 1 < W - 1; ++j) st[j] = from_f<T>(prev[j + 1]);
    if (W > 1) st[W - 2] = from_f<T>(x);
}

// ------------------------------------------------------------------ gated RMSNorm
struct NormArgs {
    int64_t R;
    int D, gs;
    float eps;
    const void *y, *z, *dout;
    const float *weight;
    void *out, *dy, *dz;
    float *dweight;
};

// 8 consecutive features of one row
template <typename T>
__device__ __forceinline__ void ld8(const T *p, float *v) {
    if constexpr (sizeof(T) == 2) {
        const uint4 u = *reinterpret_cast<const uint4 *>(p);
        const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&u);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = __bfloat1622float2(h[i]);
            v[2 * i] = f.x;
            v[2 * i + 1] = f.y;
        }
    } else {
        const float4 a = reinterpret_cast<const float4 *>(p)[0], b = reinterpret_cast<const float4 *>(p)[1];
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    }
}
template <typename T>
__device__ __forceinline__ void st8(T *p, const float *v) {
    if constexpr (sizeof(T) == 2) {
        uint4 u;
        __nv_bfloat162 *h = reinterpret_cast<__nv_bfloat162 *>(&u);
#pragma unroll
        for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
        *reinterpret_cast<uint4 *>(p) = u;
    } else {
        reinterpret_cast<float4 *>(p)[0] = make_float4(v[0], v[1], v[2], v[3]);
        reinterpret_cast<float4 *>(p)[1] = make_float4(v[4], v[5], v[6], v[7]);
    }
}

// v = y * silu(z) for 8 features at f of row r
template <typename T>
__device__ __forceinline__ void gated8(const NormArgs &a, int64_t r, int f, float *v, float *zv) {
    ld8<T>(static_cast<const T *>(a.y) + r * a.D + f, v);
    if (a.z) {
        ld8<T>(static_cast<const T *>(a.z) + r * a.D + f, zv);
#pragma unroll
        for (int i = 0; i < 8; ++i) v[i] *= silu_f(zv[i]);
    }
}

// Adds a thread's partial s (of the 8 features at f) to its group's sum.  When groups are whole
// multiples of 256 features, the 32 lanes of a warp (256 consecutive features) share a group:
// one warp sum and one shared atomic per warp instead of 32 atomics on one address.
__device__ __forceinline__ void group_add(float *sums, int f, int gs, bool valid, float s) {
    if (gs % 256 == 0) {
        s = warp_sum(valid ? s : 0.f);
        if ((threadIdx.x & 31) == 0 && valid) atomicAdd(&sums[f / gs], s);
    } else if (valid) {
        atomicAdd(&sums[f / gs], s);
    }
}

// Requires gs % 8 == 0 and D % 8 == 0 (host-checked): every 8-vector lies in one group.  The
// feature loops step by 8 blockDim features with every lane in every step (warp sums need
// the whole warp), `valid` marking the lanes past the end of the row.
template <typename T>
__global__ void __launch_bounds__(256) rmsnorm_fwd_kernel(NormArgs a) {
    extern __shared__ float gsum[];  // [D / gs]
    const int ng = a.D / a.gs;
    for (int64_t r = blockIdx.x; r < a.R; r += gridDim.x) {
        for (int g = threadIdx.x; g < ng; g += blockDim.x) gsum[g] = 0.f;
        __syncthreads();
        for (int f0 = 0; f0 < a.D; f0 += 8 * blockDim.x) {
            const int f = f0 + 8 * threadIdx.x;
            const bool valid = f < a.D;
            float s = 0.f;
            if (valid) {
                float v[8], zv[8];
                gated8<T>(a, r, f, v, zv);
#pragma unroll
                for (int i = 0; i < 8; ++i) s = fmaf(v[i], v[i], s);
            }
            group_add(gsum, f, a.gs, valid, s);
        }
        __syncthreads();
        for (int g = threadIdx.x; g < ng; g += blockDim.x) gsum[g] = rsqrtf(gsum[g] / a.gs + a.eps);
        __syncthreads();
        for (int f = 8 * threadIdx.x; f < a.D; f += 8 * blockDim.x) {
            float v[8], zv[8];
            gated8<T>(a, r, f, v, zv);
            const float inv = gsum[f / a.gs];
#pragma unroll
            for (int i = 0; i < 8; ++i) v[i] = v[i] * inv * a.weight[f + i];
            st8<T>(static_cast<T *>(a.out) + r * a.D + f, v);
        }
        __syncthreads();
    }
}

template <typename T>
__global__ void __launch_bounds__(256) rmsnorm_bwd_kernel(NormArgs a) {
    extern __shared__ float sm[];
    const int ng = a.D / a.gs;
    float *dwp = sm;            // this CTA's dweight partials: feature f + i at i (D / 8) + f / 8,
                                // owned by one thread, consecutive threads in consecutive words
    float *inv = sm + a.D;      // [ng] 1 / rms per group
    float *dot = inv + ng;      // [ng] sum over the group of dn * n
    for (int f = threadIdx.x; f < a.D; f += blockDim.x) dwp[f] = 0.f;
    for (int64_t r = blockIdx.x; r < a.R; r += gridDim.x) {
        for (int g = threadIdx.x; g < ng; g += blockDim.x) inv[g] = dot[g] = 0.f;
        __syncthreads();
        for (int f0 = 0; f0 < a.D; f0 += 8 * blockDim.x) {
            const int f = f0 + 8 * threadIdx.x;
            const bool valid = f < a.D;
            float s = 0.f;
            if (valid) {
                float v[8], zv[8];
                gated8<T>(a, r, f, v, zv);
#pragma unroll
                for (int i = 0; i < 8; ++i) s = fmaf(v[i], v[i], s);
            }
            group_add(inv, f, a.gs, valid, s);
        }
        __syncthreads();
        for (int g = threadIdx.x; g < ng; g += blockDim.x) inv[g] = rsqrtf(inv[g] / a.gs + a.eps);
        __syncthreads();
        const int D8 = a.D / 8;
        for (int f0 = 0; f0 < a.D; f0 += 8 * blockDim.x) {
            const int f = f0 + 8 * threadIdx.x;
            const bool valid = f < a.D;
            float s = 0.f;
            if (valid) {
                float v[8], zv[8], go[8];
                gated8<T>(a, r, f, v, zv);
                ld8<T>(static_cast<const T *>(a.dout) + r * a.D + f, go);
                const float iv = inv[f / a.gs];
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const float n = v[i] * iv;
                    dwp[i * D8 + f / 8] = fmaf(go[i], n, dwp[i * D8 + f / 8]);
                    s = fmaf(go[i] * a.weight[f + i], n, s);
                }
            }
            group_add(dot, f, a.gs, valid, s);
        }
        __syncthreads();
        for (int f = 8 * threadIdx.x; f < a.D; f += 8 * blockDim.x) {
            float v[8], zv[8], go[8], dyv[8], dzv[8];
            gated8<T>(a, r, f, v, zv);
            ld8<T>(static_cast<const T *>(a.dout) + r * a.D + f, go);
            const float iv = inv[f / a.gs], m = dot[f / a.gs] / a.gs;
            const float *yrow = nullptr;
            float yv[8];
            if (a.z) {
                ld8<T>(static_cast<const T *>(a.y) + r * a.D + f, yv);
                yrow = yv;
            }
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const float n = v[i] * iv;
                const float dv = (go[i] * a.weight[f + i] - n * m) * iv;  // (dn - n mean(dn n)) / rms
                if (yrow) {
                    dyv[i] = dv * silu_f(zv[i]);
                    dzv[i] = dv * yrow[i] * silu_grad_f(zv[i]);
                } else {
                    dyv[i] = dv;
                }
            }
            st8<T>(static_cast<T *>(a.dy) + r * a.D + f, dyv);
            if (a.z) st8<T>(static_cast<T *>(a.dz) + r * a.D + f, dzv);
        }
        __syncthreads();
    }
    for (int q = threadIdx.x; q < a.D; q += blockDim.x)  // q = i (D / 8) + f / 8
        atomicAdd(a.dweight + 8 * (q % (a.D / 8)) + q / (a.D / 8), dwp[q]);
}

// Register-resident rows (dim <= 8192): a CTA of NT threads per row, thread i owning the 8-feature
// vectors at 8 (i + NT j), j < VPT, so a row is read from HBM once, with every load of the row in
// flight at the same time, and never re-read.  Group sums as in the kernels above (smem, one shared atomic per warp when
// groups span whole warps).  Two sum buffers alternate between consecutive rows of a CTA, so a
// row needs no barrier after its last use of the sums.
template <typename T, int VPT, int NT>
__global__ void __launch_bounds__(NT) rmsnorm_fwd_reg_kernel(NormArgs a) {
    extern __shared__ float gsum2[];  // [2][ng]
    const int ng = a.D / a.gs;
    int par = 0;
    for (int64_t r = blockIdx.x; r < a.R; r += gridDim.x, par ^= 1) {
        float *gsum = gsum2 + par * ng;
        float v[VPT][8];
#pragma unroll
        for (int j = 0; j < VPT; ++j) {
            const int f = 8 * (threadIdx.x + NT * j);
            if (f < a.D) {
                float zv[8];
                gated8<T>(a, r, f, v[j], zv);
            }
        }
        for (int g = threadIdx.x; g < ng; g += blockDim.x) gsum[g] = 0.f;
        __syncthreads();
#pragma unroll
        for (int j = 0; j < VPT; ++j) {
            const int f = 8 * (threadIdx.x + NT * j);
            const bool valid = f < a.D;
            float sq = 0.f;
            if (valid)
#pragma unroll
                for (int i = 0; i < 8; ++i) sq = fmaf(v[j][i], v[j][i], sq);
            if (8 * NT * j < a.D) group_add(gsum, f, a.gs, valid, sq);  // whole warps take part
        }
        __syncthreads();
#pragma unroll
        for (int j = 0; j < VPT; ++j) {
            const int f = 8 * (threadIdx.x + NT * j);
            if (f < a.D) {
                const float inv = rsqrtf(gsum[f / a.gs] / a.gs + a.eps);
                const float4 w0 = reinterpret_cast<const float4 *>(a.weight + f)[0];
                const float4 w1 = reinterpret_cast<const float4 *>(a.weight + f)[1];
                const float wv[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
#pragma unroll
                for (int i = 0; i < 8; ++i) v[j][i] = v[j][i] * inv * wv[i];
                st8<T>(static_cast<T *>(a.out) + r * a.D + f, v[j]);
            }
        }
    }
}

// Eight elements of a row kept as loaded (bf16: one 16-byte register quad), unpacked on use.
template <typename T> struct Raw8;
template <> struct Raw8<__nv_bfloat16> {
    uint4 u;
    __device__ __forceinline__ void load(const __nv_bfloat16 *p) { u = *reinterpret_cast<const uint4 *>(p); }
    __device__ __forceinline__ void get(float *v) const {
        const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&u);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = __bfloat1622float2(h[i]);
            v[2 * i] = f.x;
            v[2 * i + 1] = f.y;
        }
    }
};
template <> struct Raw8<float> {
    float4 a, b;
    __device__ __forceinline__ void load(const float *p) {
        a = reinterpret_cast<const float4 *>(p)[0];
        b = reinterpret_cast<const float4 *>(p)[1];
    }
    __device__ __forceinline__ void get(float *v) const {
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    }
};

// Backward with register-resident rows, persistent over rows: y, z and dout stay as loaded, the
// gate's sigmoid is evaluated once per element (silu(z) = z s, silu'(z) = s (1 + z (1 - s))), and
// each thread keeps the dweight partials of its own features in registers until one global atomic
// per feature and CTA.
template <typename T, int VPT, int NT>
__global__ void __launch_bounds__(NT, NT <= 256 ? 2 : 1) rmsnorm_bwd_reg_kernel(NormArgs a) {
    extern __shared__ float sums[];  // [2][2 ng]: sum(v^2), then sum(dn n), per row parity
    const int ng = a.D / a.gs;
    const bool gated = a.z != nullptr;
    float dwp[VPT][8];
#pragma unroll
    for (int j = 0; j < VPT; ++j)
#pragma unroll
        for (int i = 0; i < 8; ++i) dwp[j][i] = 0.f;
    // the next row's inputs are loaded while the current row is processed
    Raw8<T> ry[VPT], rz[VPT], rg[VPT], ny[VPT], nz[VPT], nd[VPT];
    auto fetch = [&](int64_t row, Raw8<T> *yy, Raw8<T> *zz, Raw8<T> *dd) {
#pragma unroll
        for (int j = 0; j < VPT; ++j) {
            const int f = 8 * (threadIdx.x + NT * j);
            if (f < a.D) {
                const size_t o = size_t(row) * a.D + f;
                yy[j].load(static_cast<const T *>(a.y) + o);
                if (gated) zz[j].load(static_cast<const T *>(a.z) + o);
                dd[j].load(static_cast<const T *>(a.dout) + o);
            }
        }
    };
    if (blockIdx.x < a.R) fetch(blockIdx.x, ry, rz, rg);
    int par = 0;
    for (int64_t r = blockIdx.x; r < a.R; r += gridDim.x, par ^= 1) {
        float *ssq = sums + par * 2 * ng, *dot = ssq + ng;
        if (r + gridDim.x < a.R) fetch(r + gridDim.x, ny, nz, nd);
        for (int g = threadIdx.x; g < 2 * ng; g += blockDim.x) ssq[g] = 0.f;
        __syncthreads();
        float sg[VPT][8];  // sigmoid(z) of the gate; the gate factor is silu(z) = z sg (1 without the gate)
#pragma unroll
        for (int j = 0; j < VPT; ++j) {
            const int f = 8 * (threadIdx.x + NT * j);
            const bool valid = f < a.D;
            float sq = 0.f;
            if (valid) {
                float y[8], z[8];
                ry[j].get(y);
                if (gated) rz[j].get(z);
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    sg[j][i] = gated ? sigm(z[i]) : 1.f;
                    const float v = y[i] * (gated ? z[i] * sg[j][i] : 1.f);
                    sq = fmaf(v, v, sq);
                }
            }
            if (8 * NT * j < a.D) group_add(ssq, f, a.gs, valid, sq);  // whole warps take part
        }
        __syncthreads();
        float iv[VPT];
#pragma unroll
        for (int j = 0; j < VPT; ++j) {
            const int f = 8 * (threadIdx.x + NT * j);
            const bool valid = f < a.D;
            float sd = 0.f;
            iv[j] = 0.f;
            if (valid) {
                iv[j] = rsqrtf(ssq[f / a.gs] / a.gs + a.eps);
                float y[8], go[8], z[8];
                ry[j].get(y);
                rg[j].get(go);
                if (gated) rz[j].get(z);
                const float4 w0 = reinterpret_cast<const float4 *>(a.weight + f)[0];
                const float4 w1 = reinterpret_cast<const float4 *>(a.weight + f)[1];
                const float wv[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const float n = y[i] * (gated ? z[i] * sg[j][i] : 1.f) * iv[j];
                    dwp[j][i] = fmaf(go[i], n, dwp[j][i]);
                    sd = fmaf(go[i] * wv[i], n, sd);
                }
            }
            if (8 * NT * j < a.D) group_add(dot, f, a.gs, valid, sd);
        }
        __syncthreads();
#pragma unroll
        for (int j = 0; j < VPT; ++j) {
            const int f = 8 * (threadIdx.x + NT * j);
            if (f < a.D) {
                const float m = dot[f / a.gs] / a.gs;
                float y[8], go[8], dyv[8], dzv[8];
                ry[j].get(y);
                rg[j].get(go);
                const float4 w0 = reinterpret_cast<const float4 *>(a.weight + f)[0];
                const float4 w1 = reinterpret_cast<const float4 *>(a.weight + f)[1];
                const float wv[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
                float z[8];
                if (gated) rz[j].get(z);
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const float gz = (gated ? z[i] * sg[j][i] : 1.f);
                    const float n = y[i] * gz * iv[j];
                    const float dv = (go[i] * wv[i] - n * m) * iv[j];  // (dn - n mean(dn n)) / rms
                    dyv[i] = dv * gz;
                    dzv[i] = gated ? dv * y[i] * (sg[j][i] * (1.f + z[i] * (1.f - sg[j][i]))) : 0.f;
                }
                const size_t o = size_t(r) * a.D + f;
                st8<T>(static_cast<T *>(a.dy) + o, dyv);
                if (gated) st8<T>(static_cast<T *>(a.dz) + o, dzv);
            }
        }
#pragma unroll
        for (int j = 0; j < VPT; ++j) {
            ry[j] = ny[j];
            rz[j] = nz[j];
            rg[j] = nd[j];
        }
    }
#pragma unroll
    for (int j = 0; j < VPT; ++j) {
        const int f = 8 * (threadIdx.x + NT * j);
        if (f < a.D)
#pragma unroll
            for (int i = 0; i < 8; ++i) atomicAdd(a.dweight + f + i, dwp[j][i]);
    }
}

// bf16 backward with rows staged in shared memory (dim <= 4096): persistent over rows, y, z and
// dout of the next two rows (up to 24 KB each) loaded by cp.async into a ring of three buffers
// while the current row is processed from its buffer, three CTAs per SM; thread i owns the
// 8-feature vectors at 8 (i + 256 j), j < VPT, and keeps their dweight partials in registers until
// one global atomic per feature and CTA.  Both row sums come from one pass: sum(v^2) and
// sum(dout w v), since sum(dn n) = (1 / rms) sum(dout w v).
template <int VPT>
__global__ void __launch_bounds__(256, 3) rmsnorm_bwd_tile_kernel(NormArgs a) {
    using T = __nv_bfloat16;
    extern __shared__ __align__(16) unsigned char nsm[];
    const int ng = a.D / a.gs, D8 = a.D / 8;
    const bool gated = a.z != nullptr;
    float *sums = reinterpret_cast<float *>(nsm);  // [2][2 ng]: sum(v^2), then sum(dn n), per row parity
    uint4 *rows = reinterpret_cast<uint4 *>(nsm + ((sizeof(float) * 4 * ng + 15) / 16) * 16);  // [3][3][D8]
    auto stage = [&](int64_t row, int slot) {
        uint4 *dst = rows + size_t(slot) * 3 * D8;
        for (int i = threadIdx.x; i < 3 * D8; i += blockDim.x) {
            const int which = i / D8, v = i - which * D8;
            if (which == 1 && !gated) continue;
            const T *src = static_cast<const T *>(which == 0 ? a.y : which == 1 ? a.z : a.dout);
            cp_async16_zfill(dst + i, src + size_t(row) * a.D + 8 * v, true);
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
    float dwp[VPT][8];
#pragma unroll
    for (int j = 0; j < VPT; ++j)
#pragma unroll
        for (int i = 0; i < 8; ++i) dwp[j][i] = 0.f;
    if (blockIdx.x < a.R) stage(blockIdx.x, 0);
    if (blockIdx.x + gridDim.x < a.R) stage(blockIdx.x + gridDim.x, 1);
    int k = 0;
    for (int64_t r = blockIdx.x; r < a.R; r += gridDim.x, ++k) {
        const int slot = k % 3;
        float *ssq = sums + (k & 1) * 2 * ng, *dot = ssq + ng;
        if (r + 2 * int64_t(gridDim.x) < a.R) stage(r + 2 * int64_t(gridDim.x), (k + 2) % 3);
        // this row's group is complete once at most the groups of the rows after it are pending
        const int later = int(r + gridDim.x < a.R) + int(r + 2 * int64_t(gridDim.x) < a.R);
        if (later == 2)
            asm volatile("cp.async.wait_group 2;" ::: "memory");
        else if (later == 1)
            asm volatile("cp.async.wait_group 1;" ::: "memory");
        else
            asm volatile("cp.async.wait_group 0;" ::: "memory");
        for (int g = threadIdx.x; g < 2 * ng; g += blockDim.x) ssq[g] = 0.f;
        __syncthreads();
        const uint4 *ry = rows + size_t(slot) * 3 * D8, *rz = ry + D8, *rg = rz + D8;
        auto unpack = [](uint4 u, float *v) {
            const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&u);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float2 f = __bfloat1622float2(h[i]);
                v[2 * i] = f.x;
                v[2 * i + 1] = f.y;
            }
        };
        // one pass for both row sums: sum(v^2) and sum(dout w v) (= rms sum(dn n))
        float sg[VPT][8];  // sigmoid(z) of the gate; the gate factor is silu(z) = z sg (1 without the gate)
#pragma unroll
        for (int j = 0; j < VPT; ++j) {
            const int v = threadIdx.x + 256 * j, f = 8 * v;
            const bool valid = f < a.D;
            float sq = 0.f, sd = 0.f;
            if (valid) {
                float y[8], z[8], go[8];
                unpack(ry[v], y);
                unpack(rg[v], go);
                if (gated) unpack(rz[v], z);
                const float4 w0 = reinterpret_cast<const float4 *>(a.weight + f)[0];
                const float4 w1 = reinterpret_cast<const float4 *>(a.weight + f)[1];
                const float wv[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    sg[j][i] = gated ? sigm(z[i]) : 1.f;
                    const float vv = y[i] * (gated ? z[i] * sg[j][i] : 1.f);
                    sq = fmaf(vv, vv, sq);
                    sd = fmaf(go[i] * wv[i], vv, sd);
                }
            }
            if (8 * 256 * j < a.D) {  // whole warps take part
                group_add(ssq, f, a.gs, valid, sq);
                group_add(dot, f, a.gs, valid, sd);
            }
        }
        __syncthreads();
#pragma unroll
        for (int j = 0; j < VPT; ++j) {
            const int v = threadIdx.x + 256 * j, f = 8 * v;
            if (f < a.D) {
                const float iv = rsqrtf(ssq[f / a.gs] / a.gs + a.eps);
                const float m = iv * dot[f / a.gs] / a.gs;  // mean(dn n)
                float y[8], go[8], z[8], dyv[8], dzv[8];
                unpack(ry[v], y);
                unpack(rg[v], go);
                if (gated) unpack(rz[v], z);
                const float4 w0 = reinterpret_cast<const float4 *>(a.weight + f)[0];
                const float4 w1 = reinterpret_cast<const float4 *>(a.weight + f)[1];
                const float wv[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const float gz = gated ? z[i] * sg[j][i] : 1.f;
                    const float n = y[i] * gz * iv;
                    dwp[j][i] = fmaf(go[i], n, dwp[j][i]);
                    const float dv = (go[i] * wv[i] - n * m) * iv;  // (dn - n mean(dn n)) / rms
                    dyv[i] = dv * gz;
                    dzv[i] = gated ? dv * y[i] * (sg[j][i] * (1.f + z[i] * (1.f - sg[j][i]))) : 0.f;
                }
                const size_t o = size_t(r) * a.D + f;
                st8<T>(static_cast<T *>(a.dy) + o, dyv);
                if (gated) st8<T>(static_cast<T *>(a.dz) + o, dzv);
            }
        }
        __syncthreads();  // this slot's rows and sums are read: the next stage may overwrite them
    }
#pragma unroll
    for (int j = 0; j < VPT; ++j) {
        const int f = 8 * (threadIdx.x + 256 * j);
        if (f < a.D)
#pragma unroll
            for (int i = 0; i < 8; ++i) atomicAdd(a.dweight + f + i, dwp[j][i]);
    }
}

int num_sms();

template <int VPT>
cudaError_t norm_bwd_tile_launch(const NormArgs &a, cudaStream_t st) {
    const int ng = a.D / a.gs;
    const size_t smem = ((sizeof(float) * 4 * ng + 15) / 16) * 16 + size_t(3) * 3 * a.D * 2;
    auto k = rmsnorm_bwd_tile_kernel<VPT>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    int per_sm = 0;
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, 256, smem);
    if (e != cudaSuccess) return e;
    const int blocks = int(std::min<int64_t>(a.R, int64_t(num_sms()) * std::max(per_sm, 1)));
    trace_begin("gated_rmsnorm_bwd", st);
    k<<<blocks, 256, smem, st>>>(a);
    trace_end(st);
    return cudaGetLastError();
}

int num_sms() {
    int dev = 0, sms = 152;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    return std::max(sms, 1);
}

// Register-resident RMSNorm launches.  Forward (dim <= 8192): CTAs of 256 threads, VPT = ceil(dim /
// 2048) vectors per thread (measured faster at dim 4096 than 512 threads of one vector).  Backward
// (dim <= 4096): one vector per thread in CTAs of 256 or 512 threads, persistent, as many CTAs as
// the SMs hold at once.
template <typename T, int VPT>
cudaError_t norm_fwd_reg_launch(const NormArgs &a, cudaStream_t st) {
    const size_t smem = sizeof(float) * 2 * (a.D / a.gs);
    const int blocks = int(std::min<int64_t>(a.R, int64_t(num_sms()) * 16));
    trace_begin("gated_rmsnorm_fwd", st);
    rmsnorm_fwd_reg_kernel<T, VPT, 256><<<blocks, 256, smem, st>>>(a);
    trace_end(st);
    return cudaGetLastError();
}

template <typename T, int NT>
cudaError_t norm_reg_launch(const NormArgs &a, bool bwd, cudaStream_t st) {
    const int ng = a.D / a.gs;
    if (!bwd) {
        switch ((a.D + 2047) / 2048) {
            case 1: return norm_fwd_reg_launch<T, 1>(a, st);
            case 2: return norm_fwd_reg_launch<T, 2>(a, st);
            case 3: return norm_fwd_reg_launch<T, 3>(a, st);
            default: return norm_fwd_reg_launch<T, 4>(a, st);
        }
    }
    const size_t smem = sizeof(float) * 4 * ng;
    auto k = rmsnorm_bwd_reg_kernel<T, 1, NT>;
    int per_sm = 0;
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, NT, smem);
    if (e != cudaSuccess) return e;
    const int blocks = int(std::min<int64_t>(a.R, int64_t(num_sms()) * std::max(per_sm, 1)));
    trace_begin("gated_rmsnorm_bwd", st);
    k<<<blocks, NT, smem, st>>>(a);
    trace_end(st);
    return cudaGetLastError();
}

template <typename T>
cudaError_t norm_reg(const NormArgs &a, bool bwd, cudaStream_t st) {
    if (a.D <= 8 * 256) return norm_reg_launch<T, 256>(a, bwd, st);
    if (a.D <= 8 * 512) return norm_reg_launch<T, 512>(a, bwd, st);
    return norm_reg_launch<T, 512>(a, false, st);  // forward only: the backward stops at 4096
}
constexpr int kNormRegMaxDim = 8192, kNormRegMaxDimBwd = 4096;

template <typename T, int W>
cudaError_t conv_launch_w(const ConvArgs &a, bool bwd, bool vec, bool vec4, bool tile, cudaStream_t st) {
    if constexpr (sizeof(T) == 2) {
        if (tile) {  // bf16 through shared-memory tiles
            const dim3 tgrid((a.C + kTileC - 1) / kTileC, (a.L + kTileT - 1) / kTileT, a.B);
            if (!bwd) {
                trace_begin("conv1d_fwd", st);
                conv1d_fwd_tile_kernel<W><<<tgrid, 256, 0, st>>>(a);
            } else {
                auto k = conv1d_bwd_tile_kernel<W>;
                cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, int(kConvBwdTileSmem));
                trace_begin("conv1d_bwd", st);
                k<<<tgrid, 256, kConvBwdTileSmem, st>>>(a);
            }
            trace_end(st);
            return cudaGetLastError();
        }
    }
    dim3 block(32, kRows);
    dim3 grid((a.C + 63) / 64, (a.L + kRows * kRun - 1) / (kRows * kRun), a.B);
    if (grid.y == 0) return cudaSuccess;
    if (vec4 && (!bwd || W <= 4)) {  // four channels per thread: 128 channels per block column
                                     // (the backward of wider filters keeps two channels)
        grid.x = (a.C + 127) / 128;
        trace_begin(bwd ? "conv1d_bwd" : "conv1d_fwd", st);
        if constexpr (W <= 4) {
            if (bwd) conv1d_bwd4_kernel<T, W><<<grid, block, 0, st>>>(a);
        }
        if (!bwd) conv1d_fwd4_kernel<T, W><<<grid, block, 0, st>>>(a);
        trace_end(st);
        return cudaGetLastError();
    }
    if (!bwd) {
        trace_begin("conv1d_fwd", st);
        if (vec) conv1d_fwd_kernel<T, W, true><<<grid, block, 0, st>>>(a);
        else conv1d_fwd_kernel<T, W, false><<<grid, block, 0, st>>>(a);
    } else {
        trace_begin("conv1d_bwd", st);
        if (vec) conv1d_bwd_kernel<T, W, true><<<grid, block, 0, st>>>(a);
        else conv1d_bwd_kernel<T, W, false><<<grid, block, 0, st>>>(a);
    }
    trace_end(st);
    return cudaGetLastError();
}

template <typename T>
cudaError_t conv_launch(const ConvArgs &a, bool bwd, bool vec, bool vec4, bool tile, cudaStream_t st) {
    switch (a.W) {
        case 1: return conv_launch_w<T, 1>(a, bwd, vec, vec4, tile, st);
        case 2: return conv_launch_w<T, 2>(a, bwd, vec, vec4, tile, st);
        case 3: return conv_launch_w<T, 3>(a, bwd, vec, vec4, tile, st);
        case 4: return conv_launch_w<T, 4>(a, bwd, vec, vec4, tile, st);
        case 5: return conv_launch_w<T, 5>(a, bwd, vec, vec4, tile, st);
        case 6: return conv_launch_w<T, 6>(a, bwd, vec, vec4, tile, st);
        case 7: return conv_launch_w<T, 7>(a, bwd, vec, vec4, tile, st);
        default: return conv_launch_w<T, 8>(a, bwd, vec, vec4, tile, st);
    }
}

frac_status glue_fail(frac_status s, const char *msg) {
    set_last_error(msg);
    return s;
}

frac_status glue_cuda(cudaError_t e, const char *where) {
    if (e == cudaSuccess) return FRAC_OK;
    char m[160];
    std::snprintf(m, sizeof(m), "%s: %s", where, cudaGetErrorString(e));
    return glue_fail(FRAC_ERR_CUDA, m);
}

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

frac_status conv_check(const frac_conv_dims *d, bool need_seq) {
    if (!d) return glue_fail(FRAC_ERR_INVALID_ARGUMENT, "dims must not be NULL");
    if (d->batch < 1 || (need_seq && d->seqlen < 0) || d->channels < 1 || d->width < 1)
        return glue_fail(FRAC_ERR_INVALID_ARGUMENT, "need batch >= 1, seqlen >= 0, channels >= 1, width >= 1");
    if (d->width > kMaxW) return glue_fail(FRAC_ERR_UNSUPPORTED, "width above 8 is not supported");
    if (d->dtype != FRAC_DTYPE_F32 && d->dtype != FRAC_DTYPE_BF16)
        return glue_fail(FRAC_ERR_INVALID_ARGUMENT, "unknown dtype");
    if (d->flags & ~int32_t(FRAC_CONV_SILU)) return glue_fail(FRAC_ERR_INVALID_ARGUMENT, "unknown flag");
    // grid: (channels / 64, seqlen / (kRows kRun), batch) within the launch limits
    if (d->batch > 65535 || d->seqlen > int64_t(65535) * kRows * kRun || d->channels > (int64_t(1) << 24))
        return glue_fail(FRAC_ERR_UNSUPPORTED, "dimension too large");
    return FRAC_OK;
}

frac_status norm_check(const frac_norm_dims *d) {
    if (!d) return glue_fail(FRAC_ERR_INVALID_ARGUMENT, "dims must not be NULL");
    if (d->rows < 0 || d->dim < 8 || d->group_size < 8 || d->dim % d->group_size || d->group_size % 8 ||
        !(d->eps >= 0.f))
        return glue_fail(FRAC_ERR_INVALID_ARGUMENT,
                         "need rows >= 0, group_size a multiple of 8 dividing dim, eps >= 0");
    if (d->dtype != FRAC_DTYPE_F32 && d->dtype != FRAC_DTYPE_BF16)
        return glue_fail(FRAC_ERR_INVALID_ARGUMENT, "unknown dtype");
    // the backward keeps dim + 2 dim / group_size floats in shared memory (<= 160 KB)
    if (d->dim > 32768) return glue_fail(FRAC_ERR_UNSUPPORTED, "dim above 32768 is not supported");
    if (d->flags) return glue_fail(FRAC_ERR_INVALID_ARGUMENT, "flags must be 0");
    return FRAC_OK;
}

}  // namespace
}  // namespace frac

#define GLUE_REQ(p, a)                                                                             \
    do {                                                                                           \
        if (!(p) || !frac::aligned(p, a)) {                                                        \
            char m_[96];                                                                           \
            std::snprintf(m_, sizeof(m_), "%s must be non-NULL and %d-byte aligned", #p, int(a));  \
            return frac::glue_fail(FRAC_ERR_INVALID_ARGUMENT, m_);                                 \
        }                                                                                          \
    } while (0)
#define GLUE_OPT(p, a)                                                                             \
    do {                                                                                           \
        if ((p) && !frac::aligned(p, a))                                                           \
            return frac::glue_fail(FRAC_ERR_INVALID_ARGUMENT, #p " is misaligned");                \
    } while (0)

extern "C" {

frac_status frac_conv1d_fwd(const frac_conv_dims *dims, const void *x, const float *w,
                            const float *bias, const void *state_in, void *u, void *state_out,
                            void *stream) {
    frac::set_last_error("");
    frac_status s = frac::conv_check(dims, true);
    if (s) return s;
    const size_t es = dims->dtype == FRAC_DTYPE_BF16 ? 2 : 4;
    GLUE_REQ(w, 4);
    GLUE_OPT(bias, 4);
    GLUE_OPT(state_in, es);
    GLUE_OPT(state_out, es);
    if (dims->seqlen > 0) {
        GLUE_REQ(x, es);
        GLUE_REQ(u, es);
    }
    if (state_out && state_out == state_in)
        return frac::glue_fail(FRAC_ERR_INVALID_ARGUMENT, "state_out must not alias state_in");
    frac::ConvArgs a = {};
    a.B = int(dims->batch); a.L = int(dims->seqlen); a.C = int(dims->channels); a.W = int(dims->width);
    a.silu = dims->flags & FRAC_CONV_SILU;
    a.x = x; a.w = w; a.bias = bias; a.state_in = state_in; a.u = u; a.state_out = state_out;
    cudaStream_t st = (cudaStream_t)stream;
    if (a.L == 0) {  // nothing to convolve: the carried state passes through unchanged
        if (!state_out) return FRAC_OK;
        const size_t n = size_t(a.B) * a.C * (a.W - 1) * es;
        return frac::glue_cuda(state_in ? cudaMemcpyAsync(state_out, state_in, n, cudaMemcpyDeviceToDevice, st)
                                        : cudaMemsetAsync(state_out, 0, n, st),
                               "frac_conv1d_fwd");
    }
    const bool vec = a.C % 2 == 0 && frac::aligned(x, 2 * es) && frac::aligned(u, 2 * es);
    const bool vec4 = a.C % 4 == 0 && frac::aligned(x, 4 * es) && frac::aligned(u, 4 * es);
    const bool tile = a.C % 8 == 0 && frac::aligned(x, 16) && frac::aligned(u, 4);
    return frac::glue_cuda(dims->dtype == FRAC_DTYPE_BF16
                               ? frac::conv_launch<__nv_bfloat16>(a, false, vec, vec4, tile, st)
                               : frac::conv_launch<float>(a, false, vec, vec4, false, st),
                           "frac_conv1d_fwd");
}

frac_status frac_conv1d_bwd(const frac_conv_dims *dims, const void *x, const float *w,
                            const float *bias, const void *state_in, const void *du, void *dx,
                            float *dw, float *dbias, void *dstate_in, void *stream) {
    frac::set_last_error("");
    frac_status s = frac::conv_check(dims, true);
    if (s) return s;
    const size_t es = dims->dtype == FRAC_DTYPE_BF16 ? 2 : 4;
    GLUE_REQ(w, 4);
    GLUE_REQ(dw, 4);
    GLUE_OPT(bias, 4);
    GLUE_OPT(dbias, 4);
    GLUE_OPT(state_in, es);
    GLUE_OPT(dstate_in, es);
    if (dims->seqlen > 0) {
        GLUE_REQ(x, es);
        GLUE_REQ(du, es);
        GLUE_REQ(dx, es);
    }
    frac::ConvArgs a = {};
    a.B = int(dims->batch); a.L = int(dims->seqlen); a.C = int(dims->channels); a.W = int(dims->width);
    a.silu = dims->flags & FRAC_CONV_SILU;
    a.x = x; a.w = w; a.bias = bias; a.state_in = state_in; a.du = du; a.dx = dx; a.dw = dw;
    a.dbias = dbias; a.dstate = dstate_in;
    cudaStream_t st = (cudaStream_t)stream;
    cudaError_t e = cudaMemsetAsync(dw, 0, sizeof(float) * a.C * a.W, st);
    if (e == cudaSuccess && dbias) e = cudaMemsetAsync(dbias, 0, sizeof(float) * a.C, st);
    // the carried inputs that no output reads (only when L < W - 1 leaves some untouched) get 0
    if (e == cudaSuccess && dstate_in && a.W > 1)
        e = cudaMemsetAsync(dstate_in, 0, size_t(a.B) * a.C * (a.W - 1) * es, st);
    if (e == cudaSuccess && a.L > 0) {
        const bool vec = a.C % 2 == 0 && frac::aligned(x, 2 * es) && frac::aligned(du, 2 * es) &&
                         frac::aligned(dx, 2 * es);
        const bool vec4 = a.C % 4 == 0 && frac::aligned(x, 4 * es) && frac::aligned(du, 4 * es) &&
                          frac::aligned(dx, 4 * es);
        const bool tile = a.C % 8 == 0 && frac::aligned(x, 16) && frac::aligned(du, 16) && frac::aligned(dx, 4);
        e = dims->dtype == FRAC_DTYPE_BF16 ? frac::conv_launch<__nv_bfloat16>(a, true, vec, vec4, tile, st)
                                           : frac::conv_launch<float>(a, true, vec, vec4, false, st);
    }
    return frac::glue_cuda(e, "frac_conv1d_bwd");
}

frac_status frac_conv1d_step(const frac_conv_dims *dims, const void *x_t, const float *w,
                             const float *bias, void *state, void *u_t, void *stream) {
    frac::set_last_error("");
    frac_status s = frac::conv_check(dims, false);
    if (s) return s;
    const size_t es = dims->dtype == FRAC_DTYPE_BF16 ? 2 : 4;
    GLUE_REQ(x_t, es);
    GLUE_REQ(w, 4);
    GLUE_OPT(bias, 4);
    GLUE_REQ(u_t, es);
    if (dims->width > 1) GLUE_REQ(state, es);
    frac::ConvArgs a = {};
    a.B = int(dims->batch); a.L = 1; a.C = int(dims->channels); a.W = int(dims->width);
    a.silu = dims->flags & FRAC_CONV_SILU;
    a.w = w; a.bias = bias; a.state_out = state;
    cudaStream_t st = (cudaStream_t)stream;
    const int64_t n = int64_t(a.B) * a.C;
    const unsigned blocks = unsigned((n + 255) / 256);
    frac::trace_begin("conv1d_step", st);
    if (dims->dtype == FRAC_DTYPE_BF16)
        frac::conv1d_step_kernel<__nv_bfloat16><<<blocks, 256, 0, st>>>(
            a, static_cast<const __nv_bfloat16 *>(x_t), static_cast<__nv_bfloat16 *>(u_t));
    else
        frac::conv1d_step_kernel<float><<<blocks, 256, 0, st>>>(a, static_cast<const float *>(x_t),
                                                                static_cast<float *>(u_t));
    frac::trace_end(st);
    return frac::glue_cuda(cudaGetLastError(), "frac_conv1d_step");
}

frac_status frac_gated_rmsnorm_fwd(const frac_norm_dims *dims, const void *y, const void *z,
                                   const float *weight, void *out, void *stream) {
    frac::set_last_error("");
    frac_status s = frac::norm_check(dims);
    if (s) return s;
    GLUE_REQ(weight, 4);
    if (dims->rows == 0) return FRAC_OK;
    GLUE_REQ(y, 16);
    GLUE_OPT(z, 16);
    GLUE_REQ(out, 16);
    frac::NormArgs a = {};
    a.R = dims->rows; a.D = int(dims->dim); a.gs = int(dims->group_size); a.eps = dims->eps;
    a.y = y; a.z = z; a.weight = weight; a.out = out;
    cudaStream_t st = (cudaStream_t)stream;
    if (a.D <= frac::kNormRegMaxDim)
        return frac::glue_cuda(dims->dtype == FRAC_DTYPE_BF16 ? frac::norm_reg<__nv_bfloat16>(a, false, st)
                                                              : frac::norm_reg<float>(a, false, st),
                               "frac_gated_rmsnorm_fwd");
    const int blocks = int(std::min<int64_t>(a.R, int64_t(frac::num_sms()) * 16));
    const size_t smem = sizeof(float) * (a.D / a.gs);
    frac::trace_begin("gated_rmsnorm_fwd", st);
    if (dims->dtype == FRAC_DTYPE_BF16)
        frac::rmsnorm_fwd_kernel<__nv_bfloat16><<<blocks, 256, smem, st>>>(a);
    else
        frac::rmsnorm_fwd_kernel<float><<<blocks, 256, smem, st>>>(a);
    frac::trace_end(st);
    return frac::glue_cuda(cudaGetLastError(), "frac_gated_rmsnorm_fwd");
}

frac_status frac_gated_rmsnorm_bwd(const frac_norm_dims *dims, const void *y, const void *z,
                                   const float *weight, const void *dout, void *dy, void *dz,
                                   float *dweight, void *stream) {
    frac::set_last_error("");
    frac_status s = frac::norm_check(dims);
    if (s) return s;
    GLUE_REQ(weight, 4);
    GLUE_REQ(dweight, 4);
    if (dims->rows > 0) {
        GLUE_REQ(y, 16);
        GLUE_REQ(dout, 16);
        GLUE_REQ(dy, 16);
        if (z) GLUE_REQ(dz, 16);
        GLUE_OPT(z, 16);
    }
    frac::NormArgs a = {};
    a.R = dims->rows; a.D = int(dims->dim); a.gs = int(dims->group_size); a.eps = dims->eps;
    a.y = y; a.z = z; a.dout = dout; a.weight = weight; a.dy = dy; a.dz = dz; a.dweight = dweight;
    cudaStream_t st = (cudaStream_t)stream;
    cudaError_t e = cudaMemsetAsync(dweight, 0, sizeof(float) * a.D, st);
    if (e == cudaSuccess && a.R > 0 && a.D <= frac::kNormRegMaxDimBwd) {
        const bool al16 = frac::aligned(y, 16) && frac::aligned(dout, 16) && (!z || frac::aligned(z, 16));
        if (dims->dtype == FRAC_DTYPE_BF16 && al16)  // rows staged in shared memory
            e = a.D <= 2048 ? frac::norm_bwd_tile_launch<1>(a, st) : frac::norm_bwd_tile_launch<2>(a, st);
        else
            e = dims->dtype == FRAC_DTYPE_BF16 ? frac::norm_reg<__nv_bfloat16>(a, true, st)
                                               : frac::norm_reg<float>(a, true, st);
    } else if (e == cudaSuccess && a.R > 0) {
        const int blocks = int(std::min<int64_t>(a.R, int64_t(frac::num_sms()) * 4));
        const size_t smem = sizeof(float) * (a.D + 2 * (a.D / a.gs));
        auto k16 = frac::rmsnorm_bwd_kernel<__nv_bfloat16>;
        auto k32 = frac::rmsnorm_bwd_kernel<float>;
        cudaFuncSetAttribute(k16, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        cudaFuncSetAttribute(k32, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        frac::trace_begin("gated_rmsnorm_bwd", st);
        if (dims->dtype == FRAC_DTYPE_BF16)
            k16<<<blocks, 256, smem, st>>>(a);
        else
            k32<<<blocks, 256, smem, st>>>(a);
        frac::trace_end(st);
        e = cudaGetLastError();
    }
    return frac::glue_cuda(e, "frac_gated_rmsnorm_bwd");
}

}  // extern "C"
