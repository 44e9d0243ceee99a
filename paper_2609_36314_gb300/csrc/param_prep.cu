// Scan-parameter construction of the Frac layer and its backward (HBM-bound elementwise work).
//
// Per position and head, from the outputs of the layer's projections (Sec. 3.3; Algorithm 1 of
// App. D; clip ranges of App. E.3):
//   Delta  = clip(softplus(dt_raw + dt_bias_h), dt_min, dt_max)
//   alpha  = sigmoid(alpha_raw)            (1 with FRAC_PREP_ALPHA_ONE)
//   lambda = clip(softplus(lam_raw), lam_min, lam_max)
//   w_read  = softmax_m(-alpha ln tau_m + g_read_m)      (Eq. read-softmax)
//   w_write = softmax_m(-alpha ln tau_m + g_write_m)     (divided by lambda with the exact ZOH
//                                                         injection of Eq. rho-beta-def-frac)
// with the App. G ablations as flags (no softmax, no read / write prior).  The backward is the
// adjoint of the same formulas; clipping passes the gradient where the clipped value lies in
// [min, max].
//
// One thread per (position, head) row; a row's K logits are one or two 16-byte vectors when
// K * element size allows, so a warp reads and writes whole contiguous segments.  The backward
// also sums the bias and timescale gradients over positions: its grid stride is a multiple of
// the head count, so every row a thread visits has the same head and the sums stay in
// registers until one shared-memory (then global) atomic per block slot.
#include <algorithm>
#include <cstdio>
#include <initializer_list>

#include "../../include/frac.h"
#include "common.cuh"
#include "kernels.h"

namespace frac {
namespace {

struct PrepArgs {
    int64_t n;  // rows = positions x heads
    int H, K, flags;
    float dt_min, dt_max, lam_min, lam_max;
    const float *dt_raw, *dt_bias, *alpha_raw, *lam_raw, *tau;
    const void *g_read, *g_write;
    // forward outputs
    float *dt, *alpha, *lam;
    void *w_read, *w_write;
    // backward inputs / outputs
    const float *ddt, *dalpha, *dlam;
    const void *dw_read, *dw_write;
    float *ddt_raw, *dalpha_raw, *dlam_raw;
    void *dg_read, *dg_write;
    float *ddt_bias, *dtau;
};

__device__ __forceinline__ float softplus_f(float x) { return fmaxf(x, 0.f) + log1pf(expf(-fabsf(x))); }
__device__ __forceinline__ float sigmoid_f(float x) {
    const float e = expf(-fabsf(x));
    return x >= 0.f ? 1.f / (1.f + e) : e / (1.f + e);
}

// K values of one row (K <= KP); VEC: K == KP and the row is a whole number of 16-byte pieces.
template <typename T, int KP, bool VEC>
__device__ __forceinline__ void load_row(const void *base, int64_t row, int K, float *v) {
    const T *p = static_cast<const T *>(base) + row * K;
    if constexpr (VEC) {
        constexpr int PER = 16 / sizeof(T);
#pragma unroll
        for (int q = 0; q < KP / PER; ++q) {
            const uint4 u = reinterpret_cast<const uint4 *>(p)[q];
            const T *e = reinterpret_cast<const T *>(&u);
#pragma unroll
            for (int i = 0; i < PER; ++i) v[q * PER + i] = to_f(e[i]);
        }
    } else {
#pragma unroll
        for (int m = 0; m < KP; ++m) v[m] = m < K ? to_f(p[m]) : 0.f;
    }
}

template <typename T, int KP, bool VEC>
__device__ __forceinline__ void store_row(void *base, int64_t row, int K, const float *v) {
    T *p = static_cast<T *>(base) + row * K;
    if constexpr (VEC) {
        constexpr int PER = 16 / sizeof(T);
#pragma unroll
        for (int q = 0; q < KP / PER; ++q) {
            uint4 u;
            T *e = reinterpret_cast<T *>(&u);
#pragma unroll
            for (int i = 0; i < PER; ++i) e[i] = from_f<T>(v[q * PER + i]);
            reinterpret_cast<uint4 *>(p)[q] = u;
        }
    } else {
#pragma unroll
        for (int m = 0; m < KP; ++m)
            if (m < K) p[m] = from_f<T>(v[m]);
    }
}

// softmax over the first K entries in place (or nothing when the softmax is switched off)
template <int KP>
__device__ __forceinline__ void softmax_row(float *z, int K, bool on) {
    if (!on) return;
    float mx = -INFINITY;
#pragma unroll
    for (int m = 0; m < KP; ++m)
        if (m < K) mx = fmaxf(mx, z[m]);
    float s = 0.f;
#pragma unroll
    for (int m = 0; m < KP; ++m) {
        z[m] = m < K ? expf(z[m] - mx) : 0.f;
        s += z[m];
    }
    const float inv = 1.f / s;
#pragma unroll
    for (int m = 0; m < KP; ++m) z[m] *= inv;
}

// The forward of one row, shared by both kernels: Delta (and softplus before the clip and its
// argument), alpha, lambda (and softplus before the clip), ln tau, the read weights and the
// write weights b before the ZOH division.
template <typename T, int KP, bool VEC>
struct Row {
    float pre, sp_dt, dt, alpha, sp_lam, lam;
    float ltau[KP], wr[KP], b[KP];

    // ltab: ln tau of every (head, mode) in shared memory, or null (then evaluated here)
    __device__ __forceinline__ void compute(const PrepArgs &a, int64_t r, int h, const float *ltab = nullptr) {
        const int K = a.K;
        pre = a.dt_raw[r] + (a.dt_bias ? a.dt_bias[h] : 0.f);
        sp_dt = softplus_f(pre);
        dt = fminf(fmaxf(sp_dt, a.dt_min), a.dt_max);
        alpha = (a.flags & FRAC_PREP_ALPHA_ONE) ? 1.f : sigmoid_f(a.alpha_raw[r]);
        sp_lam = softplus_f(a.lam_raw[r]);
        lam = fminf(fmaxf(sp_lam, a.lam_min), a.lam_max);
        load_row<T, KP, VEC>(a.g_read, r, K, wr);
        load_row<T, KP, VEC>(a.g_write, r, K, b);
        const bool rp = !(a.flags & FRAC_PREP_NO_READ_PRIOR), wp = !(a.flags & FRAC_PREP_NO_WRITE_PRIOR);
#pragma unroll
        for (int m = 0; m < KP; ++m) {
            ltau[m] = m < K ? (ltab ? ltab[h * K + m] : logf(__ldg(a.tau + h * K + m))) : 0.f;
            const float prior = -alpha * ltau[m];
            if (rp) wr[m] += prior;
            if (wp) b[m] += prior;
        }
        const bool sm = !(a.flags & FRAC_PREP_NO_SOFTMAX);
        softmax_row<KP>(wr, K, sm);
        softmax_row<KP>(b, K, sm);
    }
};

// ln tau of every (head, mode) in shared memory when the table is at most kTauTab entries (the
// logarithm is then evaluated once per block instead of K times per row)
constexpr int kTauTab = 4096;

template <typename T, int KP, bool VEC>
__global__ void __launch_bounds__(256) param_prep_fwd_kernel(PrepArgs a) {
    __shared__ float ltab_s[kTauTab];
    const bool tab = a.H * a.K <= kTauTab;
    if (tab) {
        for (int i = threadIdx.x; i < a.H * a.K; i += blockDim.x) ltab_s[i] = logf(__ldg(a.tau + i));
        __syncthreads();
    }
    const int64_t stride = int64_t(gridDim.x) * blockDim.x;
    for (int64_t r = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; r < a.n; r += stride) {
        const int h = int(r % a.H);
        Row<T, KP, VEC> w;
        w.compute(a, r, h, tab ? ltab_s : nullptr);
        a.dt[r] = w.dt;
        a.alpha[r] = w.alpha;
        a.lam[r] = w.lam;
        if (a.flags & FRAC_PREP_ZOH_INJECTION) {
            const float il = 1.f / w.lam;
#pragma unroll
            for (int m = 0; m < KP; ++m) w.b[m] *= il;
        }
        store_row<T, KP, VEC>(a.w_read, r, a.K, w.wr);
        store_row<T, KP, VEC>(a.w_write, r, a.K, w.b);
    }
}

// adjoint of softmax (or of the identity when the softmax is off), in place on dw
template <int KP>
__device__ __forceinline__ void softmax_bwd_row(const float *w, float *dw, int K, bool on) {
    if (!on) return;
    float s = 0.f;
#pragma unroll
    for (int m = 0; m < KP; ++m)
        if (m < K) s = fmaf(w[m], dw[m], s);
#pragma unroll
    for (int m = 0; m < KP; ++m) dw[m] = m < K ? w[m] * (dw[m] - s) : 0.f;
}

template <typename T, int KP, bool VEC>
__global__ void __launch_bounds__(256, KP <= 8 ? 3 : 1) param_prep_bwd_kernel(PrepArgs a, int64_t hstride) {
    extern __shared__ float red[];  // [min(H, blockDim)][KP + 1] when H <= blockDim
    __shared__ float ltab_s[kTauTab], itab_s[kTauTab];  // ln tau and 1 / tau per (head, mode)
    const int K = a.K, H = a.H;
    const int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    const bool reduce = a.dtau || a.ddt_bias;
    const bool shared_slots = reduce && H <= int(blockDim.x);
    const bool tab = H * K <= kTauTab;
    if (tab)
        for (int q = threadIdx.x; q < H * K; q += blockDim.x) {
            const float tv = __ldg(a.tau + q);
            ltab_s[q] = logf(tv);
            itab_s[q] = 1.f / tv;
        }
    if (shared_slots)
        for (int q = threadIdx.x; q < H * (KP + 1); q += blockDim.x) red[q] = 0.f;
    if (tab || shared_slots) __syncthreads();
    const int h = int(i % H);  // every row this thread visits has this head
    float acc_bias = 0.f, acc_tau[KP];
#pragma unroll
    for (int m = 0; m < KP; ++m) acc_tau[m] = 0.f;
    const bool sm = !(a.flags & FRAC_PREP_NO_SOFTMAX);
    const bool rp = !(a.flags & FRAC_PREP_NO_READ_PRIOR), wp = !(a.flags & FRAC_PREP_NO_WRITE_PRIOR);
    for (int64_t r = i; i < hstride && r < a.n; r += hstride) {
        Row<T, KP, VEC> w;
        w.compute(a, r, h, tab ? ltab_s : nullptr);
        float dwr[KP], db[KP];
        load_row<T, KP, VEC>(a.dw_read, r, K, dwr);
        load_row<T, KP, VEC>(a.dw_write, r, K, db);
        float dlam_tot = a.dlam[r];
        if (a.flags & FRAC_PREP_ZOH_INJECTION) {  // w_write = b / lambda
            const float il = 1.f / w.lam;
            float s = 0.f;
#pragma unroll
            for (int m = 0; m < KP; ++m) {
                s = fmaf(db[m], w.b[m], s);
                db[m] *= il;
            }
            dlam_tot -= s * il * il;
        }
        softmax_bwd_row<KP>(w.wr, dwr, K, sm);  // now d(read logits)
        softmax_bwd_row<KP>(w.b, db, K, sm);    // now d(write logits)
        float dal = a.dalpha[r];
#pragma unroll
        for (int m = 0; m < KP; ++m) {
            const float dp = (rp ? dwr[m] : 0.f) + (wp ? db[m] : 0.f);  // d(-alpha ln tau_m)
            dal = fmaf(-dp, w.ltau[m], dal);
            if (m < K)
                acc_tau[m] = fmaf(dp, -w.alpha * (tab ? itab_s[h * K + m] : 1.f / __ldg(a.tau + h * K + m)), acc_tau[m]);
        }
        store_row<T, KP, VEC>(a.dg_read, r, K, dwr);
        store_row<T, KP, VEC>(a.dg_write, r, K, db);
        a.dalpha_raw[r] = (a.flags & FRAC_PREP_ALPHA_ONE) ? 0.f : dal * w.alpha * (1.f - w.alpha);
        const bool pass_dt = w.sp_dt >= a.dt_min && w.sp_dt <= a.dt_max;
        const float gdt = pass_dt ? a.ddt[r] * sigmoid_f(w.pre) : 0.f;
        a.ddt_raw[r] = gdt;
        acc_bias += gdt;
        const bool pass_lam = w.sp_lam >= a.lam_min && w.sp_lam <= a.lam_max;
        a.dlam_raw[r] = pass_lam ? dlam_tot * sigmoid_f(a.lam_raw[r]) : 0.f;
    }
    if (!reduce) return;
    if (shared_slots) {
        if (i < hstride) {
            if (a.ddt_bias) atomicAdd(&red[h * (KP + 1) + KP], acc_bias);
            if (a.dtau) {
#pragma unroll
                for (int m = 0; m < KP; ++m)  // unrolled: the sums stay in registers
                    if (m < K) atomicAdd(&red[h * (KP + 1) + m], acc_tau[m]);
            }
        }
        __syncthreads();
        for (int q = threadIdx.x; q < H * (KP + 1); q += blockDim.x) {
            const int hh = q / (KP + 1), m = q % (KP + 1);
            if (m == KP) {
                if (a.ddt_bias) atomicAdd(a.ddt_bias + hh, red[q]);
            } else if (m < K && a.dtau) {
                atomicAdd(a.dtau + hh * K + m, red[q]);
            }
        }
    } else if (i < hstride) {  // H > blockDim: the block's threads all have different heads
        if (a.ddt_bias) atomicAdd(a.ddt_bias + h, acc_bias);
        if (a.dtau) {
#pragma unroll
            for (int m = 0; m < KP; ++m)
                if (m < K) atomicAdd(a.dtau + h * K + m, acc_tau[m]);
        }
    }
}

int pick_kp(int K) { return K <= 4 ? 4 : K <= 8 ? 8 : K <= 16 ? 16 : 32; }

template <typename T, int KP>
cudaError_t launch_kp(const PrepArgs &a, bool backward, bool vec, cudaStream_t st) {
    const int threads = 256;
    int dev = 0, sms = 152;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t want = (a.n + threads - 1) / threads;
    if (!backward) {  // no sums: one row per thread
        const int blocks = int(std::max<int64_t>(1, std::min<int64_t>(want, int64_t(1) << 30)));
        trace_begin("param_prep_fwd", st);
        if (vec)
            param_prep_fwd_kernel<T, KP, true><<<blocks, threads, 0, st>>>(a);
        else
            param_prep_fwd_kernel<T, KP, false><<<blocks, threads, 0, st>>>(a);
        trace_end(st);
        return cudaGetLastError();
    }
    // the backward's per-block sums end in global atomics: one resident wave of blocks, each
    // walking its rows with a stride of whole head cycles
    const size_t smem = (a.H <= threads) ? size_t(a.H) * (KP + 1) * sizeof(float) : 0;
    int occ = 0;
    if (vec)
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, param_prep_bwd_kernel<T, KP, true>, threads, smem);
    else
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, param_prep_bwd_kernel<T, KP, false>, threads, smem);
    // at least ceil(H / 256) blocks, so that the stride holds one whole head cycle (n >= H rows)
    const int64_t cap = std::max<int64_t>(int64_t(sms) * std::max(occ, 1), (a.H + threads - 1) / threads);
    const int blocks = int(std::max<int64_t>(1, std::min<int64_t>(want, cap)));
    const int64_t total = int64_t(blocks) * threads;
    const int64_t hstride = (total / a.H) * a.H;  // >= H
    trace_begin("param_prep_bwd", st);
    if (vec)
        param_prep_bwd_kernel<T, KP, true><<<blocks, threads, smem, st>>>(a, hstride);
    else
        param_prep_bwd_kernel<T, KP, false><<<blocks, threads, smem, st>>>(a, hstride);
    trace_end(st);
    return cudaGetLastError();
}

template <typename T>
cudaError_t launch_t(const PrepArgs &a, bool backward, bool vec, cudaStream_t st) {
    switch (pick_kp(a.K)) {
        case 4: return launch_kp<T, 4>(a, backward, vec, st);
        case 8: return launch_kp<T, 8>(a, backward, vec, st);
        case 16: return launch_kp<T, 16>(a, backward, vec, st);
        default: return launch_kp<T, 32>(a, backward, vec, st);
    }
}

frac_status prep_fail(frac_status s, const char *msg) {
    set_last_error(msg);
    return s;
}

bool al(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

frac_status prep_check(const frac_dims *d, const frac_prep_config *cfg) {
    if (!d || !cfg) return prep_fail(FRAC_ERR_INVALID_ARGUMENT, "dims and cfg must not be NULL");
    if (d->batch < 1 || d->seqlen < 0 || d->nheads < 1 || d->nmodes < 1 || d->nmodes > 32)
        return prep_fail(FRAC_ERR_INVALID_ARGUMENT,
                         "need batch >= 1, seqlen >= 0, nheads >= 1 and 1 <= nmodes <= 32");
    if (d->dtype != FRAC_DTYPE_F32 && d->dtype != FRAC_DTYPE_BF16)
        return prep_fail(FRAC_ERR_INVALID_ARGUMENT, "unknown dtype");
    if (d->nheads > 65535 || d->batch * d->seqlen > (int64_t(1) << 40))
        return prep_fail(FRAC_ERR_UNSUPPORTED, "dimension too large");
    if (!(cfg->dt_min >= 0.f && cfg->dt_min <= cfg->dt_max && cfg->lam_min >= 0.f &&
          cfg->lam_min <= cfg->lam_max))
        return prep_fail(FRAC_ERR_INVALID_ARGUMENT, "need 0 <= dt_min <= dt_max and 0 <= lam_min <= lam_max");
    if (cfg->flags & ~int32_t(31) || cfg->reserved != 0)
        return prep_fail(FRAC_ERR_INVALID_ARGUMENT, "unknown FRAC_PREP_* flag or nonzero reserved field");
    return FRAC_OK;
}

// 16-byte rows when K * element size is a multiple of 16 and every logit tensor is 16-byte aligned
bool use_vec(const frac_dims *d, std::initializer_list<const void *> ptrs) {
    const size_t es = d->dtype == FRAC_DTYPE_BF16 ? 2 : 4;
    if ((size_t(d->nmodes) * es) % 16 || pick_kp(int(d->nmodes)) != d->nmodes) return false;
    for (const void *p : ptrs)
        if (!al(p, 16)) return false;
    return true;
}

}  // namespace
}  // namespace frac

#define PREP_REQ(p, a)                                                                              \
    do {                                                                                            \
        if (!(p) || !frac::al(p, a)) {                                                              \
            char m_[96];                                                                            \
            std::snprintf(m_, sizeof(m_), "%s must be non-NULL and %d-byte aligned", #p, int(a));   \
            return frac::prep_fail(FRAC_ERR_INVALID_ARGUMENT, m_);                                  \
        }                                                                                           \
    } while (0)

extern "C" {

frac_status frac_param_prep_fwd(const frac_dims *dims, const frac_prep_config *cfg,
                                const float *dt_raw, const float *dt_bias, const float *alpha_raw,
                                const float *lam_raw, const void *g_read, const void *g_write,
                                const float *tau, float *dt, float *alpha, float *lam,
                                void *w_read, void *w_write, void *stream) {
    frac::set_last_error("");
    frac_status s = frac::prep_check(dims, cfg);
    if (s) return s;
    const size_t es = dims->dtype == FRAC_DTYPE_BF16 ? 2 : 4;
    PREP_REQ(tau, 4);
    if (dt_bias && !frac::al(dt_bias, 4)) return frac::prep_fail(FRAC_ERR_INVALID_ARGUMENT, "dt_bias misaligned");
    const int64_t n = dims->batch * dims->seqlen * dims->nheads;
    if (n == 0) return FRAC_OK;
    PREP_REQ(dt_raw, 4); PREP_REQ(lam_raw, 4); PREP_REQ(dt, 4); PREP_REQ(alpha, 4); PREP_REQ(lam, 4);
    if (!(cfg->flags & FRAC_PREP_ALPHA_ONE)) PREP_REQ(alpha_raw, 4);
    PREP_REQ(g_read, es); PREP_REQ(g_write, es); PREP_REQ(w_read, es); PREP_REQ(w_write, es);
    frac::PrepArgs a = {};
    a.n = n; a.H = int(dims->nheads); a.K = int(dims->nmodes); a.flags = cfg->flags;
    a.dt_min = cfg->dt_min; a.dt_max = cfg->dt_max; a.lam_min = cfg->lam_min; a.lam_max = cfg->lam_max;
    a.dt_raw = dt_raw; a.dt_bias = dt_bias; a.alpha_raw = alpha_raw; a.lam_raw = lam_raw; a.tau = tau;
    a.g_read = g_read; a.g_write = g_write;
    a.dt = dt; a.alpha = alpha; a.lam = lam; a.w_read = w_read; a.w_write = w_write;
    const bool vec = frac::use_vec(dims, {g_read, g_write, w_read, w_write});
    cudaStream_t st = (cudaStream_t)stream;
    const cudaError_t e = dims->dtype == FRAC_DTYPE_BF16
                              ? frac::launch_t<__nv_bfloat16>(a, false, vec, st)
                              : frac::launch_t<float>(a, false, vec, st);
    if (e != cudaSuccess) {
        char m[160];
        std::snprintf(m, sizeof(m), "frac_param_prep_fwd: %s", cudaGetErrorString(e));
        return frac::prep_fail(FRAC_ERR_CUDA, m);
    }
    return FRAC_OK;
}

frac_status frac_param_prep_bwd(const frac_dims *dims, const frac_prep_config *cfg,
                                const float *dt_raw, const float *dt_bias, const float *alpha_raw,
                                const float *lam_raw, const void *g_read, const void *g_write,
                                const float *tau, const float *ddt, const float *dalpha,
                                const float *dlam, const void *dw_read, const void *dw_write,
                                float *ddt_raw, float *dalpha_raw, float *dlam_raw, void *dg_read,
                                void *dg_write, float *ddt_bias, float *dtau, void *stream) {
    frac::set_last_error("");
    frac_status s = frac::prep_check(dims, cfg);
    if (s) return s;
    const size_t es = dims->dtype == FRAC_DTYPE_BF16 ? 2 : 4;
    PREP_REQ(tau, 4);
    if ((dt_bias && !frac::al(dt_bias, 4)) || (ddt_bias && !frac::al(ddt_bias, 4)) ||
        (dtau && !frac::al(dtau, 4)))
        return frac::prep_fail(FRAC_ERR_INVALID_ARGUMENT, "dt_bias, ddt_bias or dtau misaligned");
    cudaStream_t st = (cudaStream_t)stream;
    const int H = int(dims->nheads), K = int(dims->nmodes);
    const int64_t n = dims->batch * dims->seqlen * dims->nheads;
    if (n > 0) {  // every check before anything is enqueued
        PREP_REQ(dt_raw, 4); PREP_REQ(lam_raw, 4); PREP_REQ(ddt, 4); PREP_REQ(dalpha, 4);
        PREP_REQ(dlam, 4); PREP_REQ(ddt_raw, 4); PREP_REQ(dalpha_raw, 4); PREP_REQ(dlam_raw, 4);
        if (!(cfg->flags & FRAC_PREP_ALPHA_ONE)) PREP_REQ(alpha_raw, 4);
        PREP_REQ(g_read, es); PREP_REQ(g_write, es); PREP_REQ(dw_read, es); PREP_REQ(dw_write, es);
        PREP_REQ(dg_read, es); PREP_REQ(dg_write, es);
    }
    cudaError_t e = cudaSuccess;
    if (ddt_bias) e = cudaMemsetAsync(ddt_bias, 0, sizeof(float) * H, st);
    if (e == cudaSuccess && dtau) e = cudaMemsetAsync(dtau, 0, sizeof(float) * H * K, st);
    if (e == cudaSuccess && n > 0) {
        frac::PrepArgs a = {};
        a.n = n; a.H = H; a.K = K; a.flags = cfg->flags;
        a.dt_min = cfg->dt_min; a.dt_max = cfg->dt_max; a.lam_min = cfg->lam_min; a.lam_max = cfg->lam_max;
        a.dt_raw = dt_raw; a.dt_bias = dt_bias; a.alpha_raw = alpha_raw; a.lam_raw = lam_raw; a.tau = tau;
        a.g_read = g_read; a.g_write = g_write;
        a.ddt = ddt; a.dalpha = dalpha; a.dlam = dlam; a.dw_read = dw_read; a.dw_write = dw_write;
        a.ddt_raw = ddt_raw; a.dalpha_raw = dalpha_raw; a.dlam_raw = dlam_raw;
        a.dg_read = dg_read; a.dg_write = dg_write; a.ddt_bias = ddt_bias; a.dtau = dtau;
        const bool vec = frac::use_vec(dims, {g_read, g_write, dw_read, dw_write, dg_read, dg_write});
        e = dims->dtype == FRAC_DTYPE_BF16 ? frac::launch_t<__nv_bfloat16>(a, true, vec, st)
                                           : frac::launch_t<float>(a, true, vec, st);
    }
    if (e != cudaSuccess) {
        char m[160];
        std::snprintf(m, sizeof(m), "frac_param_prep_bwd: %s", cudaGetErrorString(e));
        return frac::prep_fail(FRAC_ERR_CUDA, m);
    }
    return FRAC_OK;
}

}  // extern "C"
