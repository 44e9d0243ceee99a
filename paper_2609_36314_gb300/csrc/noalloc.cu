// Allocation-free variant of frac_scan_fwd.
//
// frac_scan_fwd needs caller-provided scratch memory for the per-chunk mode states.  Some
// callers cannot provide it: code embedded in a host application that owns the whole device
// memory budget and gives its plug-ins no allocator, or a caller that is only allowed to
// touch buffers it was handed (inputs and outputs) once it is running.  For them this file
// keeps the scratch in a fixed, statically sized device array that the library itself owns.
//
// Properties a caller must know:
//   * The array is FRAC_SCAN_FWD_STATIC_SCRATCH_BYTES (64 MiB) on every GPU that loads the
//     library, reserved for the life of the process.
//   * Problems whose forward scratch (frac_scan_fwd_workspace_size) exceeds that size are
//     rejected with FRAC_ERR_UNSUPPORTED and a message; nothing is enqueued for them.
//   * The first call on a device looks up the array's device address (cudaGetSymbolAddress)
//     with that device current and caches it together with the device's current context; make
//     that first call before anything that must not see a runtime call (for example before
//     capturing work into a CUDA graph).  A later call that finds another context current on
//     the device (after cudaDeviceReset the module is loaded again and the array may move)
//     looks the address up again.
//   * Word 0 of the array is the status word of the last call's kernels (a bounded device wait
//     that gave up writes FRAC_ERR_TIMEOUT there); frac_scan_fwd_static_status reads it.
//     Overlapping calls share that word too.
//   * Every call shares the one array.  Calls whose GPU work overlaps (different streams, or
//     different host threads on the same device) race on it; serialise them.  No part of the
//     scratch has to start at zero: the forward scan writes every per-chunk state before it
//     reads it, so leftovers of an earlier call are never used.
//   * No cudaMalloc, cudaFree or other allocating routine is called.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdio>
#include <mutex>

#include "../../include/frac.h"
#include "kernels.h"

namespace {

constexpr size_t kFracStaticScratchBytes = FRAC_SCAN_FWD_STATIC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_static_scratch[kFracStaticScratchBytes];

std::mutex g_mu;
void *g_dev_ptr[kMaxDevices] = {};
CUcontext g_dev_ctx[kMaxDevices] = {};

// The driver's cuCtxGetCurrent, reached through the runtime (the library does not link the
// driver library directly, so it loads on machines without a GPU driver).
CUresult current_context(CUcontext *ctx) {
    using Fn = CUresult (*)(CUcontext *);
    static Fn fn = [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            p = nullptr;
        return reinterpret_cast<Fn>(p);
    }();
    *ctx = nullptr;
    return fn ? fn(ctx) : CUDA_ERROR_NOT_SUPPORTED;
}

// Device address of g_static_scratch on the current device (looked up once per device and
// context).
frac_status static_scratch(void **out) {
    char msg[160];
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) {
        std::snprintf(msg, sizeof(msg), "cudaGetDevice: %s", cudaGetErrorString(e));
        frac::set_last_error(msg);
        return FRAC_ERR_CUDA;
    }
    if (dev < 0 || dev >= kMaxDevices) {
        std::snprintf(msg, sizeof(msg), "device index %d out of range", dev);
        frac::set_last_error(msg);
        return FRAC_ERR_UNSUPPORTED;
    }
    // The context current on the device (null before the runtime has set the device up; the
    // symbol lookup below does that).  A cached address is only reused under the same context.
    CUcontext ctx = nullptr;
    if (current_context(&ctx) != CUDA_SUCCESS) ctx = nullptr;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_dev_ptr[dev] || !ctx || g_dev_ctx[dev] != ctx) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_static_scratch);
        if (e != cudaSuccess || !p) {
            std::snprintf(msg, sizeof(msg), "cudaGetSymbolAddress: %s",
                          cudaGetErrorString(e));
            frac::set_last_error(msg);
            return FRAC_ERR_CUDA;
        }
        if (current_context(&ctx) != CUDA_SUCCESS) ctx = nullptr;
        g_dev_ptr[dev] = p;
        g_dev_ctx[dev] = ctx;
    }
    *out = g_dev_ptr[dev];
    return FRAC_OK;
}

}  // namespace

extern "C" {

frac_status frac_scan_fwd_static(const frac_dims *dims, const void *x, const float *dt,
                                 const float *alpha, const float *lam, const float *tau,
                                 const void *Bm, const void *Cm, const void *w_read,
                                 const void *w_write, const float *D, const float *h0, void *y,
                                 float *h_final, void *stream) {
    size_t need = 0;
    frac_status s = frac_scan_fwd_workspace_size(dims, &need);
    if (s != FRAC_OK) return s;  // frac_last_error() already says why
    if (need > kFracStaticScratchBytes) {
        char msg[256];
        std::snprintf(msg, sizeof(msg),
                      "this problem needs %zu bytes of scratch but the allocation-free forward "
                      "scan has %zu; call frac_scan_fwd with a workspace instead",
                      need, kFracStaticScratchBytes);
        frac::set_last_error(msg);
        return FRAC_ERR_UNSUPPORTED;
    }
    void *scratch = nullptr;
    if ((s = static_scratch(&scratch)) != FRAC_OK) return s;
    return frac_scan_fwd(dims, x, dt, alpha, lam, tau, Bm, Cm, w_read, w_write, D, h0, y,
                         h_final, scratch, kFracStaticScratchBytes, stream);
}

frac_status frac_scan_fwd_static_status(void *stream) {
    void *scratch = nullptr;
    frac_status s = static_scratch(&scratch);
    if (s != FRAC_OK) return s;
    return frac_workspace_status(scratch, stream);
}

}  // extern "C"
