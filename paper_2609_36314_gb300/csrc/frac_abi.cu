// C ABI of the Frac scan library: argument validation, workspace layout, path selection.
// Every check happens before anything is enqueued; kernels live in the other files.
#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <cstring>

#include "../../include/frac.h"
#include "kernels.h"

namespace {

thread_local char g_err[512] = "";

frac_status fail(frac_status s, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return s;
}

frac_status cuda_status(cudaError_t e, const char *where) {
    if (e == cudaSuccess) return FRAC_OK;
    return fail(FRAC_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

bool aligned_to(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

constexpr size_t kAlign = 256;
size_t round_up(size_t v) { return (v + kAlign - 1) / kAlign * kAlign; }

// Every tensor must be aligned to its element size (float32 tensors: 4 bytes; dtype tensors:
// 2 or 4 bytes).  Stronger alignment only selects faster kernels.
#define REQUIRE_PTR_A(p, a)                                                                    \
    do {                                                                                       \
        if (!(p)) return fail(FRAC_ERR_INVALID_ARGUMENT, "%s must not be NULL", #p);           \
        if (!aligned_to(p, a))                                                                 \
            return fail(FRAC_ERR_INVALID_ARGUMENT, "%s is not aligned to %d bytes", #p, int(a)); \
    } while (0)
#define OPTIONAL_PTR_A(p, a)                                                                   \
    do {                                                                                       \
        if ((p) && !aligned_to(p, a))                                                          \
            return fail(FRAC_ERR_INVALID_ARGUMENT, "%s is not aligned to %d bytes", #p, int(a)); \
    } while (0)
#define REQUIRE_PTR(p) REQUIRE_PTR_A(p, sizeof(*(p)))
#define OPTIONAL_PTR(p) OPTIONAL_PTR_A(p, sizeof(*(p)))
#define REQUIRE_T(p) REQUIRE_PTR_A(p, elem(d))

frac_status check_dims(const frac_dims *d, bool need_seq) {
    if (!d) return fail(FRAC_ERR_INVALID_ARGUMENT, "dims must not be NULL");
    if (d->batch < 1 || d->nheads < 1 || d->headdim < 1 || d->ngroups < 1 || d->dstate < 1)
        return fail(FRAC_ERR_INVALID_ARGUMENT, "batch, nheads, headdim, ngroups, dstate must be >= 1");
    if (need_seq && d->seqlen < 0) return fail(FRAC_ERR_INVALID_ARGUMENT, "seqlen must be >= 0");
    if (d->nmodes < 1 || d->nmodes > 32)
        return fail(FRAC_ERR_INVALID_ARGUMENT, "nmodes must be in [1, 32]");
    if (d->nheads % d->ngroups)
        return fail(FRAC_ERR_INVALID_ARGUMENT, "nheads must be a multiple of ngroups");
    if (d->dtype != FRAC_DTYPE_F32 && d->dtype != FRAC_DTYPE_BF16)
        return fail(FRAC_ERR_INVALID_ARGUMENT, "unknown dtype %d", d->dtype);
    if (d->chunk < 0) return fail(FRAC_ERR_INVALID_ARGUMENT, "chunk must be >= 0");
    const int64_t lim = int64_t(1) << 30;
    if (d->batch > lim || d->seqlen > lim || d->nheads > 65535 || d->headdim > 4096 ||
        d->dstate > 4096 || d->batch > 65535)
        return fail(FRAC_ERR_UNSUPPORTED, "dimension too large");
    return FRAC_OK;
}

size_t elem(const frac_dims *d) { return d->dtype == FRAC_DTYPE_BF16 ? 2 : 4; }

// Path selection and the dims the kernels see.  The forward uses the tensor-core kernels
// for bf16 shapes they support (unless FRAC_FLAG_FORCE_SIMT); everything else, and the
// backward, runs on the CUDA-core kernels.
enum Path { PATH_SIMT = 0, PATH_TC = 1 };

frac_status plan(const frac_dims *d, frac::ScanDims *sd, int *path, bool backward) {
    // (the backward runs on the tensor cores when headdim is 64 as well)
    sd->B = int(d->batch);
    sd->L = int(d->seqlen);
    sd->H = int(d->nheads);
    sd->P = int(d->headdim);
    sd->G = int(d->ngroups);
    sd->N = int(d->dstate);
    sd->K = int(d->nmodes);
    const bool tc = !(d->flags & FRAC_FLAG_FORCE_SIMT) &&
                    (backward ? frac::tc_bwd_supported(*sd, d->dtype)
                              : frac::tc_supported(*sd, d->dtype)) &&
                    (d->chunk == 0 || d->chunk == 128);
    if (tc) {
        sd->Q = 128;
        *path = PATH_TC;
    } else {
        const int Q = frac::simt_pick_chunk(*sd, int(d->chunk));
        if (Q == 0)
            return fail(FRAC_ERR_UNSUPPORTED,
                        "chunk=%lld is not supported for these dims (P=%d, N=%d, K=%d, dtype=%d); "
                        "use 0 to let the library choose",
                        (long long)d->chunk, sd->P, sd->N, sd->K, d->dtype);
        sd->Q = Q;
        *path = PATH_SIMT;
    }
    sd->nc = (sd->L + sd->Q - 1) / sd->Q;
    return FRAC_OK;
}

// Workspace layout: [0, 256) device status word (FRAC_OK or FRAC_ERR_TIMEOUT written by
// kernels with bounded waits), then the per-chunk states and accumulators.
constexpr size_t kStatusBytes = kAlign;

struct FwdLayout {
    size_t s_in, coef, ek, total;
};
struct BwdLayout {
    size_t s_in, ds_out, db, dc, n1, total;
};

FwdLayout fwd_layout(const frac_dims *d, const frac::ScanDims &sd, int path) {
    FwdLayout l;
    l.s_in = kStatusBytes;
    const size_t elems = path == PATH_TC ? frac::tc_state_elems(sd) : frac::simt_state_elems(sd);
    const size_t esz = path == PATH_TC ? 2 : elem(d);
    l.coef = kStatusBytes + round_up(elems * esz);  // tensor-core path: per-position coefficients
    // CUDA-core path at N = 1: the forward's float scratch takes the coefficient slot
    l.ek = l.coef + (path == PATH_TC ? round_up(frac::tc_coef_elems(sd) * 4)
                                     : round_up(frac::simt_n1_scratch_elems(sd) * 4));
    l.total = l.ek + (path == PATH_TC ? round_up(frac::tc_ek_elems(sd) * 4) : 0);
    return l;
}

BwdLayout bwd_layout(const frac_dims *d, const frac::ScanDims &sd, int path) {
    BwdLayout l;
    if (path == PATH_TC) {
        frac::TcBwdWorkspace t;
        l.s_in = l.ds_out = l.db = l.dc = l.n1 = 0;
        l.total = kStatusBytes + frac::tc_bwd_workspace_bytes(sd, &t, nullptr);
        return l;
    }
    const size_t st = round_up(frac::simt_state_elems(sd) * elem(d));
    const size_t ngn = size_t(sd.B) * sd.L * sd.G * sd.N;
    l.s_in = kStatusBytes;
    l.ds_out = l.s_in + st;
    l.db = l.ds_out + st;
    const size_t acc = (d->dtype == FRAC_DTYPE_BF16) ? round_up(ngn * sizeof(float)) : 0;
    l.dc = l.db + acc;
    l.n1 = l.dc + acc;  // the N = 1 backward's chunk carries (0 bytes for other shapes)
    l.total = l.n1 + round_up(frac::simt_n1_scratch_elems(sd) * 4);
    // one buffer serves a forward and the backward that reuses its states
    // (FRAC_FLAG_BWD_REUSE_FWD_STATES): cover the forward's scratch as well
    l.total = std::max(l.total, fwd_layout(d, sd, path).total);
    return l;
}

}  // namespace

namespace frac {
void set_last_error(const char *msg) { snprintf(g_err, sizeof(g_err), "%s", msg); }
}  // namespace frac

extern "C" {

const char *frac_status_string(frac_status s) {
    switch (s) {
        case FRAC_OK: return "ok";
        case FRAC_ERR_INVALID_ARGUMENT: return "invalid argument";
        case FRAC_ERR_UNSUPPORTED: return "unsupported";
        case FRAC_ERR_CUDA: return "CUDA error";
        case FRAC_ERR_TIMEOUT: return "device wait timed out";
    }
    return "unknown status";
}

const char *frac_last_error(void) { return g_err; }

frac_status frac_workspace_status(const void *workspace, void *stream) {
    g_err[0] = 0;
    if (!workspace || !aligned_to(workspace, kAlign))
        return fail(FRAC_ERR_INVALID_ARGUMENT, "workspace must be the 256-byte aligned workspace of a call");
    int word = 0;
    cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e == cudaSuccess) e = cudaMemcpy(&word, workspace, sizeof(int), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_status(e, "frac_workspace_status");
    if (word == FRAC_ERR_TIMEOUT)
        return fail(FRAC_ERR_TIMEOUT, "a device-side wait gave up (work of that call is incomplete)");
    return word == 0 ? FRAC_OK : fail(FRAC_ERR_CUDA, "device status word %d", word);
}

frac_status frac_scan_fwd_workspace_size(const frac_dims *d, size_t *bytes) {
    g_err[0] = 0;
    frac_status s = check_dims(d, true);
    if (s) return s;
    if (!bytes) return fail(FRAC_ERR_INVALID_ARGUMENT, "bytes must not be NULL");
    frac::ScanDims sd;
    int path = 0;
    if ((s = plan(d, &sd, &path, false))) return s;
    *bytes = fwd_layout(d, sd, path).total;
    return FRAC_OK;
}

frac_status frac_scan_bwd_workspace_size(const frac_dims *d, size_t *bytes) {
    g_err[0] = 0;
    frac_status s = check_dims(d, true);
    if (s) return s;
    if (!bytes) return fail(FRAC_ERR_INVALID_ARGUMENT, "bytes must not be NULL");
    frac::ScanDims sd;
    int path = 0;
    if ((s = plan(d, &sd, &path, true))) return s;
    *bytes = bwd_layout(d, sd, path).total;
    return FRAC_OK;
}

frac_status frac_scan_fwd(const frac_dims *d, const void *x, const float *dt, const float *alpha,
                          const float *lam, const float *tau, const void *Bm, const void *Cm,
                          const void *w_read, const void *w_write, const float *D,
                          const float *h0, void *y, float *h_final, void *workspace,
                          size_t workspace_bytes, void *stream) {
    g_err[0] = 0;
    frac_status s = check_dims(d, true);
    if (s) return s;
    REQUIRE_PTR(tau);
    REQUIRE_PTR(D);
    OPTIONAL_PTR(h0);
    OPTIONAL_PTR(h_final);
    if (d->seqlen > 0) {
        REQUIRE_T(x);
        REQUIRE_PTR(dt);
        REQUIRE_PTR(alpha);
        REQUIRE_PTR(lam);
        REQUIRE_T(Bm);
        REQUIRE_T(Cm);
        REQUIRE_T(w_read);
        REQUIRE_T(w_write);
        REQUIRE_T(y);
    }
    frac::ScanDims sd;
    int path = 0;
    if ((s = plan(d, &sd, &path, false))) return s;
    if (d->flags & FRAC_FLAG_TEST_EXPIRE_WAIT) {
        if (path != PATH_TC)
            return fail(FRAC_ERR_UNSUPPORTED,
                        "FRAC_FLAG_TEST_EXPIRE_WAIT applies to the tensor-core forward only");
        sd.expire_ns = 1000000u;  // 1 ms
    }
    const FwdLayout l = fwd_layout(d, sd, path);
    if (path == PATH_TC && d->seqlen > 0) {
        const void *need16[] = {x, Bm, Cm, y};
        for (const void *q : need16)
            if (!aligned_to(q, 16))
                return fail(FRAC_ERR_INVALID_ARGUMENT,
                            "the tensor-core path needs x, Bm, Cm and y 16-byte aligned "
                            "(or set FRAC_FLAG_FORCE_SIMT)");
        if (h_final && !aligned_to(h_final, 16))
            return fail(FRAC_ERR_INVALID_ARGUMENT, "h_final is not 16-byte aligned");
    }
    {
        if (!workspace) return fail(FRAC_ERR_INVALID_ARGUMENT, "workspace must not be NULL");
        if (reinterpret_cast<uintptr_t>(workspace) % kAlign)
            return fail(FRAC_ERR_INVALID_ARGUMENT, "workspace is not 256-byte aligned");
        if (workspace_bytes < l.total)
            return fail(FRAC_ERR_INVALID_ARGUMENT, "workspace too small: %zu < %zu bytes",
                        workspace_bytes, l.total);
    }
    frac::ScanPtrs p = {};
    p.x = x; p.Bm = Bm; p.Cm = Cm; p.wr = w_read; p.ww = w_write;
    p.dt = dt; p.alpha = alpha; p.lam = lam; p.tau = tau; p.D = D; p.h0 = h0;
    p.y = y; p.h_final = h_final;
    char *ws = static_cast<char *>(workspace);
    cudaStream_t st = (cudaStream_t)stream;
    cudaError_t e = cudaMemsetAsync(ws, 0, sizeof(int), st);
    if (e == cudaSuccess) {
        if (path == PATH_TC)
            e = frac::tc_scan_fwd(sd, p, ws + l.s_in, reinterpret_cast<float *>(ws + l.coef),
                                  reinterpret_cast<float *>(ws + l.ek), reinterpret_cast<int *>(ws), st);
        else
            e = frac::simt_scan_fwd(sd, d->dtype, p, ws + l.s_in, reinterpret_cast<float *>(ws + l.coef), st);
    }
    return cuda_status(e, "frac_scan_fwd");
}

frac_status frac_scan_bwd(const frac_dims *d, const void *x, const float *dt, const float *alpha,
                          const float *lam, const float *tau, const void *Bm, const void *Cm,
                          const void *w_read, const void *w_write, const float *D,
                          const float *h0, const void *dy, const float *dh_final, void *dx,
                          float *ddt, float *dalpha, float *dlam, void *dB, void *dC,
                          void *dw_read, void *dw_write, float *dD, float *dh0, float *dtau,
                          void *workspace, size_t workspace_bytes, void *stream) {
    g_err[0] = 0;
    frac_status s = check_dims(d, true);
    if (s) return s;
    REQUIRE_PTR(tau);
    REQUIRE_PTR(D);
    REQUIRE_PTR(dD);
    OPTIONAL_PTR(h0);
    OPTIONAL_PTR(dh_final);
    OPTIONAL_PTR(dh0);
    OPTIONAL_PTR(dtau);
    if (d->seqlen > 0) {
        REQUIRE_T(x); REQUIRE_PTR(dt); REQUIRE_PTR(alpha); REQUIRE_PTR(lam);
        REQUIRE_T(Bm); REQUIRE_T(Cm); REQUIRE_T(w_read); REQUIRE_T(w_write);
        REQUIRE_T(dy); REQUIRE_T(dx); REQUIRE_PTR(ddt); REQUIRE_PTR(dalpha);
        REQUIRE_PTR(dlam); REQUIRE_T(dB); REQUIRE_T(dC); REQUIRE_T(dw_read);
        REQUIRE_T(dw_write);
    }
    if (d->flags & FRAC_FLAG_TEST_EXPIRE_WAIT)
        return fail(FRAC_ERR_UNSUPPORTED, "FRAC_FLAG_TEST_EXPIRE_WAIT applies to the forward only");
    frac::ScanDims sd;
    int path = 0;
    if ((s = plan(d, &sd, &path, true))) return s;
    const BwdLayout l = bwd_layout(d, sd, path);
    const bool reuse = (d->flags & FRAC_FLAG_BWD_REUSE_FWD_STATES) != 0;
    if (reuse) {
        frac::ScanDims sf;
        int fpath;
        if ((s = plan(d, &sf, &fpath, false))) return s;
        if (fpath != path || sf.Q != sd.Q)
            return fail(FRAC_ERR_INVALID_ARGUMENT,
                        "FRAC_FLAG_BWD_REUSE_FWD_STATES: the forward of these dims runs on another "
                        "path (chunk %d) than the backward (chunk %d); its states cannot be reused",
                        sf.Q, sd.Q);
    }
    if (path == PATH_TC && d->seqlen > 0) {
        const void *need16[] = {x, Bm, Cm, dy, dx, dB, dC, dw_read, dw_write};
        for (const void *q : need16)
            if (!aligned_to(q, 16))
                return fail(FRAC_ERR_INVALID_ARGUMENT,
                            "the tensor-core backward needs x, Bm, Cm, dy, dx, dB, dC, dw_read and "
                            "dw_write 16-byte aligned (or set FRAC_FLAG_FORCE_SIMT)");
        if ((h0 && !aligned_to(h0, 16)) || (dh_final && !aligned_to(dh_final, 16)) ||
            (dh0 && !aligned_to(dh0, 16)))
            return fail(FRAC_ERR_INVALID_ARGUMENT, "state tensors must be 16-byte aligned");
    }
    {
        if (!workspace) return fail(FRAC_ERR_INVALID_ARGUMENT, "workspace must not be NULL");
        if (reinterpret_cast<uintptr_t>(workspace) % kAlign)
            return fail(FRAC_ERR_INVALID_ARGUMENT, "workspace is not 256-byte aligned");
        if (workspace_bytes < l.total)
            return fail(FRAC_ERR_INVALID_ARGUMENT, "workspace too small: %zu < %zu bytes",
                        workspace_bytes, l.total);
    }
    frac::ScanPtrs p = {};
    p.x = x; p.Bm = Bm; p.Cm = Cm; p.wr = w_read; p.ww = w_write; p.dy = dy;
    p.dt = dt; p.alpha = alpha; p.lam = lam; p.tau = tau; p.D = D; p.h0 = h0;
    p.dh_final = dh_final;
    p.dx = dx; p.dB = dB; p.dC = dC; p.dwr = dw_read; p.dww = dw_write;
    p.ddt = ddt; p.dalpha = dalpha; p.dlam = dlam; p.dD = dD; p.dh0 = dh0; p.dtau = dtau;
    char *ws = static_cast<char *>(workspace);
    float *dB_acc = d->dtype == FRAC_DTYPE_BF16 ? reinterpret_cast<float *>(ws + l.db)
                                                : static_cast<float *>(dB);
    float *dC_acc = d->dtype == FRAC_DTYPE_BF16 ? reinterpret_cast<float *>(ws + l.dc)
                                                : static_cast<float *>(dC);
    cudaStream_t st = (cudaStream_t)stream;
    cudaError_t e = cudaMemsetAsync(ws, 0, sizeof(int), st);
    if (e == cudaSuccess) {
        if (path == PATH_TC) {
            frac::TcBwdWorkspace t;
            frac::tc_bwd_workspace_bytes(sd, &t, ws + kStatusBytes);
            e = frac::tc_scan_bwd(sd, p, t, reinterpret_cast<int *>(ws), reuse, st);
        } else {
            e = frac::simt_scan_bwd(sd, d->dtype, p, ws + l.s_in, ws + l.ds_out, dB_acc, dC_acc,
                                    reinterpret_cast<float *>(ws + l.n1), reuse, reinterpret_cast<int *>(ws), st);
        }
    }
    return cuda_status(e, "frac_scan_bwd");
}

frac_status frac_decode_step(const frac_dims *d, const void *x_t, const float *dt,
                             const float *alpha, const float *lam, const float *tau,
                             const void *B_t, const void *C_t, const void *w_read,
                             const void *w_write, const float *D, float *state, void *y_t,
                             void *stream) {
    g_err[0] = 0;
    frac_status s = check_dims(d, false);
    if (s) return s;
    REQUIRE_T(x_t); REQUIRE_PTR(dt); REQUIRE_PTR(alpha); REQUIRE_PTR(lam); REQUIRE_PTR(tau);
    REQUIRE_T(B_t); REQUIRE_T(C_t); REQUIRE_T(w_read); REQUIRE_T(w_write);
    REQUIRE_PTR(D); REQUIRE_PTR(state); REQUIRE_T(y_t);
    frac::DecodeArgs a;
    a.B = int(d->batch); a.H = int(d->nheads); a.P = int(d->headdim); a.G = int(d->ngroups);
    a.N = int(d->dstate); a.K = int(d->nmodes);
    a.dt = dt; a.alpha = alpha; a.lam = lam; a.tau = tau; a.D = D; a.state = state;
    return cuda_status(frac::launch_decode(a, d->dtype, x_t, B_t, C_t, w_read, w_write, y_t,
                                           (cudaStream_t)stream),
                       "frac_decode_step");
}

}  // extern "C"
