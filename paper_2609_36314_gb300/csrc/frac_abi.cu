// C ABI of the Frac scan library: argument validation, workspace layout, path selection.
// Every check happens before anything is enqueued; kernels live in the other files.
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

// Path selection and the dims the kernels see.
frac_status plan(const frac_dims *d, frac::ScanDims *sd) {
    sd->B = int(d->batch);
    sd->L = int(d->seqlen);
    sd->H = int(d->nheads);
    sd->P = int(d->headdim);
    sd->G = int(d->ngroups);
    sd->N = int(d->dstate);
    sd->K = int(d->nmodes);
    const int Q = frac::simt_pick_chunk(*sd, int(d->chunk));
    if (Q == 0)
        return fail(FRAC_ERR_UNSUPPORTED,
                    "no chunk size fits these dims on the CUDA-core path (chunk=%lld, P=%d, N=%d, K=%d)",
                    (long long)d->chunk, sd->P, sd->N, sd->K);
    sd->Q = Q;
    sd->nc = (sd->L + Q - 1) / Q;
    return FRAC_OK;
}

struct FwdLayout {
    size_t s_in, total;
};
struct BwdLayout {
    size_t s_in, ds_out, db, dc, total;
};

FwdLayout fwd_layout(const frac_dims *d, const frac::ScanDims &sd) {
    FwdLayout l;
    l.s_in = 0;
    l.total = round_up(frac::simt_state_elems(sd) * elem(d));
    return l;
}

BwdLayout bwd_layout(const frac_dims *d, const frac::ScanDims &sd) {
    BwdLayout l;
    const size_t st = round_up(frac::simt_state_elems(sd) * elem(d));
    const size_t ngn = size_t(sd.B) * sd.L * sd.G * sd.N;
    l.s_in = 0;
    l.ds_out = st;
    l.db = 2 * st;
    const size_t acc = (d->dtype == FRAC_DTYPE_BF16) ? round_up(ngn * sizeof(float)) : 0;
    l.dc = l.db + acc;
    l.total = l.dc + acc;
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

frac_status frac_scan_fwd_workspace_size(const frac_dims *d, size_t *bytes) {
    g_err[0] = 0;
    frac_status s = check_dims(d, true);
    if (s) return s;
    if (!bytes) return fail(FRAC_ERR_INVALID_ARGUMENT, "bytes must not be NULL");
    frac::ScanDims sd;
    if ((s = plan(d, &sd))) return s;
    *bytes = fwd_layout(d, sd).total;
    return FRAC_OK;
}

frac_status frac_scan_bwd_workspace_size(const frac_dims *d, size_t *bytes) {
    g_err[0] = 0;
    frac_status s = check_dims(d, true);
    if (s) return s;
    if (!bytes) return fail(FRAC_ERR_INVALID_ARGUMENT, "bytes must not be NULL");
    frac::ScanDims sd;
    if ((s = plan(d, &sd))) return s;
    *bytes = bwd_layout(d, sd).total;
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
    if ((s = plan(d, &sd))) return s;
    const FwdLayout l = fwd_layout(d, sd);
    if (l.total > 0) {
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
    return cuda_status(frac::simt_scan_fwd(sd, d->dtype, p, ws + l.s_in, (cudaStream_t)stream),
                       "frac_scan_fwd");
}

frac_status frac_scan_bwd(const frac_dims *d, const void *x, const float *dt, const float *alpha,
                          const float *lam, const float *tau, const void *Bm, const void *Cm,
                          const void *w_read, const void *w_write, const float *D,
                          const float *h0, const void *dy, const float *dh_final, void *dx,
                          float *ddt, float *dalpha, float *dlam, void *dB, void *dC,
                          void *dw_read, void *dw_write, float *dD, float *dh0, void *workspace,
                          size_t workspace_bytes, void *stream) {
    g_err[0] = 0;
    frac_status s = check_dims(d, true);
    if (s) return s;
    REQUIRE_PTR(tau);
    REQUIRE_PTR(D);
    REQUIRE_PTR(dD);
    OPTIONAL_PTR(h0);
    OPTIONAL_PTR(dh_final);
    OPTIONAL_PTR(dh0);
    if (d->seqlen > 0) {
        REQUIRE_T(x); REQUIRE_PTR(dt); REQUIRE_PTR(alpha); REQUIRE_PTR(lam);
        REQUIRE_T(Bm); REQUIRE_T(Cm); REQUIRE_T(w_read); REQUIRE_T(w_write);
        REQUIRE_T(dy); REQUIRE_T(dx); REQUIRE_PTR(ddt); REQUIRE_PTR(dalpha);
        REQUIRE_PTR(dlam); REQUIRE_T(dB); REQUIRE_T(dC); REQUIRE_T(dw_read);
        REQUIRE_T(dw_write);
    }
    frac::ScanDims sd;
    if ((s = plan(d, &sd))) return s;
    const BwdLayout l = bwd_layout(d, sd);
    if (l.total > 0) {
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
    p.ddt = ddt; p.dalpha = dalpha; p.dlam = dlam; p.dD = dD; p.dh0 = dh0;
    char *ws = static_cast<char *>(workspace);
    float *dB_acc = d->dtype == FRAC_DTYPE_BF16 ? reinterpret_cast<float *>(ws + l.db)
                                                : static_cast<float *>(dB);
    float *dC_acc = d->dtype == FRAC_DTYPE_BF16 ? reinterpret_cast<float *>(ws + l.dc)
                                                : static_cast<float *>(dC);
    return cuda_status(frac::simt_scan_bwd(sd, d->dtype, p, ws + l.s_in, ws + l.ds_out, dB_acc,
                                           dC_acc, (cudaStream_t)stream),
                       "frac_scan_bwd");
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
