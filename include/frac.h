/*
 * frac.h -- C ABI of the GB300 (sm_103a) Frac selective fractional state-space scan.
 *
 * The layer (arXiv 2609.36314, Sec. 3.2 and Algorithm 1 of App. D), with the mode
 * state lifted to an N-dimensional outer product per head (N = 1, B = C = 1 is
 * Algorithm 1 itself):
 *
 *   e_t        = Delta_t * lambda_t^(1/alpha_t)                (Eq. tau-eff: tau~ = tau / lambda^(1/alpha))
 *   rho_{t,m}  = exp(-e_t / tau_m)                             (Eq. rho-beta-def-frac)
 *   kappa_{t,m}= (1 - rho_{t,m}) * w_write_{t,m}               (Algorithm 1 steps 3 and 6; the remark after it)
 *   S_{t,m}    = rho_{t,m} S_{t-1,m} + kappa_{t,m} x_t B_t^T   (Eq. frac-selective-update; S_{t,m} is P x N)
 *   y_t        = sum_m w_read_{t,m} S_{t,m} C_t + D x_t        (Eq. frac-readout; skip D u_t of Sec. 3.3)
 *
 * w_read / w_write are the already-normalised read and write mode weights of
 * Eq. read-softmax (computed upstream).  Head h reads B/C group g = h / (H / G).
 *
 * Conventions shared by every entry point
 *   - Tensor arguments are device pointers owned by the caller, row-major and contiguous,
 *     aligned at least to their element size, and must not alias each other (except where
 *     stated).  16-byte alignment of every tensor lets the library pick its vectorised and
 *     TMA-fed kernels; otherwise it uses kernels with scalar accesses.  The library
 *     allocates no device memory in any call; the only device memory it owns is the fixed
 *     scratch array of frac_scan_fwd_static (a static device array of the module).  Between
 *     calls it keeps a thread-local error message, the launch trace when tracing is on, and
 *     the cached address of that array.
 *   - `stream` is a cudaStream_t (NULL = the legacy default stream).  Every call only
 *     enqueues work on `stream`; results are valid once the stream has completed.
 *   - Element types: x, B, C, w_read, w_write, y and their gradients use `dims->dtype`
 *     (FRAC_DTYPE_F32 or FRAC_DTYPE_BF16).  Delta, alpha, lambda, tau, D, all mode states
 *     (h0, h_final, state, dh_final, dh0) and the gradients of Delta, alpha, lambda, D are
 *     always float32.  Arithmetic is float32 (tensor-core products take bf16 operands with
 *     float32 accumulation on the bf16 path).
 *   - Controls must satisfy Delta > 0, 0 < alpha <= 1, lambda > 0, tau > 0.  e_t is clamped
 *     to 64 * max_m tau_{h,m} (every mode's retention is then <= e^-64); the gradient of a
 *     clamped e_t is zero.
 *   - Return values: FRAC_OK, or FRAC_ERR_INVALID_ARGUMENT (bad dims, NULL or misaligned
 *     pointer, workspace too small) and FRAC_ERR_UNSUPPORTED (a shape the kernels do not
 *     handle) before anything is enqueued, or FRAC_ERR_CUDA if a launch failed.
 *     frac_last_error() then holds a readable reason for the calling thread.
 *
 * Layouts
 *   x, y, dy, dx             [batch, seqlen, nheads, headdim]
 *   dt, alpha, lam (+grads)  [batch, seqlen, nheads]               float32
 *   Bm, Cm (+grads)          [batch, seqlen, ngroups, dstate]
 *   w_read, w_write (+grads) [batch, seqlen, nheads, nmodes]
 *   tau                      [nheads, nmodes]                       float32
 *   D, dD                    [nheads]                               float32
 *   h0, h_final, dh_final, dh0, state   [batch, nheads, nmodes, headdim, dstate]   float32
 */
#ifndef FRAC_H_
#define FRAC_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    FRAC_OK = 0,
    FRAC_ERR_INVALID_ARGUMENT = 1,
    FRAC_ERR_UNSUPPORTED = 2,
    FRAC_ERR_CUDA = 3,
    FRAC_ERR_TIMEOUT = 4
} frac_status;

typedef enum { FRAC_DTYPE_F32 = 0, FRAC_DTYPE_BF16 = 1 } frac_dtype;

/* Bits of frac_dims.flags. */
enum {
    /* Use the CUDA-core chunked kernels even where tensor-core ones exist.  Without it, bf16
       calls with headdim 64, dstate in {64, 128} and nmodes in {4, 8} run the forward and the
       backward on the tensor cores (TMA-fed tcgen05 MMAs, chunk 128); they need the dtype
       tensors and the states 16-byte aligned.  On the CUDA-core path, dstate 1 (the paper's
       scalar B, C per position) runs the forward as the direct per-mode recurrence. */
    FRAC_FLAG_FORCE_SIMT = 1,
    /* frac_scan_bwd only: the workspace already holds the per-chunk states that a frac_scan_fwd
       call with the same inputs, h0 and dims left in this same workspace (give both calls one
       buffer of frac_scan_bwd_workspace_size bytes), so the backward does not recompute them.
       Rejected with FRAC_ERR_INVALID_ARGUMENT when the forward and backward would run on
       different paths (then the states are not compatible). */
    FRAC_FLAG_BWD_REUSE_FWD_STATES = 2,
    /* Test hook of the bounded device waits (frac_scan_fwd and frac_scan_fwd_static on the
       tensor-core path only; FRAC_ERR_UNSUPPORTED elsewhere): every CTA of the forward state
       pass first waits about a millisecond on a barrier that nothing signals, gives up, records
       FRAC_ERR_TIMEOUT in the call's status word and exits the way a kernel whose wait ran out
       does.  y and h_final are then incomplete; frac_workspace_status (or
       frac_scan_fwd_static_status) returns FRAC_ERR_TIMEOUT.  Not for production use. */
    FRAC_FLAG_TEST_EXPIRE_WAIT = 4
};

typedef struct {
    int64_t batch;   /* B >= 1 */
    int64_t seqlen;  /* L >= 0 (ignored by frac_decode_step) */
    int64_t nheads;  /* H >= 1 */
    int64_t headdim; /* P >= 1 */
    int64_t ngroups; /* G >= 1, H % G == 0 */
    int64_t dstate;  /* N >= 1 */
    int64_t nmodes;  /* K, 1 <= K <= 32 */
    int64_t chunk;   /* Q: 0 = implementation's choice; otherwise one of the sizes the selected
                        path supports (128 on the tensor-core forward; 16, 32 or 64 on the
                        CUDA-core kernels).  Results do not depend on Q beyond rounding. */
    int32_t dtype;   /* frac_dtype */
    int32_t flags;   /* FRAC_FLAG_* */
} frac_dims;

/*
 * Bytes of scratch device memory frac_scan_fwd needs for these dims (per-chunk mode states
 * handed from the chunk-serial state pass to the chunk-parallel output kernel; on the
 * tensor-core path also the per-position mode coefficients).
 */
frac_status frac_scan_fwd_workspace_size(const frac_dims *dims, size_t *bytes);

/*
 * Chunked parallel forward scan (training / prefill), the Remark after Eq. read-softmax:
 * the affine recurrence evaluated chunk by chunk with chunk-local cumulative log-decays,
 * the stable intra-chunk coefficient Gamma of App. F, cross-chunk state passing, and the
 * skip D fused into the output.
 *   x, dt, alpha, lam, tau, Bm, Cm, w_read, w_write, D : inputs (layouts above)
 *   h0       : initial mode state, or NULL for zeros
 *   y        : output [B, L, H, P] (dtype)
 *   h_final  : final mode state S_L (float32), or NULL; it is the decode cache
 *   workspace: >= frac_scan_fwd_workspace_size bytes, 256-byte aligned; contents undefined on
 *              entry; on exit it holds the per-chunk states (see FRAC_FLAG_BWD_REUSE_FWD_STATES);
 *              must not be used concurrently by another call.
 */
frac_status frac_scan_fwd(const frac_dims *dims, const void *x, const float *dt,
                          const float *alpha, const float *lam, const float *tau,
                          const void *Bm, const void *Cm, const void *w_read,
                          const void *w_write, const float *D, const float *h0, void *y,
                          float *h_final, void *workspace, size_t workspace_bytes,
                          void *stream);

/* Bytes of scratch device memory frac_scan_bwd needs for these dims. */
frac_status frac_scan_bwd_workspace_size(const frac_dims *dims, size_t *bytes);

/*
 * Backward of frac_scan_fwd (the adjoint of the recurrence; the paper trains through it but
 * prints no formulas).  Recomputes the forward mode states from the inputs, then walks the
 * chunks in reverse carrying dS, and forms every gradient chunk-locally.  The gradient through
 * the decay, rho_t <dS_t, S_{t-1}>, is evaluated per position from terms that each carry their
 * own decay factor, so it stays accurate when lambda^(1/alpha) is large.
 *   dy       : upstream gradient of y (dtype)
 *   dh_final : upstream gradient of h_final (float32), or NULL for zeros
 *   dx, dB, dC, dw_read, dw_write : gradients (dtype, layouts of their inputs)
 *   ddt, dalpha, dlam : gradients (float32)
 *   dD       : gradient of D (float32 [H]), summed over batch and sequence
 *   dh0      : gradient of h0 (float32), or NULL if not wanted
 *   dtau     : gradient of the timescales tau (float32 [H, K], summed over batch and sequence),
 *              or NULL if not wanted: the learned-timescale variant (App. G).  It is the e_t-
 *              weighted per-mode decay gradient, gathered chunk by chunk from terms whose spans
 *              of e_t sum in closed form; its sums use float atomics (rounding order not fixed).
 * dB / dC sum over the heads of each group.  All outputs are overwritten (not accumulated).
 */
frac_status frac_scan_bwd(const frac_dims *dims, const void *x, const float *dt,
                          const float *alpha, const float *lam, const float *tau,
                          const void *Bm, const void *Cm, const void *w_read,
                          const void *w_write, const float *D, const float *h0,
                          const void *dy, const float *dh_final, void *dx, float *ddt,
                          float *dalpha, float *dlam, void *dB, void *dC, void *dw_read,
                          void *dw_write, float *dD, float *dh0, float *dtau, void *workspace,
                          size_t workspace_bytes, void *stream);

/*
 * One decode step (Algorithm 1: a single token, recurrent form with the cached state):
 * updates every mode of `state` in place and writes y_t.  One pass over the state.
 *   x_t [B, H, P], B_t/C_t [B, G, N], w_read/w_write [B, H, K] : dtype
 *   dt, alpha, lam [B, H], tau [H, K], D [H] : float32
 *   state [B, H, K, P, N] float32, read and written (may not alias any other argument)
 *   y_t   [B, H, P] : dtype
 * dims->seqlen and dims->chunk are ignored.
 */
frac_status frac_decode_step(const frac_dims *dims, const void *x_t, const float *dt,
                             const float *alpha, const float *lam, const float *tau,
                             const void *B_t, const void *C_t, const void *w_read,
                             const void *w_write, const float *D, float *state, void *y_t,
                             void *stream);

/*
 * Allocation-free forward scan.  The paper has no counterpart; this exists for callers that
 * cannot hand the library scratch memory: for example code running inside a host application
 * that owns the whole device-memory budget and gives its plug-ins no allocator, or code that
 * may only touch the buffers it was given once it is running.  Same arguments and results as
 * frac_scan_fwd without the workspace: the per-chunk mode states go to a fixed device array
 * of FRAC_SCAN_FWD_STATIC_SCRATCH_BYTES that the library owns on every GPU that loads it, held
 * until the process exits.  No device memory is allocated by the call.
 *   - Problems whose frac_scan_fwd_workspace_size exceeds that size are rejected with
 *     FRAC_ERR_UNSUPPORTED (frac_last_error() says how much they need); nothing is enqueued.
 *   - The first call on a device looks up the array's address on that device (a CUDA runtime
 *     query, made with that device current); make the first call before any stream capture.
 *     The address is cached with the context that was current; a call that finds another
 *     context (for example after cudaDeviceReset) looks it up again, which must then also
 *     happen outside a stream capture.
 *   - All calls share the array.  Calls whose GPU work overlaps (other streams, other host
 *     threads on the same device) race on it and must be serialised by the caller.  Nothing in
 *     it needs to start at zero: every per-chunk state is written before it is read.
 *   - A kernel whose bounded device wait gave up leaves y and h_final incomplete and records
 *     FRAC_ERR_TIMEOUT in the array's status word, which frac_scan_fwd_static_status reads;
 *     overlapping calls share that word as well.
 */
#define FRAC_SCAN_FWD_STATIC_SCRATCH_BYTES ((size_t)64 << 20)
frac_status frac_scan_fwd_static(const frac_dims *dims, const void *x, const float *dt,
                                 const float *alpha, const float *lam, const float *tau,
                                 const void *Bm, const void *Cm, const void *w_read,
                                 const void *w_write, const float *D, const float *h0, void *y,
                                 float *h_final, void *stream);

/*
 * Status of the last frac_scan_fwd_static call on the current device: waits for `stream` and
 * returns FRAC_ERR_TIMEOUT if one of that call's kernels gave up on a bounded device-side wait
 * (its outputs are then incomplete), FRAC_OK otherwise (the word is reset by every call).
 * Like frac_workspace_status for the library's own array; allocates nothing.
 */
frac_status frac_scan_fwd_static_status(void *stream);

/*
 * Scan-parameter construction (the fused "scan parameter" kernel of App. F, and its backward).
 * From the outputs of the layer's projections it forms the scan's controls and mode weights,
 * per position (b, t) and head h (Sec. 3.3; Eq. read-softmax; Algorithm 1 of App. D):
 *   Delta   = clip(softplus(dt_raw + dt_bias_h), dt_min, dt_max)    (linear map with learned bias,
 *                                                                     then softplus; clip of App. E.3)
 *   alpha   = sigmoid(alpha_raw)                                     (0 < alpha < 1)
 *   lambda  = clip(softplus(lam_raw), lam_min, lam_max)              (clip of App. E.3)
 *   w_read  = softmax_m(-alpha ln tau_m + g_read_m)                  (Eq. read-softmax)
 *   w_write = softmax_m(-alpha ln tau_m + g_write_m)                 (same form, own logits)
 * g_read / g_write are the mode-wise residual logits (the learned maps applied to the content
 * signal).  The outputs feed frac_scan_fwd / frac_scan_bwd / frac_decode_step directly.
 * Variants (frac_prep_config.flags):
 *   FRAC_PREP_ZOH_INJECTION : w_write is divided by lambda, so that the scan's
 *       kappa = (1 - rho) w_write is the exact zero-order-hold injection (1 - rho~)/lambda of
 *       Eq. rho-beta-def-frac instead of Algorithm 1's 1 - rho~.
 *   FRAC_PREP_NO_SOFTMAX    : weights = the logits themselves (App. G ablation "w/o softmax R/W";
 *       the normalisation is removed and nothing replaces it).
 *   FRAC_PREP_NO_READ_PRIOR / FRAC_PREP_NO_WRITE_PRIOR : drop -alpha ln tau from the read / write
 *       logits (App. G ablations "w/o write prior"; both: the "pure multiscale bank").
 *   FRAC_PREP_ALPHA_ONE     : alpha = 1 for every token (App. G ablation; alpha_raw may be NULL
 *       and gets a zero gradient).
 * dims: batch and seqlen (rows = batch x seqlen positions; seqlen 1 for a decode step), nheads,
 * nmodes (1..32) and dtype (of the logits, the weights and their gradients) are used; the other
 * fields are ignored.  Layouts:
 *   dt_raw, alpha_raw, lam_raw, dt, alpha, lam (+ grads)  [batch, seqlen, nheads]  float32
 *   g_read, g_write, w_read, w_write (+ grads)             [batch, seqlen, nheads, nmodes]  dtype
 *   dt_bias, ddt_bias [nheads] float32 (NULL = no bias / not wanted); tau, dtau [nheads, nmodes]
 * Arithmetic is float32.  Errors as for the scan calls (everything checked before anything is
 * enqueued); no workspace is needed.
 */
typedef struct {
    float dt_min, dt_max;   /* clip of Delta: the language-modelling setting uses [1e-4, 1] */
    float lam_min, lam_max; /* clip of lambda: [0.25, 4] there */
    int32_t flags;          /* FRAC_PREP_* */
    int32_t reserved;       /* must be 0 */
} frac_prep_config;

enum {
    FRAC_PREP_ZOH_INJECTION = 1,
    FRAC_PREP_NO_SOFTMAX = 2,
    FRAC_PREP_NO_READ_PRIOR = 4,
    FRAC_PREP_NO_WRITE_PRIOR = 8,
    FRAC_PREP_ALPHA_ONE = 16
};

frac_status frac_param_prep_fwd(const frac_dims *dims, const frac_prep_config *cfg,
                                const float *dt_raw, const float *dt_bias, const float *alpha_raw,
                                const float *lam_raw, const void *g_read, const void *g_write,
                                const float *tau, float *dt, float *alpha, float *lam,
                                void *w_read, void *w_write, void *stream);

/*
 * Backward of frac_param_prep_fwd: from the gradients of its outputs (ddt, dalpha, dlam,
 * dw_read, dw_write: typically those frac_scan_bwd returned) to the gradients of its inputs.
 * Clipping passes the gradient where the clipped value lies inside [min, max] (bounds
 * included).  ddt_bias [nheads] sums the Delta gradient over positions; dtau [nheads, nmodes]
 * is the part of the timescale gradient that flows through the -alpha ln tau prior (add
 * frac_scan_bwd's dtau for learned timescales).  Both are overwritten; NULL = not wanted.
 * The sums over positions use float atomics: their rounding order is not fixed.
 */
frac_status frac_param_prep_bwd(const frac_dims *dims, const frac_prep_config *cfg,
                                const float *dt_raw, const float *dt_bias, const float *alpha_raw,
                                const float *lam_raw, const void *g_read, const void *g_write,
                                const float *tau, const float *ddt, const float *dalpha,
                                const float *dlam, const void *dw_read, const void *dw_write,
                                float *ddt_raw, float *dalpha_raw, float *dlam_raw, void *dg_read,
                                void *dg_write, float *ddt_bias, float *dtau, void *stream);

/*
 * Depthwise causal 1-D convolution of the FracMixer content branch (Sec. 3.3: u_t comes from a
 * local depthwise causal convolution along the sequence; width d_conv = 4 in App. E.2 / E.4):
 *   pre[b, t, c] = bias_c + sum_{j=0}^{W-1} w[c, j] x[b, t - (W-1) + j, c]
 *   u = pre, or u = silu(pre) = pre * sigmoid(pre) with FRAC_CONV_SILU (the activation of the
 *   Mamba-family mixers the layer follows; the paper names only the convolution)
 * Positions before the sequence start read a carried state of the W - 1 previous inputs
 * (state_in [B, C, W-1], oldest first; NULL = zeros), which makes prefill -> decode and split
 * sequences exact.  Layouts: x, u, du, dx [B, L, C] and states in dims->dtype; w [C, W], bias
 * [C] (NULL = none) and their gradients float32.  W <= 8, L <= 16,776,960.  Arithmetic is
 * float32.
 */
typedef struct {
    int64_t batch;    /* B >= 1 */
    int64_t seqlen;   /* L >= 0 (ignored by frac_conv1d_step) */
    int64_t channels; /* C >= 1 */
    int64_t width;    /* W, 1 <= W <= 8 */
    int32_t dtype;    /* frac_dtype of x, u, the states and their gradients */
    int32_t flags;    /* FRAC_CONV_* */
} frac_conv_dims;

enum { FRAC_CONV_SILU = 1 };

/* Forward over a sequence.  state_out [B, C, W-1] (or NULL) receives the last W - 1 inputs
   (the carried state for a continuation); it must not alias state_in. */
frac_status frac_conv1d_fwd(const frac_conv_dims *dims, const void *x, const float *w,
                            const float *bias, const void *state_in, void *u, void *state_out,
                            void *stream);

/* Backward of frac_conv1d_fwd's u: dx; dw [C, W] and dbias [C] summed over batch and sequence
   (overwritten; float atomics, rounding order not fixed); dstate_in [B, C, W-1] (or NULL) the
   gradient of the carried inputs. */
frac_status frac_conv1d_bwd(const frac_conv_dims *dims, const void *x, const float *w,
                            const float *bias, const void *state_in, const void *du, void *dx,
                            float *dw, float *dbias, void *dstate_in, void *stream);

/* One decode step: x_t, u_t [B, C]; state [B, C, W-1] is read and shifted in place (the newest
   input x_t enters at the end). */
frac_status frac_conv1d_step(const frac_conv_dims *dims, const void *x_t, const float *w,
                             const float *bias, void *state, void *u_t, void *stream);

/*
 * Gated RMS normalisation of the scan output before the output projection (Sec. 3.3 "gated
 * normalization", read as the Mamba2 form the layer design follows):
 *   v = y * silu(z)  (v = y when z is NULL),   out = v / sqrt(mean_group(v^2) + eps) * weight
 * with the mean over consecutive groups of group_size features of each row.  y, z, out and
 * their gradients [rows, dim] in dtype (16-byte aligned); weight, dweight [dim] float32.
 * group_size must be a multiple of 8 that divides dim; dim <= 32768.
 */
typedef struct {
    int64_t rows;       /* >= 0 (e.g. batch x seqlen) */
    int64_t dim;        /* features per row */
    int64_t group_size; /* features per normalisation group (dim for one group) */
    float eps;          /* >= 0, e.g. 1e-5 */
    int32_t dtype;      /* frac_dtype */
    int32_t flags;      /* 0 */
} frac_norm_dims;

frac_status frac_gated_rmsnorm_fwd(const frac_norm_dims *dims, const void *y, const void *z,
                                   const float *weight, void *out, void *stream);

/* Backward: dy, dz (NULL when z is NULL) and dweight (overwritten, summed over rows by float
   atomics: rounding order not fixed). */
frac_status frac_gated_rmsnorm_bwd(const frac_norm_dims *dims, const void *y, const void *z,
                                   const float *weight, const void *dout, void *dy, void *dz,
                                   float *dweight, void *stream);

/*
 * Kernel tracing (a profiling aid, off by default).  While enabled, every kernel the library
 * launches is bracketed by two CUDA events recorded on its launch stream (do not enable it
 * while a stream is being captured into a CUDA graph).  frac_trace_collect waits for the
 * recorded events and returns, per kernel name, the launch count and summed device time since
 * the last frac_trace_reset; it writes at most `capacity` entries and the total in *count.
 */
typedef struct {
    char name[64];
    int32_t launches;
    double total_ms;
} frac_trace_entry;

frac_status frac_trace_enable(int on);
frac_status frac_trace_collect(frac_trace_entry *out, int capacity, int *count);
frac_status frac_trace_reset(void);

/*
 * Waits for `stream` and reports the device status word of a scan call's workspace:
 * FRAC_ERR_TIMEOUT if one of the call's kernels gave up on a bounded device-side wait (its
 * outputs are then incomplete), FRAC_OK otherwise.  The word is reset by every scan call.
 */
frac_status frac_workspace_status(const void *workspace, void *stream);

/* Static description of a status code. */
const char *frac_status_string(frac_status status);

/* Detail of the last failure on the calling thread ("" if none). */
const char *frac_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* FRAC_H_ */
