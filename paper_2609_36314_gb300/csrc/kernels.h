// Internal interface between the C-ABI layer and the kernels (not installed).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace frac {

// Sets the message frac_last_error() returns on the calling thread.
void set_last_error(const char *msg);

// Tracing hooks (no-ops unless frac_trace_enable(1)); bracket each kernel launch.
void trace_begin(const char *name, cudaStream_t st);
void trace_end(cudaStream_t st);

struct DecodeArgs {
    int B, H, P, G, N, K;
    const float *dt, *alpha, *lam, *tau, *D;
    float *state;
};

cudaError_t launch_decode(const DecodeArgs &a, int dtype, const void *x, const void *Bt,
                          const void *Ct, const void *wr, const void *ww, void *y,
                          cudaStream_t st);

// Problem dimensions as the chunked kernels see them.
struct ScanDims {
    int B, L, H, P, G, N, K;
    int Q;   // chunk length
    int nc;  // number of chunks = ceil(L / Q)
    // Test hook (FRAC_FLAG_TEST_EXPIRE_WAIT): when nonzero, the forward state pass's CTAs first
    // wait this many nanoseconds on a barrier that nothing signals, then take the timeout path.
    unsigned expire_ns = 0;
};

// Pointers of one scan call.  Element types follow the dtype of the call.
struct ScanPtrs {
    const void *x, *Bm, *Cm, *wr, *ww, *dy;
    const float *dt, *alpha, *lam, *tau, *D, *h0, *dh_final;
    void *y, *dx, *dB, *dC, *dwr, *dww;
    float *h_final, *ddt, *dalpha, *dlam, *dD, *dh0;
    float *dtau;  // [H, K] timescale gradient, or null when not wanted
};

// CUDA-core (SIMT) chunked path; works for float32 and bf16 I/O.
int simt_pick_chunk(const ScanDims &d, int requested);     // 0 if the shape is unsupported
size_t simt_state_elems(const ScanDims &d);                 // per-chunk state workspace elements
// float scratch of the N = 1 forward (local end states and chunk decays); 0 for other shapes
size_t simt_n1_scratch_elems(const ScanDims &d);
cudaError_t simt_scan_fwd(const ScanDims &d, int dtype, const ScanPtrs &p, void *S_in, float *n1_scratch,
                          cudaStream_t st);
// reuse_states: S_in already holds the forward's per-chunk states (no recompute)
// n1_scratch: simt_n1_scratch_elems floats (the N = 1 backward's chunk carries)
// err: the call's device status word (a kernel whose bounded wait gave up writes FRAC_ERR_TIMEOUT)
cudaError_t simt_scan_bwd(const ScanDims &d, int dtype, const ScanPtrs &p, void *S_in,
                          void *dS_out, float *dB_acc, float *dC_acc, float *n1_scratch,
                          bool reuse_states, int *err, cudaStream_t st);

// Tensor-core (tcgen05) path: bf16 inputs, chunk 128, P = 64, N in {64, 128}, K in {4, 8}.
bool tc_supported(const ScanDims &d, int dtype);
size_t tc_state_elems(const ScanDims &d);  // bf16 elements of the per-chunk state workspace
size_t tc_coef_elems(const ScanDims &d);   // float elements of the per-position coefficients
// floats per position of the {E hi, E lo, 0, 0, kappa[K]} array (padded to 16 bytes x 2^i)
__host__ __device__ inline int tc_ek_width(int K) { return K == 8 ? 16 : 8; }
size_t tc_ek_elems(const ScanDims &d);
// coef: [B, L, H, 4, K] float (f, s, u, exp(-E/tau) per position), written by the forward
cudaError_t tc_scan_fwd(const ScanDims &d, const ScanPtrs &p, void *S_in, float *coef, float *ek,
                        int *err, cudaStream_t st);
// Per-position mode coefficients of every chunk (the first kernel of both passes).
// ek: [B, L, H, tc_ek_width(K)] float: the in-chunk cumulative log-decay E (hi, lo) and kappa
cudaError_t tc_coef_launch(const ScanDims &d, const ScanPtrs &p, float *coef, float *ek, cudaStream_t st);
// Chunk-serial state pass on the tensor cores (forward: U = x, V = B, coefficients s; reverse:
// U = dy, V = C, coefficients f).
cudaError_t tc_state_pass_launch(const ScanDims &d, bool rev, const void *U, const void *V,
                                 const float *coef, const float *init, void *emit, float *fin,
                                 int *err, cudaStream_t st);
bool tc_make_map3(CUtensorMap *m, const void *ptr, uint64_t d0, uint64_t d1, uint64_t d2,
                  uint64_t stride1_bytes, uint64_t stride2_bytes, uint32_t b0, uint32_t b1,
                  uint32_t b2, int swizzle_bytes = 128);
// 3-D float32 tensor map with 128- or 64-byte swizzle (b0 = 32 or 16 floats)
bool tc_make_map3_f32(CUtensorMap *m, const void *ptr, uint64_t d0, uint64_t d1, uint64_t d2,
                      uint64_t stride1_bytes, uint64_t stride2_bytes, uint32_t b0, uint32_t b1,
                      uint32_t b2, int swizzle_bytes);
// 4-D float32 tensor map with 128-byte swizzle (box[0] = 32 floats)
bool tc_make_map4_f32(CUtensorMap *m, const void *ptr, const uint64_t dims[4], const uint64_t strides_bytes[3],
                      const uint32_t box[4]);
// Tensor-core backward (headdim 64 in addition to the forward's conditions).
bool tc_bwd_supported(const ScanDims &d, int dtype);
struct TcBwdWorkspace {  // S_in and coef first, at the offsets the forward uses
    void *S_in, *dS_out;                     // bf16 per-chunk states
    float *dx_acc, *dwr_acc, *dkap_acc;      // [B,L,H,P], [B,L,H,K] x 2
    float *ab_acc, *rect, *cdot, *mh_total;  // [B,L,H,2], [B,L,H], [B,H,nc,K], [B,nc,G,Q,Q]
    float *coef;                             // [B,L,H,4,K]: f, s, u, exp(-E/tau)
    float *ek;                               // [B,L,H,tc_ek_width(K)]: E (hi, lo), kappa
    float *dB_acc, *dC_acc;                  // [B,L,G,N] x 2
    float *inter_acc;                        // [B,L,H,2,K]: inter-chunk dw_read, dkappa (dtau)
};
size_t tc_bwd_workspace_bytes(const ScanDims &d, TcBwdWorkspace *layout, char *base);
// The intra-chunk pairs of the timescale gradient (both paths; a no-op unless p.dtau): adds
// tau^-2 sum_{k<t} (E_t - E_k) w_read_t kappa_k exp(-(E_t - E_k)/tau) G_tk H_tk per mode.
cudaError_t dtau_pairs_launch(const ScanDims &d, int dtype, const ScanPtrs &p, cudaStream_t st);
cudaError_t tc_scan_bwd(const ScanDims &d, const ScanPtrs &p, const TcBwdWorkspace &ws, int *err,
                        bool reuse_states, cudaStream_t st);

}  // namespace frac
