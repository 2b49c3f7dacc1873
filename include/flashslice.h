/*
 * flashslice.h -- C ABI of the GB300 slice -> token mix -> deslice library.
 *
 * The operation is the coupling of Transolver's physics-attention sublayer
 * with a constant token core (paper Sec. 2 "The Transolver layer" and Eq. (1);
 * Appendix G.1 "Single-tile kernels" / "G-blocked kernels").  Per batch b and
 * head h, with x = x_mid[b,:,h,:] (N x d), f = fx[b,:,h,:] (N x d),
 * W = W_slice[h] (d x G), beta = bias[h] (G), tau = tau[h]:
 *
 *   a_ng   = (x_n . W[:,g] + beta_g) / tau           slice logits
 *   w_ng   = exp(a_ng - lse_n),  lse_n = log sum_g exp(a_ng)
 *   S_g    = sum_n w_ng,   U_g = sum_n w_ng f_n      (partials over points)
 *   z_g    = U_g / (S_g + eps)                       tokens
 *   z'_g   = sum_k M[g,k] z_k                        constant G x G mix
 *   out_n  = sum_g w_ng z'_g                         deslice, tied weights
 *
 * The N x H x G weight tensor w is never written to memory: every pass
 * recomputes it tile by tile from x_mid and the per-point statistic lse.
 *
 * Conventions for every entry point
 *  - All tensor pointers are DEVICE pointers owned by the caller.  The library
 *    never allocates, frees or synchronises (except fs_device_status, which
 *    synchronises `stream` to read the status word).  Every call is
 *    asynchronous on `stream` (a cudaStream_t; NULL = legacy default stream).
 *  - Layouts are dense, row-major, contiguous:
 *      x_mid, fx, out, dout, dx_mid, dfx : [B, N, H, d]   dtype of the shape
 *      W_slice, dW                       : [H, d, G]      fp32
 *      bias, dbias                       : [H, G]         fp32
 *      tau, dtau                         : [H]            fp32
 *      M, dM                             : [H, G, G]      fp32, M[h][g][k]
 *      tokens, tokens_mixed, d_tokens*   : [B, H, G, d]   fp32
 *      wsum                              : [B, H, G]      fp32
 *      lse                               : [B, H, N]      fp32, natural log
 *    Channel c of a point's C = H*d features is head c / d, lane c % d.
 *  - Every pointer must be 16-byte aligned.
 *  - `ws` is caller-owned scratch of at least fs_workspace_bytes(shape, op)
 *    bytes (16-byte aligned).  Its first word is a device status word that
 *    each call resets; fs_device_status reads it.
 *  - Host-side validation fails with FS_ERR_INVALID / FS_ERR_UNSUPPORTED
 *    before anything is launched.  Device-side problems (tau <= 0 or not
 *    finite; a bounded wait that gave up) are written to the status word and
 *    the affected kernel skips its work; no kernel traps.
 *  - Results are deterministic: no floating-point atomics; partial sums over
 *    points are reduced in a fixed order, so repeated calls on the same
 *    device agree bit for bit.
 *  - Supported: d in {16, 32, 64}; G in [1, 4096]; B*H <= 65535; B*N*H*d < 2^40.
 *    Kernels (fs_path_for_shape, fs_backward_path_for_shape say which):
 *      FS_BF16, d = 32, G <= 1024: the forward on tcgen05 tensor cores, fp32
 *        accumulation, at the dot level of fs_shape.dot (below).
 *      FS_BF16, d = 32, N >= 2 (any supported G): the backward on tensor cores,
 *        always with split products; past G = 640 its passes run over ranges of
 *        at most 640 slots, whose dx_mid and dfx contributions are summed in bf16.
 *      FS_F32, d = 32, G <= 1024, B*N*H*G >= 2^24: the forward on tensor cores
 *        with every operand split into two bf16 halves (normwise relative error
 *        ~1e-5); the backward in fp32 FMA.
 *      everything else: fp32 FMA (SIMT) kernels.
 *
 * Call sequence of one coupling (a training step):
 *   fs_slice_fwd   (x_mid, fx)            -> tokens, wsum, lse
 *   fs_mix         (M, tokens)            -> tokens_mixed   (or fs_mix_channels)
 *   fs_deslice_fwd (x_mid, tokens_mixed, lse) -> out
 *   fs_deslice_bwd (..., dout)            -> d_tokens_mixed, dx_mid, dW, dbias, dtau
 *   fs_mix_bwd     (M, tokens, d_tokens_mixed) -> d_tokens, dM
 *   fs_slice_bwd   (..., d_tokens, accumulate = 1) -> dfx; adds to dx_mid, dW, dbias, dtau
 * Each call that takes `ws` gets scratch sized by fs_workspace_bytes for its op.
 */
#ifndef FLASHSLICE_H
#define FLASHSLICE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* fs_stream_t; /* identical to cudaStream_t */

typedef enum fs_status {
  FS_OK = 0,
  FS_ERR_INVALID = 1,     /* null/misaligned pointer, bad size, workspace too small */
  FS_ERR_UNSUPPORTED = 2, /* well-formed shape that no kernel implements (e.g. d = 48) */
  FS_ERR_CUDA = 3,        /* a CUDA runtime call or kernel launch failed */
  FS_ERR_TIMEOUT = 4,     /* device: a bounded wait gave up (status word only) */
  FS_ERR_BAD_TAU = 5,     /* device: some tau[h] <= 0 or not finite (status word only) */
  FS_ERR_SCRATCH_TOO_SMALL = 6 /* fs_slice_fwd_noalloc: the shape needs more than its fixed scratch */
} fs_status;

typedef enum fs_dtype { FS_F32 = 0, FS_BF16 = 1 } fs_dtype;

/* Arithmetic of the point-by-slot products for FS_BF16 shapes on the tensor
 * cores (the paper's "dot levels", App. G.2; fp32 accumulation throughout):
 *   FS_DOT_BF16   both operands of every product in bf16: W log2(e)/tau and the
 *                 slice weights rounded to bf16 (the paper's "bf16" level).
 *                 Outputs within ~1e-2 relative of exact.
 *   FS_DOT_BF16X2 W log2(e)/tau and the slice weights each carried as two bf16
 *                 halves (hi + lo, ~2^-16 relative) in the statistics and slice
 *                 passes, and in the deslice where its images fit in shared
 *                 memory (G <= 768): tokens, weight sums and lse to ~1e-4,
 *                 which the temperature gradient needs (a near-cancelling sum).
 *                 Slower: two more K-steps per logits block, twice the slice
 *                 products.
 * Ignored for FS_F32 shapes (split into bf16 halves on the tensor cores, or
 * fp32 FMA) and on the SIMT path. */
typedef enum fs_dot { FS_DOT_BF16 = 0, FS_DOT_BF16X2 = 1 } fs_dot;

typedef struct fs_shape {
  int64_t B;     /* batch size, >= 1 */
  int64_t N;     /* points per sample, >= 1 */
  int32_t H;     /* heads, >= 1 */
  int32_t d;     /* head width (value width equals it), 16, 32 or 64 */
  int32_t G;     /* slices per head, 1..4096 */
  int32_t dtype; /* fs_dtype of the [B,N,H,d] point tensors */
  float eps;     /* added to the weight sums before normalising, >= 0 (paper: 1e-5) */
  int32_t dot;   /* fs_dot: product arithmetic of the tensor-core path */
} fs_shape;

typedef enum fs_op {
  FS_OP_SLICE_FWD = 0,
  FS_OP_DESLICE_FWD = 1,
  FS_OP_DESLICE_BWD = 2,
  FS_OP_SLICE_BWD = 3,
  FS_OP_STATS = 4,
  FS_OP_COUPLING_BWD = 5
} fs_op;

/* Bytes of scratch `ws` that entry point `op` needs for this shape on the
 * current device (0 for an invalid shape).  Depends on the device's SM count. */
size_t fs_workspace_bytes(const fs_shape* s, int op);

/* Slice (Sec. 2; App. G.1 "G-blocked kernels": statistics, slot-owned partial
 * numerators and weight sums, normalisation after the partials are combined).
 *   in : x_mid, fx [B,N,H,d]; W_slice [H,d,G]; bias [H,G]; tau [H]
 *   out: tokens [B,H,G,d] = U/(S+eps) if finalize != 0, else the unnormalised
 *        numerators U (for a cross-device sum before fs_slice_finalize);
 *        wsum [B,H,G] = S; lse [B,H,N] (may be NULL: then kept in ws only). */
fs_status fs_slice_fwd(const fs_shape* s, const void* x_mid, const void* fx,
                       const float* W_slice, const float* bias, const float* tau,
                       float* tokens, float* wsum, float* lse, int finalize,
                       void* ws, size_t ws_bytes, fs_stream_t stream);

/* The statistics pass alone (App. G.1, the per-point statistic of the G-blocked
 * kernels): lse [B,H,N] (natural log) of the logits of these weights, exactly as
 * fs_slice_fwd writes it.  With fs_slice_fwd_lse it splits fs_slice_fwd in two,
 * so that fx can still be on its way to the device while the statistics run;
 * it also gives an untied deslice or a FrozenSlice layer its statistics.
 * ws: FS_OP_STATS's workspace. */
fs_status fs_stats(const fs_shape* s, const void* x_mid, const float* W_slice,
                   const float* bias, const float* tau, float* lse, void* ws,
                   size_t ws_bytes, fs_stream_t stream);

/* Slice given its statistics: fs_slice_fwd with lse [B,H,N] an input (as
 * fs_slice_fwd writes it, natural log) and no statistics pass.  For the
 * FrozenSlice variant (Sec. 3, the variants table: the slice weights of layer 1
 * reused by every layer), where a later layer slices its own fx with the
 * layer-1 logits input, weights and statistics; and for any caller that
 * already holds lse for these weights.  ws: FS_OP_SLICE_FWD's workspace. */
fs_status fs_slice_fwd_lse(const fs_shape* s, const void* x_mid, const void* fx,
                           const float* W_slice, const float* bias, const float* tau,
                           const float* lse, float* tokens, float* wsum, int finalize,
                           void* ws, size_t ws_bytes, fs_stream_t stream);

/* tokens <- tokens / (wsum + eps), in place ("column normalisation after
 * partials have been combined", App. G.1). */
fs_status fs_slice_finalize(const fs_shape* s, float* tokens, const float* wsum,
                            fs_stream_t stream);

/* Constant token mix, the core of Eq. (1) acting on the slot index:
 * tokens_mixed[b,h,g,:] = sum_k M[h,g,k] tokens[b,h,k,:].  Out-of-place only: an
 * output that shares any byte with an input is rejected (FS_ERR_INVALID). */
fs_status fs_mix(const fs_shape* s, const float* M, const float* tokens,
                 float* tokens_mixed, fs_stream_t stream);

/* The attention-free core (Sec. 2 after Eq. (1); "NoTokenAttn" in the Sec. 3
 * variants table): A is the identity, so the tokens do not interact, and a
 * learned linear map acts on the channels of each token, one per head:
 * tokens_mixed[b,h,g,c] = sum_k Wc[h,c,k] tokens[b,h,g,k].  Wc [H,d,d] fp32.
 * Out-of-place only (overlapping input and output: FS_ERR_INVALID).  It may
 * replace fs_mix, or follow it (the two commute). */
fs_status fs_mix_channels(const fs_shape* s, const float* Wc, const float* tokens,
                          float* tokens_mixed, fs_stream_t stream);

/* Backward of fs_mix_channels: d_tokens[b,h,g,k] = sum_c Wc[h,c,k]
 * d_tokens_mixed[b,h,g,c] (overwritten); dWc [H,d,d] = sum over b and g of
 * d_tokens_mixed tokens^T (overwritten).  Outputs that overlap an input or each
 * other: FS_ERR_INVALID. */
fs_status fs_mix_channels_bwd(const fs_shape* s, const float* Wc, const float* tokens,
                              const float* d_tokens_mixed, float* d_tokens, float* dWc,
                              fs_stream_t stream);

/* Deslice with tied weights (Sec. 2; App. G.1): out[b,n,h,:] = sum_g w z'_g.
 *   lse: statistics from fs_slice_fwd; NULL makes the call compute them first
 *   (into ws).  out has the dtype of the shape.  The Untied variant (Sec. 3, the
 *   variants table: the deslice gets its own projection and temperature) passes
 *   its own W_slice, bias, tau and lse = NULL. */
fs_status fs_deslice_fwd(const fs_shape* s, const void* x_mid, const float* W_slice,
                         const float* bias, const float* tau, const float* tokens_mixed,
                         const float* lse, void* out, void* ws, size_t ws_bytes,
                         fs_stream_t stream);

/* Backward of the deslice given dout (App. G.1 "Backward uses separate
 * point-owned and slot-owned kernels"; temperature gradient App. G.2):
 *   d_tokens_mixed [B,H,G,d] = sum_n w_ng dout_n  (always overwritten)
 *   dx_mid [B,N,H,d], dW [H,d,G], dbias [H,G], dtau [H]: the contribution of
 *   the deslice weights; written if accumulate == 0, added if accumulate != 0.
 *   lse: the statistics of these weights from the forward, or NULL (an untied
 *   deslice, which kept none): the call then computes them into ws.  The backward
 *   forms its weights from fp32 logits and needs lse to ~1e-5: on tensor-core
 *   shapes (fs_path_for_shape == 1) with dot = FS_DOT_BF16, whose lse comes
 *   from logits with bf16-rounded W log2(e)/tau, it recomputes lse with split
 *   products into ws; otherwise it uses the caller's lse. */
fs_status fs_deslice_bwd(const fs_shape* s, const void* x_mid, const float* W_slice,
                         const float* bias, const float* tau, const float* tokens_mixed,
                         const float* lse, const void* dout, float* d_tokens_mixed,
                         void* dx_mid, float* dW, float* dbias, float* dtau,
                         int accumulate, void* ws, size_t ws_bytes, fs_stream_t stream);

/* Backward of the mix: d_tokens = M^T d_tokens_mixed per (b,h) (overwritten);
 * dM [H,G,G] = sum_b d_tokens_mixed tokens^T (overwritten).  Outputs that overlap
 * an input or each other: FS_ERR_INVALID. */
fs_status fs_mix_bwd(const fs_shape* s, const float* M, const float* tokens,
                     const float* d_tokens_mixed, float* d_tokens, float* dM,
                     fs_stream_t stream);

/* Backward of the slice given d_tokens (the gradient w.r.t. the normalised
 * tokens); tokens and wsum are the forward's normalised tokens and S; lse as
 * in fs_deslice_bwd (NULL: computed; recomputed with split products for
 * FS_DOT_BF16).
 *   dfx [B,N,H,d] (overwritten); dx_mid, dW, dbias, dtau: written if
 *   accumulate == 0, added if accumulate != 0. */
fs_status fs_slice_bwd(const fs_shape* s, const void* x_mid, const void* fx,
                       const float* W_slice, const float* bias, const float* tau,
                       const float* tokens, const float* wsum, const float* lse,
                       const float* d_tokens, void* dx_mid, void* dfx, float* dW,
                       float* dbias, float* dtau, int accumulate, void* ws,
                       size_t ws_bytes, fs_stream_t stream);

/* The whole backward of one coupling in one call: the results of
 *   fs_deslice_bwd(..., accumulate) ; fs_mix_bwd ; fs_slice_bwd(..., accumulate = 1)
 * (App. G.1 backward; App. G.2 temperature gradient; the mix backward of Eq. (1)).
 *   d_tokens_mixed, d_tokens [B,H,G,d], dfx [B,N,H,d], dM [H,G,G]: overwritten;
 *   dx_mid [B,N,H,d], dW [H,d,G], dbias [H,G], dtau [H]: the sum of both calls'
 *   contributions, written if accumulate == 0, added if accumulate != 0.
 *   tokens, wsum, tokens_mixed, lse: the forward's (lse may be NULL, as in the
 *   separate calls).  ws: fs_workspace_bytes(s, FS_OP_COUPLING_BWD).
 * The two calls' da_ng share the weights, so one point pass over (point, slot)
 * forms da_D + da_S and dx from it, and one slot pass dW, dbias, dtau, instead of
 * one of each per call; d_tokens_mixed comes first, as the slice's unnormalised
 * numerators with dout for fx.  This holds on the tensor-core backward
 * (fs_backward_path_for_shape == 1) and on the fp32 SIMT one.  Results agree with
 * the separate calls to rounding (for instance dx is summed before its one rounding
 * to the input dtype instead of after each call's).  M, tokens and tokens_mixed
 * overlapping an output, or two outputs overlapping each other: FS_ERR_INVALID. */
fs_status fs_coupling_bwd(const fs_shape* s, const void* x_mid, const void* fx,
                          const float* W_slice, const float* bias, const float* tau,
                          const float* M, const float* tokens, const float* wsum,
                          const float* tokens_mixed, const float* lse, const void* dout,
                          float* d_tokens_mixed, float* d_tokens, void* dx_mid, void* dfx,
                          float* dW, float* dbias, float* dtau, float* dM, int accumulate,
                          void* ws, size_t ws_bytes, fs_stream_t stream);

/* Fixed-scratch variant of fs_slice_fwd.  The paper has no counterpart.
 *
 * For callers that cannot give the library device memory at the call site: a
 * program that lays out all of its device memory once at start-up and may not
 * allocate afterwards, or a caller (a plain C host, a foreign-language binding)
 * that holds no device allocator of its own.  Instead of a workspace argument,
 * this entry point uses one scratch buffer of FS_NOALLOC_SCRATCH_BYTES that is
 * part of the library's device code (a static device array), so neither the
 * caller nor the library allocates anything for the call.
 *   - Arguments, outputs and numerics are those of fs_slice_fwd (it runs the
 *     same kernels).  A shape whose fs_workspace_bytes(s, FS_OP_SLICE_FWD)
 *     exceeds FS_NOALLOC_SCRATCH_BYTES is rejected with
 *     FS_ERR_SCRATCH_TOO_SMALL before anything is launched; invalid or
 *     unsupported shapes give fs_slice_fwd's errors.
 *   - The first call on a device (with that device current) looks up the
 *     scratch's device address through the CUDA runtime; later calls on that
 *     device reuse it while the device's context stays the same.  After a
 *     cudaDeviceReset, or with another context current, the next call looks the
 *     address up again.  Make each call that does the lookup (the first one, and
 *     the first after a reset or context change) before any stream capture.
 *   - Each call clears the status word at the start of the scratch; nothing
 *     else in the scratch has to start at zero.
 *   - There is ONE scratch per device.  Calls that can overlap in time (on
 *     different streams, or from different host threads) race on it and
 *     corrupt each other's results: serialise them.
 *   - scratch: if not NULL, receives the scratch's device address, which
 *     fs_device_status accepts to read the call's device status. */
#define FS_NOALLOC_SCRATCH_BYTES ((size_t)16 << 20)
fs_status fs_slice_fwd_noalloc(const fs_shape* s, const void* x_mid, const void* fx,
                               const float* W_slice, const float* bias, const float* tau,
                               float* tokens, float* wsum, float* lse, int finalize,
                               const void** scratch, fs_stream_t stream);

/* Synchronises `stream` and returns the device status word of `ws`
 * (FS_OK, FS_ERR_TIMEOUT or FS_ERR_BAD_TAU), or FS_ERR_CUDA. */
fs_status fs_device_status(const void* ws, fs_stream_t stream);

/* Static, human-readable name of a status code. */
const char* fs_status_string(fs_status st);

/* Kernel path the library takes for this shape: 0 = SIMT fp32 kernels,
 * 1 = tcgen05 tensor-core kernels.  For tests and benchmarks. */
int fs_path_for_shape(const fs_shape* s);

/* Kernel path of the backward (fs_deslice_bwd, fs_slice_bwd) for this shape:
 * 0 = SIMT fp32 kernels, 1 = tcgen05 tensor-core kernels (bf16, d = 32,
 * N >= 2, any supported G, over slot ranges past G = 640; the weights with split
 * products whatever s->dot says).
 * For tests and benchmarks. */
int fs_backward_path_for_shape(const fs_shape* s);

/* Number of kernels the forward (slice + mix + deslice) launches for this shape. */
int fs_forward_launch_count(const fs_shape* s);

/* Number of kernels the backward (fs_deslice_bwd + fs_mix_bwd + fs_slice_bwd)
 * launches for this shape.  lse_given: nonzero when both backward calls get the
 * forward's lse (each call that must recompute the statistics launches that pass
 * again).  Memsets are not counted.  -1 for an invalid or unsupported shape. */
int fs_backward_launch_count(const fs_shape* s, int lse_given);

/* Number of kernels fs_coupling_bwd launches for this shape (lse_given as above;
 * the one call recomputes the statistics at most once).  -1 for an invalid or
 * unsupported shape. */
int fs_coupling_bwd_launch_count(const fs_shape* s, int lse_given);

#ifdef __cplusplus
}
#endif

#endif /* FLASHSLICE_H */
