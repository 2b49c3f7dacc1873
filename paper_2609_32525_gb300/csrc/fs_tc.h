// Tensor-core (tcgen05 / TMEM / TMA) forward path for bf16 inputs on sm_103a.
#pragma once

#include "fs_internal.h"

namespace fs {

// True when the bf16 tensor-core forward kernels implement this shape.
bool tc_forward_supported(const Shape& s);
// Kernels launched by tc_slice_fwd + tc_deslice_fwd (the mix is not counted).
int tc_forward_launch_count(const Shape& s);
// Kernels launched by tc_stats.
int tc_stats_launch_count(const Shape& s);
// Workspace the tensor-core slice needs for its split-N partials and its
// prepared operand images; the deslice needs only the latter.
size_t tc_slice_partials_bytes(const Shape& s);
size_t tc_slice_prep_bytes(const Shape& s);
size_t tc_deslice_prep_bytes(const Shape& s);

cudaError_t tc_stats(const Shape& s, const void* x, const float* W, const float* bias, const float* tau,
                     float* lse, void* prep, uint32_t* status, cudaStream_t st);
cudaError_t tc_slice_fwd(const Shape& s, const void* x, const void* f, const float* W, const float* bias,
                         const float* tau, float* tokens, float* wsum, float* lse, int finalize, float* part,
                         void* prep, uint32_t* status, cudaStream_t st);
// The slice given the statistics lse (the statistics pass is skipped).
cudaError_t tc_slice_fwd_lse(const Shape& s, const void* x, const void* f, const float* W, const float* bias,
                             const float* tau, const float* lse, float* tokens, float* wsum, int finalize,
                             float* part, void* prep, uint32_t* status, cudaStream_t st);
cudaError_t tc_deslice_fwd(const Shape& s, const void* x, const float* W, const float* bias, const float* tau,
                           const float* zp, const float* lse, void* out, void* prep, uint32_t* status,
                           cudaStream_t st);

// Rows pass of the backward (the deslice kernel in backward mode 1 or 2) on
// prepared operands: W image, Z-layout image of t (hi then lo, G*128 bytes per
// (b,h)), lse point-extra rows; writes delta (and, mode 2, dfx), or adds to them
// when accumulate != 0 (a later slot range of the same points), and adds the two
// per-warpgroup partials of sum_g w dS to wds (which must start at zero).
cudaError_t tc_rows_bwd(const Shape& s, int mode, const void* x, const uint8_t* wimg, const uint8_t* zimg,
                        const void* px, const void* v, void* dfx, float* delta, float* wds, const float* dS,
                        int accumulate, uint32_t* status, cudaStream_t st);
size_t tc_rows_smem(const Shape& s, int mode, bool ps, bool hilo);

// ---- tensor-core backward (fs_tc_bwd.cu) ----
// True when the tensor-core backward implements this shape: bf16, d = 32, N >= 2,
// G <= 4096.  Its passes hold the operand images of at most 640 slots (padded to
// whole 128-slot blocks); a larger G runs them over slot ranges.
bool tc_backward_supported(const Shape& s);
// Workspace of one tensor-core backward call (mode 1 deslice, 2 slice).
size_t tc_backward_bytes(const Shape& s, int mode);
// Kernels launched by tc_deslice_bwd (mode 1) or tc_slice_bwd (mode 2).
int tc_backward_launch_count(const Shape& s, int mode);
cudaError_t tc_deslice_bwd(const Shape& s, const void* x, const float* W, const float* bias, const float* tau,
                           const float* zp, const float* lse, const void* dout, float* dzp, void* dx, float* dW,
                           float* db, float* dtau, int accumulate, void* ws_tc, uint32_t* status, cudaStream_t st);
// The coupling's whole backward (deslice, mix, slice) with one point pass for both
// calls' dx; workspace and kernel count.
size_t tc_coupling_bwd_bytes(const Shape& s);
int tc_coupling_bwd_launch_count(const Shape& s);
cudaError_t tc_coupling_bwd(const Shape& s, const void* x, const void* f, const void* dout, const float* W,
                            const float* bias, const float* tau, const float* M, const float* z, const float* wsum,
                            const float* zp, const float* lse, float* dzp, float* dz, float* dM, void* dx, void* dfx,
                            float* dW, float* db, float* dtau, int accumulate, float* dUS, void* ws_tc,
                            uint32_t* status, cudaStream_t st);
cudaError_t tc_slice_bwd(const Shape& s, const void* x, const void* f, const float* W, const float* bias,
                         const float* tau, const float* z, const float* wsum, const float* lse, const float* dz,
                         void* dx, void* dfx, float* dW, float* db, float* dtau, int accumulate, float* dUS,
                         void* ws_tc, uint32_t* status, cudaStream_t st);

}  // namespace fs
