// Tensor-core (tcgen05 / TMEM / TMA) forward path for bf16 inputs on sm_103a.
#pragma once

#include "fs_internal.h"

namespace fs {

// True when the bf16 tensor-core forward kernels implement this shape.
bool tc_forward_supported(const Shape& s);
// Kernels launched by tc_slice_fwd + tc_deslice_fwd (the mix is not counted).
int tc_forward_launch_count(const Shape& s);
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
cudaError_t tc_deslice_fwd(const Shape& s, const void* x, const float* W, const float* bias, const float* tau,
                           const float* zp, const float* lse, void* out, void* prep, uint32_t* status,
                           cudaStream_t st);

}  // namespace fs
