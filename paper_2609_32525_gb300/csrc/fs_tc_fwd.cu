// Tensor-core forward path (sm_103a).  Not yet implemented: every shape takes
// the SIMT kernels.
#include "fs_tc.h"

namespace fs {

bool tc_forward_supported(const Shape&) { return false; }
int tc_forward_launch_count(const Shape&) { return 0; }
size_t tc_slice_partials_bytes(const Shape&) { return 0; }
size_t tc_slice_prep_bytes(const Shape&) { return 0; }
size_t tc_deslice_prep_bytes(const Shape&) { return 0; }

cudaError_t tc_stats(const Shape&, const void*, const float*, const float*, const float*, float*, void*,
                     uint32_t*, cudaStream_t) {
  return cudaErrorNotSupported;
}
cudaError_t tc_slice_fwd(const Shape&, const void*, const void*, const float*, const float*, const float*,
                         float*, float*, float*, int, float*, void*, uint32_t*, cudaStream_t) {
  return cudaErrorNotSupported;
}
cudaError_t tc_deslice_fwd(const Shape&, const void*, const float*, const float*, const float*, const float*,
                           const float*, void*, void*, uint32_t*, cudaStream_t) {
  return cudaErrorNotSupported;
}

}  // namespace fs
