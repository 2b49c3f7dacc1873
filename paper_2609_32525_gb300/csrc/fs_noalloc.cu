// fs_slice_fwd_noalloc: the slice forward on a scratch buffer that is part of
// this library's device code, for callers that cannot provide a workspace.
// Contract: include/flashslice.h.  Nothing here allocates device memory: the
// scratch is a static device array, placed by the CUDA driver when the
// library's device code is loaded, and the call runs the same host code and
// kernels as fs_slice_fwd with that array as its workspace.
#include "flashslice.h"

#include <cuda_runtime.h>

#include <mutex>

// The fixed scratch (one per device).
static __device__ __align__(256) unsigned char g_noalloc_scratch[FS_NOALLOC_SCRATCH_BYTES];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_mutex;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch on the current device.  The lookup (a CUDA
// runtime call) runs on the first call per device only; later calls read the
// cached address.
fs_status scratch_address(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return FS_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return FS_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_mutex);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return FS_ERR_CUDA;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return FS_OK;
}

}  // namespace

extern "C" fs_status fs_slice_fwd_noalloc(const fs_shape* s, const void* x_mid, const void* fx,
                                          const float* W_slice, const float* bias, const float* tau,
                                          float* tokens, float* wsum, float* lse, int finalize,
                                          const void** scratch, fs_stream_t stream) {
  const size_t need = fs_workspace_bytes(s, FS_OP_SLICE_FWD);
  if (need == 0)  // invalid or unsupported shape: fs_slice_fwd reports which, before any launch
    return fs_slice_fwd(s, x_mid, fx, W_slice, bias, tau, tokens, wsum, lse, finalize, nullptr, 0, stream);
  if (need > FS_NOALLOC_SCRATCH_BYTES) return FS_ERR_SCRATCH_TOO_SMALL;
  void* ws = nullptr;
  if (fs_status e = scratch_address(&ws)) return e;
  if (scratch) *scratch = ws;
  // fs_slice_fwd clears the status word at the start of ws (the only part of
  // the workspace that must start at zero) before its first kernel.
  return fs_slice_fwd(s, x_mid, fx, W_slice, bias, tau, tokens, wsum, lse, finalize, ws, FS_NOALLOC_SCRATCH_BYTES,
                      stream);
}
