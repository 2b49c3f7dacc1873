// fs_slice_fwd_noalloc: the slice forward on a scratch buffer that is part of
// this library's device code, for callers that cannot provide a workspace.
// Contract: include/flashslice.h.  Nothing here allocates device memory: the
// scratch is a static device array, placed by the CUDA driver when the
// library's device code is loaded, and the call runs the same host code and
// kernels as fs_slice_fwd with that array as its workspace.
#include "flashslice.h"

#include <cuda.h>
#include <cuda_runtime.h>

#include <mutex>

// The fixed scratch (one per device).
static __device__ __align__(256) unsigned char g_noalloc_scratch[FS_NOALLOC_SCRATCH_BYTES];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_mutex;

// The scratch address looked up on a device, and the unique id of the context it
// was looked up in: a device reset, or another context made current, gives a new
// id, and the address is looked up again.
struct Entry {
  unsigned long long ctx_id;
  void* addr;
};
Entry g_entry[kMaxDevices] = {};

using CtxGetCurrent = CUresult (*)(CUcontext*);
using CtxGetId = CUresult (*)(CUcontext, unsigned long long*);
CtxGetCurrent g_get_current = nullptr;
CtxGetId g_get_id = nullptr;
std::once_flag g_once;

// Unique id (for the life of the process) of the calling thread's current context.
bool current_context_id(unsigned long long* id) {
  std::call_once(g_once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_get_current = reinterpret_cast<CtxGetCurrent>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_get_id = reinterpret_cast<CtxGetId>(p);
  });
  CUcontext c = nullptr;
  return g_get_current && g_get_id && g_get_current(&c) == CUDA_SUCCESS && c != nullptr &&
         g_get_id(c, id) == CUDA_SUCCESS;
}

// Device address of the scratch on the current device, in the current context.
// The lookup (a CUDA runtime call) runs on the first call per device and again
// after the device's context has changed; other calls read the cached address.
fs_status scratch_address(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return FS_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return FS_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_mutex);
  unsigned long long id = 0;
  const bool have_id = current_context_id(&id);
  if (have_id && g_entry[dev].addr != nullptr && g_entry[dev].ctx_id == id) {
    *out = g_entry[dev].addr;
    return FS_OK;
  }
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return FS_ERR_CUDA;
  // The lookup makes the device's primary context current if none was: its id now.
  if (current_context_id(&id))
    g_entry[dev] = Entry{id, p};
  else
    g_entry[dev] = Entry{0, nullptr};  // no context id available: look up again next time
  *out = p;
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
