// C ABI of the library: host-side validation, workspace layout, kernel dispatch.
// Declarations and the contract of every entry point: include/flashslice.h.
#include "fs_internal.h"
#include "fs_tc.h"

#include <algorithm>
#include <cmath>
#include <cstring>
#include <initializer_list>

namespace fs {

int num_sms() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) return 1;
  return n;
}

int slot_splits(const Shape& s) {
  const int64_t gblocks = (s.G + 127) / 128;
  const int64_t units = s.BH() * gblocks;
  int64_t P = (2LL * num_sms() + units - 1) / units;
  const int64_t max_by_n = (s.N + 63) / 64;
  if (P > max_by_n) P = max_by_n;
  if (P < 1) P = 1;
  if (P > 1024) P = 1024;
  return (int)P;
}

namespace {

constexpr size_t kAlign = 256;

bool valid_shape(const fs_shape* s) {
  if (!s) return false;
  if (s->B < 1 || s->N < 1 || s->H < 1 || s->d < 1 || s->G < 1) return false;
  if (s->dtype != FS_F32 && s->dtype != FS_BF16) return false;
  if (!(s->eps >= 0.f) || !std::isfinite(s->eps)) return false;
  if (s->dot != FS_DOT_BF16 && s->dot != FS_DOT_BF16X2) return false;
  const double elems = (double)s->B * (double)s->N * (double)s->H * (double)s->d;
  if (elems >= 1099511627776.0) return false;  // 2^40
  return true;
}

bool supported_shape(const fs_shape* s) {
  return (s->d == 16 || s->d == 32 || s->d == 64) && s->G <= 4096 && (int64_t)s->B * s->H <= 65535;
}

Shape to_shape(const fs_shape* s) { return Shape{s->B, s->N, s->H, s->d, s->G, s->dtype, s->eps, s->dot}; }

bool aligned(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// A byte range [p, p + n) of a caller buffer.
struct Span {
  const void* p;
  size_t n;
};
// True when two ranges share a byte.
bool overlap(Span a, Span b) {
  const uintptr_t a0 = reinterpret_cast<uintptr_t>(a.p), b0 = reinterpret_cast<uintptr_t>(b.p);
  return a.n && b.n && a0 < b0 + b.n && b0 < a0 + a.n;
}
// The out-of-place calls (the mixes and their backward) read every input while
// they write: no output may share a byte with an input or with another output.
bool disjoint(std::initializer_list<Span> ins, std::initializer_list<Span> outs) {
  for (const Span& o : outs) {
    for (const Span& i : ins)
      if (overlap(o, i)) return false;
    for (const Span& o2 : outs)
      if (&o2 != &o && overlap(o, o2)) return false;
  }
  return true;
}

// Byte sizes of the regions each op places in `ws` (each 256-byte aligned).
struct Regions {
  size_t status, partials, stats, delta, dus, dtau_p, tc, total;
};

Regions regions(const Shape& s, int op) {
  Regions r{};
  const int P = slot_splits(s);
  const size_t BHG = (size_t)s.BH() * s.G;
  const size_t pts = (size_t)s.BH() * s.N;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = align_up(off + bytes, kAlign);
    return o;
  };
  r.status = take(sizeof(uint32_t));
  switch (op) {
    case FS_OP_SLICE_FWD: {
      size_t part = (size_t)P * BHG * (s.d + 1) * sizeof(float);
      const size_t tcb = tc_slice_partials_bytes(s);
      if (tcb > part) part = tcb;
      r.partials = take(part);
      r.stats = take(pts * sizeof(float));
      r.tc = take(tc_slice_prep_bytes(s));
      break;
    }
    case FS_OP_DESLICE_FWD:
      r.stats = take(pts * sizeof(float));
      r.tc = take(tc_deslice_prep_bytes(s));
      break;
    case FS_OP_STATS:
      r.tc = take(tc_deslice_prep_bytes(s));
      break;
    case FS_OP_DESLICE_BWD:
      if (tc_backward_supported(s)) {
        r.stats = take(pts * sizeof(float));
        r.tc = take(std::max(tc_backward_bytes(s, 1), tc_deslice_prep_bytes(s)));
        break;
      }
      r.delta = take(pts * sizeof(float));
      r.partials = take((size_t)P * BHG * (2 * s.d + 2) * sizeof(float));
      r.dtau_p = take((size_t)s.BH() * simt_point_blocks(s) * sizeof(float));
      r.stats = take(pts * sizeof(float));
      r.tc = take(tc_deslice_prep_bytes(s));
      break;
    case FS_OP_SLICE_BWD:
      r.dus = take(BHG * (s.d + 1) * sizeof(float));
      if (tc_backward_supported(s)) {
        r.stats = take(pts * sizeof(float));
        r.tc = take(std::max(tc_backward_bytes(s, 2), tc_deslice_prep_bytes(s)));
        break;
      }
      r.delta = take(pts * sizeof(float));
      r.partials = take((size_t)P * BHG * (s.d + 2) * sizeof(float));
      r.dtau_p = take((size_t)s.BH() * simt_point_blocks(s) * sizeof(float));
      r.stats = take(pts * sizeof(float));
      r.tc = take(tc_deslice_prep_bytes(s));
      break;
    case FS_OP_COUPLING_BWD:
      if (tc_backward_supported(s)) {
        r.dus = take(BHG * (s.d + 1) * sizeof(float));
        r.stats = take(pts * sizeof(float));
        r.tc = take(std::max(tc_coupling_bwd_bytes(s), tc_deslice_prep_bytes(s)));
        break;
      }
      // the fused SIMT backward: dU|dS, delta, the slot partials (which first hold
      // the d z' partials), the points' temperature terms, the statistics
      r.dus = take(BHG * (s.d + 1) * sizeof(float));
      r.delta = take(pts * sizeof(float));
      r.partials = take((size_t)P * BHG * (s.d + 2) * sizeof(float));
      r.dtau_p = take((size_t)s.BH() * simt_point_blocks(s) * sizeof(float));
      r.stats = take(pts * sizeof(float));
      r.tc = take(tc_deslice_prep_bytes(s));
      break;
    default:
      return Regions{};
  }
  r.total = off;
  return r;
}

template <typename T>
T* at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<char*>(ws) + off);
}

fs_status check_ws(const Shape& s, int op, void* ws, size_t ws_bytes) {
  const Regions r = regions(s, op);
  if (!ws || !aligned(ws) || ws_bytes < r.total) return FS_ERR_INVALID;
  return FS_OK;
}

fs_status cuda_status(cudaError_t e) { return e == cudaSuccess ? FS_OK : FS_ERR_CUDA; }

// Every ws-using call starts by clearing its status word.
cudaError_t reset_status(void* ws, cudaStream_t st) { return cudaMemsetAsync(ws, 0, sizeof(uint32_t), st); }

// The backward forms its weights from fp32 logits, so it needs lse to ~1e-5.  On
// tensor-core shapes with bf16 products the forward's lse comes from logits with
// bf16-rounded W log2(e)/tau: the backward recomputes it with split products (the
// statistics pass, into ws).  With split products (and on the SIMT path) the
// caller's lse is already that accurate and is used as it is.  A caller without
// statistics for these weights (an untied deslice, Sec. 3) passes NULL and the
// backward computes them.
cudaError_t backward_stats(const Shape& sh, const void* x_mid, const float* W_slice, const float* bias,
                           const float* tau, const float* lse, void* ws, const Regions& r, uint32_t* status,
                           cudaStream_t st, const float** lse_use) {
  *lse_use = lse;
  // fp32 shapes take the fp32 SIMT backward: it gets exact fp32 statistics (the
  // forward's come from split bf16 products on the tensor cores).
  const bool tc = tc_forward_supported(sh) && sh.dtype == FS_BF16;
  const bool fp32_tc = tc_forward_supported(sh) && sh.dtype == FS_F32;
  if (lse && !fp32_tc && (!tc || sh.dot == FS_DOT_BF16X2)) return cudaSuccess;
  float* buf = at<float>(ws, r.stats);
  *lse_use = buf;
  if (!tc) return simt_stats(sh, x_mid, W_slice, bias, tau, buf, status, st);
  Shape split = sh;
  split.dot = FS_DOT_BF16X2;
  return tc_stats(split, x_mid, W_slice, bias, tau, buf, at<void>(ws, r.tc), status, st);
}

#define FS_CHECK_SHAPE(s)                               \
  do {                                                  \
    if (!valid_shape(s)) return FS_ERR_INVALID;         \
    if (!supported_shape(s)) return FS_ERR_UNSUPPORTED; \
  } while (0)

#define FS_CHECK_PTR(p)                                      \
  do {                                                       \
    if (!(p) || !aligned(p)) return FS_ERR_INVALID;          \
  } while (0)

#define FS_CUDA(call)                                          \
  do {                                                         \
    cudaError_t e_ = (call);                                   \
    if (e_ != cudaSuccess) return FS_ERR_CUDA;                 \
  } while (0)

}  // namespace
}  // namespace fs

using namespace fs;

extern "C" {

size_t fs_workspace_bytes(const fs_shape* s, int op) {
  if (!valid_shape(s) || !supported_shape(s)) return 0;
  return regions(to_shape(s), op).total;
}

const char* fs_status_string(fs_status st) {
  switch (st) {
    case FS_OK: return "FS_OK";
    case FS_ERR_INVALID: return "FS_ERR_INVALID: invalid argument";
    case FS_ERR_UNSUPPORTED: return "FS_ERR_UNSUPPORTED: shape not implemented";
    case FS_ERR_CUDA: return "FS_ERR_CUDA: CUDA runtime or launch failure";
    case FS_ERR_TIMEOUT: return "FS_ERR_TIMEOUT: device wait gave up";
    case FS_ERR_BAD_TAU: return "FS_ERR_BAD_TAU: tau <= 0 or not finite";
    case FS_ERR_SCRATCH_TOO_SMALL:
      return "FS_ERR_SCRATCH_TOO_SMALL: the shape needs more than the fixed scratch of fs_slice_fwd_noalloc";
  }
  return "unknown fs_status";
}

int fs_path_for_shape(const fs_shape* s) {
  if (!valid_shape(s) || !supported_shape(s)) return -1;
  return tc_forward_supported(to_shape(s)) ? 1 : 0;
}

int fs_backward_path_for_shape(const fs_shape* s) {
  if (!valid_shape(s) || !supported_shape(s)) return -1;
  return tc_backward_supported(to_shape(s)) ? 1 : 0;
}

int fs_forward_launch_count(const fs_shape* s) {
  if (!valid_shape(s) || !supported_shape(s)) return -1;
  const Shape sh = to_shape(s);
  if (tc_forward_supported(sh)) return tc_forward_launch_count(sh) + 1;  // + mix
  return 3 /*stats, partials, reduce*/ + 1 /*mix*/ + 1 /*deslice*/;
}

// Kernels of backward_stats for one backward call: none when it takes the caller's lse.
int backward_stats_launches(const Shape& sh, int lse_given) {
  const bool tc = tc_forward_supported(sh) && sh.dtype == FS_BF16;
  const bool fp32_tc = tc_forward_supported(sh) && sh.dtype == FS_F32;
  if (lse_given && !fp32_tc && (!tc || sh.dot == FS_DOT_BF16X2)) return 0;
  Shape split = sh;
  split.dot = FS_DOT_BF16X2;
  return tc ? tc_stats_launch_count(split) : 1;
}

int fs_backward_launch_count(const fs_shape* s, int lse_given) {
  if (!valid_shape(s) || !supported_shape(s)) return -1;
  const Shape sh = to_shape(s);
  // Each backward call recomputes the statistics unless backward_stats takes the caller's lse.
  const int stats = backward_stats_launches(sh, lse_given);
  const int mix_bwd = 2;  // d_tokens, dM
  if (tc_backward_supported(sh))
    return 2 * stats + tc_backward_launch_count(sh, 1) + mix_bwd + tc_backward_launch_count(sh, 2);
  return 2 * stats + 5 /*point, slot, three reductions*/ + mix_bwd + 5 /*prologue, point, slot, two reductions*/;
}

int fs_coupling_bwd_launch_count(const fs_shape* s, int lse_given) {
  if (!valid_shape(s) || !supported_shape(s)) return -1;
  const Shape sh = to_shape(s);
  if (!tc_backward_supported(sh)) return backward_stats_launches(sh, lse_given) + simt_coupling_bwd_launch_count();
  const bool tc = tc_forward_supported(sh);
  const int stats = (lse_given && sh.dot == FS_DOT_BF16X2) ? 0 : (tc ? 2 : 1);  // the statistics once
  return stats + tc_coupling_bwd_launch_count(sh);
}

fs_status fs_slice_fwd(const fs_shape* s, const void* x_mid, const void* fx, const float* W_slice,
                       const float* bias, const float* tau, float* tokens, float* wsum, float* lse,
                       int finalize, void* ws, size_t ws_bytes, fs_stream_t stream) {
  FS_CHECK_SHAPE(s);
  FS_CHECK_PTR(x_mid); FS_CHECK_PTR(fx); FS_CHECK_PTR(W_slice); FS_CHECK_PTR(bias); FS_CHECK_PTR(tau);
  FS_CHECK_PTR(tokens); FS_CHECK_PTR(wsum);
  if (lse && !aligned(lse)) return FS_ERR_INVALID;
  const Shape sh = to_shape(s);
  if (fs_status e = check_ws(sh, FS_OP_SLICE_FWD, ws, ws_bytes)) return e;
  const Regions r = regions(sh, FS_OP_SLICE_FWD);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  uint32_t* status = at<uint32_t>(ws, r.status);
  float* lse_buf = lse ? lse : at<float>(ws, r.stats);
  FS_CUDA(reset_status(ws, st));
  if (tc_forward_supported(sh)) {
    return cuda_status(tc_slice_fwd(sh, x_mid, fx, W_slice, bias, tau, tokens, wsum, lse_buf, finalize,
                                    at<float>(ws, r.partials), at<void>(ws, r.tc), status, st));
  }
  const int P = slot_splits(sh);
  float* part = at<float>(ws, r.partials);
  FS_CUDA(simt_stats(sh, x_mid, W_slice, bias, tau, lse_buf, status, st));
  FS_CUDA(simt_slice_partials(sh, P, x_mid, fx, W_slice, bias, tau, lse_buf, part, status, st));
  FS_CUDA(simt_reduce_tokens(sh, P, part, sh.G, tokens, wsum, finalize, st));
  return FS_OK;
}

fs_status fs_stats(const fs_shape* s, const void* x_mid, const float* W_slice, const float* bias, const float* tau,
                   float* lse, void* ws, size_t ws_bytes, fs_stream_t stream) {
  FS_CHECK_SHAPE(s);
  FS_CHECK_PTR(x_mid); FS_CHECK_PTR(W_slice); FS_CHECK_PTR(bias); FS_CHECK_PTR(tau); FS_CHECK_PTR(lse);
  const Shape sh = to_shape(s);
  if (fs_status e = check_ws(sh, FS_OP_STATS, ws, ws_bytes)) return e;
  const Regions r = regions(sh, FS_OP_STATS);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  uint32_t* status = at<uint32_t>(ws, r.status);
  FS_CUDA(reset_status(ws, st));
  if (tc_forward_supported(sh))
    return cuda_status(tc_stats(sh, x_mid, W_slice, bias, tau, lse, at<void>(ws, r.tc), status, st));
  return cuda_status(simt_stats(sh, x_mid, W_slice, bias, tau, lse, status, st));
}

fs_status fs_slice_fwd_lse(const fs_shape* s, const void* x_mid, const void* fx, const float* W_slice,
                           const float* bias, const float* tau, const float* lse, float* tokens, float* wsum,
                           int finalize, void* ws, size_t ws_bytes, fs_stream_t stream) {
  FS_CHECK_SHAPE(s);
  FS_CHECK_PTR(x_mid); FS_CHECK_PTR(fx); FS_CHECK_PTR(W_slice); FS_CHECK_PTR(bias); FS_CHECK_PTR(tau);
  FS_CHECK_PTR(lse); FS_CHECK_PTR(tokens); FS_CHECK_PTR(wsum);
  const Shape sh = to_shape(s);
  if (fs_status e = check_ws(sh, FS_OP_SLICE_FWD, ws, ws_bytes)) return e;
  const Regions r = regions(sh, FS_OP_SLICE_FWD);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  uint32_t* status = at<uint32_t>(ws, r.status);
  FS_CUDA(reset_status(ws, st));
  if (tc_forward_supported(sh))
    return cuda_status(tc_slice_fwd_lse(sh, x_mid, fx, W_slice, bias, tau, lse, tokens, wsum, finalize,
                                        at<float>(ws, r.partials), at<void>(ws, r.tc), status, st));
  const int P = slot_splits(sh);
  float* part = at<float>(ws, r.partials);
  FS_CUDA(simt_slice_partials(sh, P, x_mid, fx, W_slice, bias, tau, lse, part, status, st));
  FS_CUDA(simt_reduce_tokens(sh, P, part, sh.G, tokens, wsum, finalize, st));
  return FS_OK;
}

fs_status fs_slice_finalize(const fs_shape* s, float* tokens, const float* wsum, fs_stream_t stream) {
  FS_CHECK_SHAPE(s);
  FS_CHECK_PTR(tokens); FS_CHECK_PTR(wsum);
  return cuda_status(simt_finalize(to_shape(s), tokens, wsum, reinterpret_cast<cudaStream_t>(stream)));
}

fs_status fs_mix(const fs_shape* s, const float* M, const float* tokens, float* tokens_mixed,
                 fs_stream_t stream) {
  FS_CHECK_SHAPE(s);
  FS_CHECK_PTR(M); FS_CHECK_PTR(tokens); FS_CHECK_PTR(tokens_mixed);
  const size_t tb = (size_t)s->B * s->H * s->G * s->d * 4, mb = (size_t)s->H * s->G * s->G * 4;
  if (!disjoint({{M, mb}, {tokens, tb}}, {{tokens_mixed, tb}})) return FS_ERR_INVALID;
  return cuda_status(simt_mix(to_shape(s), M, tokens, tokens_mixed, reinterpret_cast<cudaStream_t>(stream)));
}

fs_status fs_mix_channels(const fs_shape* s, const float* Wc, const float* tokens, float* tokens_mixed,
                          fs_stream_t stream) {
  FS_CHECK_SHAPE(s);
  FS_CHECK_PTR(Wc); FS_CHECK_PTR(tokens); FS_CHECK_PTR(tokens_mixed);
  const size_t tb = (size_t)s->B * s->H * s->G * s->d * 4, wb = (size_t)s->H * s->d * s->d * 4;
  if (!disjoint({{Wc, wb}, {tokens, tb}}, {{tokens_mixed, tb}})) return FS_ERR_INVALID;
  return cuda_status(simt_mix_channels(to_shape(s), Wc, tokens, tokens_mixed, reinterpret_cast<cudaStream_t>(stream)));
}

fs_status fs_mix_channels_bwd(const fs_shape* s, const float* Wc, const float* tokens, const float* d_tokens_mixed,
                              float* d_tokens, float* dWc, fs_stream_t stream) {
  FS_CHECK_SHAPE(s);
  FS_CHECK_PTR(Wc); FS_CHECK_PTR(tokens); FS_CHECK_PTR(d_tokens_mixed); FS_CHECK_PTR(d_tokens); FS_CHECK_PTR(dWc);
  const size_t tb = (size_t)s->B * s->H * s->G * s->d * 4, wb = (size_t)s->H * s->d * s->d * 4;
  if (!disjoint({{Wc, wb}, {tokens, tb}, {d_tokens_mixed, tb}}, {{d_tokens, tb}, {dWc, wb}})) return FS_ERR_INVALID;
  return cuda_status(simt_mix_channels_bwd(to_shape(s), Wc, tokens, d_tokens_mixed, d_tokens, dWc,
                                           reinterpret_cast<cudaStream_t>(stream)));
}

fs_status fs_deslice_fwd(const fs_shape* s, const void* x_mid, const float* W_slice, const float* bias,
                         const float* tau, const float* tokens_mixed, const float* lse, void* out, void* ws,
                         size_t ws_bytes, fs_stream_t stream) {
  FS_CHECK_SHAPE(s);
  FS_CHECK_PTR(x_mid); FS_CHECK_PTR(W_slice); FS_CHECK_PTR(bias); FS_CHECK_PTR(tau);
  FS_CHECK_PTR(tokens_mixed); FS_CHECK_PTR(out);
  if (lse && !aligned(lse)) return FS_ERR_INVALID;
  const Shape sh = to_shape(s);
  if (fs_status e = check_ws(sh, FS_OP_DESLICE_FWD, ws, ws_bytes)) return e;
  const Regions r = regions(sh, FS_OP_DESLICE_FWD);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  uint32_t* status = at<uint32_t>(ws, r.status);
  FS_CUDA(reset_status(ws, st));
  const float* lse_use = lse;
  if (!lse_use) {
    float* buf = at<float>(ws, r.stats);
    if (tc_forward_supported(sh)) FS_CUDA(tc_stats(sh, x_mid, W_slice, bias, tau, buf, at<void>(ws, r.tc), status, st));
    else FS_CUDA(simt_stats(sh, x_mid, W_slice, bias, tau, buf, status, st));
    lse_use = buf;
  }
  if (tc_forward_supported(sh))
    return cuda_status(tc_deslice_fwd(sh, x_mid, W_slice, bias, tau, tokens_mixed, lse_use, out,
                                      at<void>(ws, r.tc), status, st));
  return cuda_status(simt_deslice(sh, x_mid, W_slice, bias, tau, tokens_mixed, lse_use, out, status, st));
}

fs_status fs_deslice_bwd(const fs_shape* s, const void* x_mid, const float* W_slice, const float* bias,
                         const float* tau, const float* tokens_mixed, const float* lse, const void* dout,
                         float* d_tokens_mixed, void* dx_mid, float* dW, float* dbias, float* dtau, int accumulate,
                         void* ws, size_t ws_bytes, fs_stream_t stream) {
  FS_CHECK_SHAPE(s);
  FS_CHECK_PTR(x_mid); FS_CHECK_PTR(W_slice); FS_CHECK_PTR(bias); FS_CHECK_PTR(tau);
  FS_CHECK_PTR(tokens_mixed); FS_CHECK_PTR(dout); FS_CHECK_PTR(d_tokens_mixed);
  if (lse && !aligned(lse)) return FS_ERR_INVALID;
  FS_CHECK_PTR(dx_mid); FS_CHECK_PTR(dW); FS_CHECK_PTR(dbias); FS_CHECK_PTR(dtau);
  const Shape sh = to_shape(s);
  if (fs_status e = check_ws(sh, FS_OP_DESLICE_BWD, ws, ws_bytes)) return e;
  const Regions r = regions(sh, FS_OP_DESLICE_BWD);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  FS_CUDA(reset_status(ws, st));
  const float* lse_use = nullptr;
  FS_CUDA(backward_stats(sh, x_mid, W_slice, bias, tau, lse, ws, r, at<uint32_t>(ws, r.status), st, &lse_use));
  if (tc_backward_supported(sh))
    return cuda_status(tc_deslice_bwd(sh, x_mid, W_slice, bias, tau, tokens_mixed, lse_use, dout, d_tokens_mixed,
                                      dx_mid, dW, dbias, dtau, accumulate, at<void>(ws, r.tc),
                                      at<uint32_t>(ws, r.status), st));
  return cuda_status(simt_deslice_bwd(sh, slot_splits(sh), x_mid, W_slice, bias, tau, tokens_mixed, lse_use, dout,
                                      d_tokens_mixed, dx_mid, dW, dbias, dtau, accumulate, at<float>(ws, r.delta),
                                      at<float>(ws, r.partials), at<float>(ws, r.dtau_p),
                                      at<uint32_t>(ws, r.status), st));
}

fs_status fs_mix_bwd(const fs_shape* s, const float* M, const float* tokens, const float* d_tokens_mixed,
                     float* d_tokens, float* dM, fs_stream_t stream) {
  FS_CHECK_SHAPE(s);
  FS_CHECK_PTR(M); FS_CHECK_PTR(tokens); FS_CHECK_PTR(d_tokens_mixed); FS_CHECK_PTR(d_tokens); FS_CHECK_PTR(dM);
  const size_t tb = (size_t)s->B * s->H * s->G * s->d * 4, mb = (size_t)s->H * s->G * s->G * 4;
  if (!disjoint({{M, mb}, {tokens, tb}, {d_tokens_mixed, tb}}, {{d_tokens, tb}, {dM, mb}})) return FS_ERR_INVALID;
  return cuda_status(simt_mix_bwd(to_shape(s), M, tokens, d_tokens_mixed, d_tokens, dM,
                                  reinterpret_cast<cudaStream_t>(stream)));
}

fs_status fs_slice_bwd(const fs_shape* s, const void* x_mid, const void* fx, const float* W_slice,
                       const float* bias, const float* tau, const float* tokens, const float* wsum,
                       const float* lse, const float* d_tokens, void* dx_mid, void* dfx, float* dW, float* dbias,
                       float* dtau, int accumulate, void* ws, size_t ws_bytes, fs_stream_t stream) {
  FS_CHECK_SHAPE(s);
  FS_CHECK_PTR(x_mid); FS_CHECK_PTR(fx); FS_CHECK_PTR(W_slice); FS_CHECK_PTR(bias); FS_CHECK_PTR(tau);
  FS_CHECK_PTR(tokens); FS_CHECK_PTR(wsum); FS_CHECK_PTR(d_tokens);
  if (lse && !aligned(lse)) return FS_ERR_INVALID;
  FS_CHECK_PTR(dx_mid); FS_CHECK_PTR(dfx); FS_CHECK_PTR(dW); FS_CHECK_PTR(dbias); FS_CHECK_PTR(dtau);
  const Shape sh = to_shape(s);
  if (fs_status e = check_ws(sh, FS_OP_SLICE_BWD, ws, ws_bytes)) return e;
  const Regions r = regions(sh, FS_OP_SLICE_BWD);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  FS_CUDA(reset_status(ws, st));
  const float* lse_use = nullptr;
  FS_CUDA(backward_stats(sh, x_mid, W_slice, bias, tau, lse, ws, r, at<uint32_t>(ws, r.status), st, &lse_use));
  if (tc_backward_supported(sh))
    return cuda_status(tc_slice_bwd(sh, x_mid, fx, W_slice, bias, tau, tokens, wsum, lse_use, d_tokens, dx_mid, dfx,
                                    dW, dbias, dtau, accumulate, at<float>(ws, r.dus), at<void>(ws, r.tc),
                                    at<uint32_t>(ws, r.status), st));
  return cuda_status(simt_slice_bwd(sh, slot_splits(sh), x_mid, fx, W_slice, bias, tau, tokens, wsum, lse_use,
                                    d_tokens, dx_mid, dfx, dW, dbias, dtau, accumulate, at<float>(ws, r.delta),
                                    at<float>(ws, r.dus), at<float>(ws, r.partials), at<float>(ws, r.dtau_p),
                                    at<uint32_t>(ws, r.status), st));
}

fs_status fs_coupling_bwd(const fs_shape* s, const void* x_mid, const void* fx, const float* W_slice,
                          const float* bias, const float* tau, const float* M, const float* tokens,
                          const float* wsum, const float* tokens_mixed, const float* lse, const void* dout,
                          float* d_tokens_mixed, float* d_tokens, void* dx_mid, void* dfx, float* dW, float* dbias,
                          float* dtau, float* dM, int accumulate, void* ws, size_t ws_bytes, fs_stream_t stream) {
  FS_CHECK_SHAPE(s);
  FS_CHECK_PTR(x_mid); FS_CHECK_PTR(fx); FS_CHECK_PTR(W_slice); FS_CHECK_PTR(bias); FS_CHECK_PTR(tau);
  FS_CHECK_PTR(M); FS_CHECK_PTR(tokens); FS_CHECK_PTR(wsum); FS_CHECK_PTR(tokens_mixed); FS_CHECK_PTR(dout);
  if (lse && !aligned(lse)) return FS_ERR_INVALID;
  FS_CHECK_PTR(d_tokens_mixed); FS_CHECK_PTR(d_tokens); FS_CHECK_PTR(dx_mid); FS_CHECK_PTR(dfx);
  FS_CHECK_PTR(dW); FS_CHECK_PTR(dbias); FS_CHECK_PTR(dtau); FS_CHECK_PTR(dM);
  // the mix backward inside reads M, tokens and d_tokens_mixed while it writes d_tokens and dM
  const size_t tb = (size_t)s->B * s->H * s->G * s->d * 4, mb = (size_t)s->H * s->G * s->G * 4;
  if (!disjoint({{M, mb}, {tokens, tb}, {tokens_mixed, tb}}, {{d_tokens_mixed, tb}, {d_tokens, tb}, {dM, mb}}))
    return FS_ERR_INVALID;
  const Shape sh = to_shape(s);
  if (fs_status e = check_ws(sh, FS_OP_COUPLING_BWD, ws, ws_bytes)) return e;
  if (!tc_backward_supported(sh)) {
    const Regions r = regions(sh, FS_OP_COUPLING_BWD);
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    uint32_t* status = at<uint32_t>(ws, r.status);
    FS_CUDA(reset_status(ws, st));
    const float* lse_use = nullptr;
    FS_CUDA(backward_stats(sh, x_mid, W_slice, bias, tau, lse, ws, r, status, st, &lse_use));
    return cuda_status(simt_coupling_bwd(sh, slot_splits(sh), x_mid, fx, dout, W_slice, bias, tau, M, tokens, wsum,
                                         tokens_mixed, lse_use, d_tokens_mixed, d_tokens, dM, dx_mid, dfx, dW, dbias,
                                         dtau, accumulate, at<float>(ws, r.delta), at<float>(ws, r.dus),
                                         at<float>(ws, r.partials), at<float>(ws, r.dtau_p), status, st));
  }
  const Regions r = regions(sh, FS_OP_COUPLING_BWD);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  FS_CUDA(reset_status(ws, st));
  const float* lse_use = nullptr;
  FS_CUDA(backward_stats(sh, x_mid, W_slice, bias, tau, lse, ws, r, at<uint32_t>(ws, r.status), st, &lse_use));
  return cuda_status(tc_coupling_bwd(sh, x_mid, fx, dout, W_slice, bias, tau, M, tokens, wsum, tokens_mixed, lse_use,
                                     d_tokens_mixed, d_tokens, dM, dx_mid, dfx, dW, dbias, dtau, accumulate,
                                     at<float>(ws, r.dus), at<void>(ws, r.tc), at<uint32_t>(ws, r.status), st));
}

fs_status fs_device_status(const void* ws, fs_stream_t stream) {
  if (!ws || !aligned(ws)) return FS_ERR_INVALID;
  uint32_t v = 0;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(&v, ws, sizeof(v), cudaMemcpyDeviceToHost, st) != cudaSuccess) return FS_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return FS_ERR_CUDA;
  return static_cast<fs_status>(v);
}

}  // extern "C"
