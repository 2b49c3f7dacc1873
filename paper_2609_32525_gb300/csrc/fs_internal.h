// Internal declarations shared by the library's translation units (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <cstdint>
#include <cstddef>

#include "flashslice.h"

namespace fs {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// Status word codes written by kernels (same values as fs_status).
constexpr uint32_t kDevOk = 0, kDevTimeout = 4, kDevBadTau = 5;

struct Shape {
  int64_t B, N;
  int H, d, G;
  int dtype;
  float eps;
  int dot;  // fs_dot
  int64_t BH() const { return B * (int64_t)H; }
  int64_t points() const { return B * N; }
};

inline size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

int num_sms();
// Number of point splits for slot-owned kernels (fixed for a shape on a device).
int slot_splits(const Shape& s);

// ---- SIMT kernels (fs_simt.cu) -------------------------------------------------
// Point blocks per (b, h) of the SIMT point-owned kernels; the backward's dt_part
// buffer holds one float per (b, h, point block).
int64_t simt_point_blocks(const Shape& s);
cudaError_t simt_stats(const Shape& s, const void* x, const float* W, const float* bias,
                       const float* tau, float* lse, uint32_t* status, cudaStream_t st);
cudaError_t simt_slice_partials(const Shape& s, int P, const void* x, const void* f,
                                const float* W, const float* bias, const float* tau,
                                const float* lse, float* part, uint32_t* status, cudaStream_t st);
// Fixed-order sum of split partials [P, B*H, Gs, d+1] (Gs >= G slot rows per (b, h);
// the first G are reduced) into tokens (normalised when finalize) and wsum.
cudaError_t simt_reduce_tokens(const Shape& s, int P, const float* part, int Gs, float* tokens,
                               float* wsum, int finalize, cudaStream_t st);
cudaError_t simt_finalize(const Shape& s, float* tokens, const float* wsum, cudaStream_t st);
cudaError_t simt_mix(const Shape& s, const float* M, const float* z, float* zp, cudaStream_t st);
// The attention-free core: zp[b,h,g,:] = Wc[h] z[b,h,g,:]; its backward dz = Wc^T dzp,
// dWc = sum over b and g of dzp z^T.
cudaError_t simt_mix_channels(const Shape& s, const float* Wc, const float* z, float* zp, cudaStream_t st);
cudaError_t simt_mix_channels_bwd(const Shape& s, const float* Wc, const float* z, const float* dzp, float* dz,
                                  float* dWc, cudaStream_t st);
cudaError_t simt_mix_bwd(const Shape& s, const float* M, const float* z, const float* dzp,
                         float* dz, float* dM, cudaStream_t st);
cudaError_t simt_deslice(const Shape& s, const void* x, const float* W, const float* bias,
                         const float* tau, const float* zp, const float* lse, void* out,
                         uint32_t* status, cudaStream_t st);
cudaError_t simt_deslice_bwd(const Shape& s, int P, const void* x, const float* W,
                             const float* bias, const float* tau, const float* zp,
                             const float* lse, const void* dout, float* dzp, void* dx,
                             float* dW, float* db, float* dtau, int accumulate, float* delta,
                             float* part, float* dt_part, uint32_t* status, cudaStream_t st);
// dUS[bh][g] = (dz_g / (S_g + eps), -(dz_g . z_g) / (S_g + eps)) (d + 1 floats per slot).
cudaError_t simt_slice_bwd_prep(const Shape& s, const float* z, const float* wsum, const float* dz, float* dUS,
                                cudaStream_t st);
// Fixed-order reduction of slot-owned backward partials part[P][B*H][Gs][PS]
// (Gs >= G slot rows per (b, h), the first G reduced; PS = 2d + 2 with the token
// gradient first when has_dzp, else d + 2) into dW, dbias (and dzp), and of
// dt_part[B*H][nblk] into dtau.
cudaError_t simt_reduce_bwd(const Shape& s, int P, const float* part, int Gs, int PS, int has_dzp, const float* tau,
                            float* dzp, float* dW, float* db, float* dtau, const float* dt_part, int64_t nblk,
                            int accumulate, cudaStream_t st);
// The token gradient alone from partials whose first d words per slot are dz'.
// The coupling's whole backward on the SIMT kernels (fs_coupling_bwd on shapes the
// tensor-core backward does not take); delta, dUS, part, dt_part as in the calls above
// (part holds P * B*H * G * (d + 2) floats).
cudaError_t simt_coupling_bwd(const Shape& s, int P, const void* x, const void* fx, const void* dout,
                              const float* W, const float* bias, const float* tau, const float* M, const float* z,
                              const float* wsum, const float* zp, const float* lse, float* dzp, float* dz,
                              float* dM, void* dx, void* dfx, float* dW, float* db, float* dtau, int accumulate,
                              float* delta, float* dUS, float* part, float* dt_part, uint32_t* status,
                              cudaStream_t st);
int simt_coupling_bwd_launch_count();
cudaError_t simt_reduce_dzp(const Shape& s, int P, const float* part, int Gs, int PS, float* dzp, cudaStream_t st);
cudaError_t simt_slice_bwd(const Shape& s, int P, const void* x, const void* f, const float* W,
                           const float* bias, const float* tau, const float* z,
                           const float* wsum, const float* lse, const float* dz, void* dx,
                           void* dfx, float* dW, float* db, float* dtau, int accumulate,
                           float* delta, float* dUS, float* part, float* dt_part,
                           uint32_t* status, cudaStream_t st);

}  // namespace fs
