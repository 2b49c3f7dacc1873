// Pieces shared by the tensor-core kernels of the forward (fs_tc_fwd.cu) and the
// backward (fs_tc_bwd.cu): tile constants, the operand images and their prep
// kernels, block bookkeeping, the logits MMA chain, the slice-weight helpers and
// the host-side tensor maps, splits and launch helpers.  Internal linkage: every
// translation unit that includes it gets its own copy.
#pragma once

#include "fs_tc.h"
#include "fs_tc_ptx.cuh"

#include <cuda_bf16.h>
#include <cudaTypedefs.h>
#include <mutex>

namespace fs {
namespace {

using namespace tc;

constexpr int kThreads = 384;
constexpr int kTile = 128;        // points per tile
constexpr int kGC = 128;          // slots per logits block
constexpr int kD = 32;            // head width of the tensor-core path
constexpr int kSoftmaxWarp0 = 4;  // warps 4..11: two softmax warpgroups
constexpr int kStages = 3;        // x-tile pipeline depth (stats / deslice)
constexpr int kSliceStages = 8;   // slice pipeline depth (it streams x, F and px for every 128 slots)
constexpr int kSBuf = 3;          // S buffers (logits run up to two blocks ahead)
constexpr uint32_t kXBytes = kTile * 64;   // 128 points x 32 bf16
constexpr uint32_t kExBytes = kTile * 32;  // 128 rows x 16 bf16
constexpr uint32_t kFBlock = kTile * 32;   // 128 points x 16 channels
constexpr uint32_t kPxBytes = kTile * 16;  // 128 point-extra rows of 8 bf16 (k = 0..7)
constexpr uint64_t kWaitNs = 2000000000ull;

// ---- operand images written by the prep kernels -------------------------------------------
// W image for head h (kWRow = 160 bytes per slot): G rows (slots) x 64 B of
// W' = W*log2e/tau rounded to bf16 (64B swizzle), then G rows x 32 B of
// [b'_hi, b'_lo, 1, 1, 0...] (32B swizzle), then G rows x 64 B of the residual
// W' - bf16(W') rounded to bf16 (64B swizzle).  The statistics and slice passes
// use both halves of W' (their lse, tokens and weight sums then carry no
// systematic per-slot rounding of the weights); the deslice uses the first half.
constexpr uint32_t kWRow = 160;
__device__ __forceinline__ uint32_t off_sw64(int row, int k) {  // k in [0, 32)
  const int chunk = k >> 3;
  return (uint32_t)((row >> 3) * 512 + (row & 7) * 64 + ((chunk ^ ((row & 7) >> 1)) << 4) + (k & 7) * 2);
}
__device__ __forceinline__ uint32_t off_sw32(int row, int k) {  // k in [0, 16)
  const int chunk = k >> 3;
  return (uint32_t)((row >> 3) * 256 + (row & 7) * 32 + ((chunk ^ ((row & 7) >> 2)) << 4) + (k & 7) * 2);
}
// Z' image for (b,h): blocks of 64 slots, each 32 rows (channels) x 128 B (128B swizzle).
__device__ __forceinline__ uint32_t off_z(int c, int g) {
  const int kb = g >> 6, w = g & 63;
  return (uint32_t)(kb * 4096 + (c >> 3) * 1024 + (c & 7) * 128 + (((w >> 3) ^ (c & 7)) << 4) + (w & 7) * 2);
}

// Slots [G, Gp) pad the image to whole 128-slot blocks: W' = 0 and b' = -1e30, so
// their logits are -1e30 and their weights exactly 0 in every pass.
// Thread (h, q, g): for q < 4 the 16-byte pieces of channels [8q, 8q + 8) of slot g
// in both halves of W'; for q = 4 the slot's extra row.  Consecutive threads take
// consecutive slots, so the reads of W [H, d, G] coalesce.
__global__ void k_prep_w(const float* __restrict__ W, const float* __restrict__ bias, const float* __restrict__ tau,
                         uint8_t* __restrict__ img, int H, int G, int Gp, uint32_t* status) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (int64_t)H * 5 * Gp) return;
  const int g = (int)(i % Gp);
  const int q = (int)((i / Gp) % 5);
  const int h = (int)(i / ((int64_t)5 * Gp));
  const float t = tau[h];
  if (!(t > 0.f && t < INFINITY)) {
    atomicCAS(status, 0u, (uint32_t)FS_ERR_BAD_TAU);
    return;
  }
  const float scale = kLog2e / t;
  const bool real = g < G;
  uint8_t* base = img + (size_t)h * Gp * kWRow;
  if (q < 4) {
    uint32_t hi[4], lo[4];
#pragma unroll
    for (int e = 0; e < 4; e++) {
      const int k = 8 * q + 2 * e;
      const float w0 = real ? W[((int64_t)h * kD + k) * G + g] * scale : 0.f;
      const float w1 = real ? W[((int64_t)h * kD + k + 1) * G + g] * scale : 0.f;
      const uint32_t p = pack_bf16(w0, w1);
      hi[e] = p;
      lo[e] = pack_bf16(w0 - __uint_as_float(p << 16), w1 - __uint_as_float(p & 0xFFFF0000u));
    }
    const uint32_t off = off_sw64(g, 8 * q);
    *reinterpret_cast<uint4*>(base + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
    *reinterpret_cast<uint4*>(base + (size_t)Gp * 96 + off) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
    return;
  }
  // The extra row [b'_hi, b'_lo, 1, 1, 1, 0 ...]; k = 2, 3, 4 multiply the three bf16
  // parts of the point side's -lse2 (zero in the statistics pass).
  const float b2 = real ? bias[(int64_t)h * G + g] * scale : -1e30f;
  const uint32_t bp = pack_bf16(b2, 0.f) & 0xFFFFu;
  const float bhi = __uint_as_float(bp << 16);
  const uint32_t blo = pack_bf16(b2 - bhi, 0.f) & 0xFFFFu;
  uint8_t* ep = base + (size_t)Gp * 64;
  *reinterpret_cast<uint4*>(ep + off_sw32(g, 0)) = make_uint4(bp | (blo << 16), 0x3F803F80u, 0x3F80u, 0u);
  *reinterpret_cast<uint4*>(ep + off_sw32(g, 8)) = make_uint4(0u, 0u, 0u, 0u);
}

// Padding slots [G, Gp) get zero rows (their weights are 0, and 0 * 0 stays 0).
__global__ void k_prep_z(const float* __restrict__ zp, uint8_t* __restrict__ img, int64_t BH, int G, int Gp) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t total = BH * Gp * kD;
  if (i >= total) return;
  const int c = (int)(i % kD);
  const int g = (int)((i / kD) % Gp);
  const int64_t bh = i / ((int64_t)kD * Gp);
  __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(img + (size_t)bh * Gp * 64);
  out[off_z(c, g) / 2] = __float2bfloat16_rn(g < G ? zp[(bh * G + g) * kD + c] : 0.f);
}

// Z-layout image (blocks of 64 slots, 32 channel rows x 128 B, 128B swizzle) of
// t [BH][G][tstride] per (b,h): the bf16 half, then the residual half (Gp*128 bytes
// per (b,h)); padding slots [G, Gp) are zero.
__global__ void k_prep_z2(const float* __restrict__ t, int tstride, uint8_t* __restrict__ img, int64_t BH, int G,
                          int Gp) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= BH * Gp * kD) return;
  const int c = (int)(i % kD);
  const int g = (int)((i / kD) % Gp);
  const int64_t bh = i / ((int64_t)kD * Gp);
  const float v = g < G ? t[(bh * G + g) * tstride + c] : 0.f;
  __nv_bfloat16* hp = reinterpret_cast<__nv_bfloat16*>(img + (size_t)bh * Gp * 128);
  __nv_bfloat16* lp = reinterpret_cast<__nv_bfloat16*>(img + (size_t)bh * Gp * 128 + (size_t)Gp * 64);
  const __nv_bfloat16 hi = __float2bfloat16_rn(v);
  hp[off_z(c, g) / 2] = hi;
  lp[off_z(c, g) / 2] = __float2bfloat16_rn(v - __bfloat162float(hi));
}

// ---- shared pieces -------------------------------------------------------------------------
struct Work {
  int64_t bh;      // batch * H + head
  int64_t tile0;   // first point tile of this CTA
  int ntiles;      // number of point tiles (the host keeps all point indices below 2^31)
};

// Tile i and slot block c of block q = i * nb + c, kept up to date while q walks
// with a fixed stride, so that no loop divides by the runtime block count (a
// 64-bit division per block cost as much as a block's exponentials).
struct BlockPos {
  int i, c;
  __device__ __forceinline__ BlockPos(int q0, int nb) : i(0), c(q0) {
    while (c >= nb) { c -= nb; ++i; }
  }
  __device__ __forceinline__ void step(int by, int nb) {
    c += by;
    while (c >= nb) { c -= nb; ++i; }
  }
};

// CTA (split p of unit bh) processes a contiguous range of point tiles.
__device__ __forceinline__ Work work_of(int64_t N, int splits, int p, int64_t bh) {
  Work w;
  w.bh = bh;
  const int64_t tiles = (N + kTile - 1) / kTile;
  w.tile0 = tiles * p / splits;
  w.ntiles = (int)(tiles * (p + 1) / splits - w.tile0);
  return w;
}

// The constant point-side extra block: every row [1, 1, 0 x 14] (32B swizzle).
__device__ __forceinline__ void write_const_extra(uint8_t* ex) {
  for (int r = threadIdx.x; r < kTile; r += blockDim.x) {
    const uint32_t base = smem_u32(ex) + (uint32_t)((r >> 3) * 256 + (r & 7) * 32);
    const uint32_t sw = (uint32_t)((r & 7) >> 2);
    st_shared_v4(base + ((0u ^ sw) << 4), 0x3F803F80u, 0u, 0u, 0u);
    st_shared_v4(base + ((1u ^ sw) << 4), 0u, 0u, 0u, 0u);
  }
}

// Descriptors of the two kinds of point-side extra block: the constant one
// (32B swizzle) and the per-tile one loaded by TMA (no swizzle; the k = 0..7
// core matrices at px, the zero k = 8..15 half kPxBytes further on).
__device__ __forceinline__ uint64_t const_extra_desc(uint32_t ex_s) { return sdesc(ex_s, 16, 256, kSw32); }
__device__ __forceinline__ uint64_t point_extra_desc(uint32_t px_s) { return sdesc(px_s, kPxBytes, 128, 0); }
__device__ __forceinline__ void zero_smem(uint8_t* p, uint32_t bytes) {
  for (uint32_t o = threadIdx.x * 16; o < bytes; o += blockDim.x * 16) st_shared_v4(smem_u32(p) + o, 0u, 0u, 0u, 0u);
}

// Base-2 logits of 128 points x 128 slots (chunk c of the W image) into TMEM.
//   point_major: A = points (x tile), B = slots (W);  else A = slots, B = points.
//   xe: descriptor of the point-side extra block.
//   wl_img: the residual half of W' (0: bf16 W' only, K = 48; else K = 80).
//   xr_s: the residual half of x, fp32 inputs (0: none; else two more K-steps, x_r W'_hi).
__device__ __forceinline__ void issue_logits(uint32_t tmem_d, uint32_t x_s, uint64_t xe, uint32_t w_img,
                                             uint32_t we_img, uint32_t wl_img, int c, bool point_major,
                                             uint32_t xr_s = 0) {
  constexpr uint32_t idesc = idesc_bf16(128, kGC, false, false);
  const uint32_t wc = w_img + (uint32_t)c * kGC * 64;
  const uint32_t wec = we_img + (uint32_t)c * kGC * 32;
  const uint64_t x0 = sdesc(x_s, 16, 512, kSw64), x1 = sdesc(x_s + 32, 16, 512, kSw64);
  const uint64_t w0 = sdesc(wc, 16, 512, kSw64), w1 = sdesc(wc + 32, 16, 512, kSw64);
  const uint64_t we = sdesc(wec, 16, 256, kSw32);
  if (point_major) {
    mma_ss_w(tmem_d, x0, w0, idesc, 0);
    mma_ss_w(tmem_d, x1, w1, idesc, 1);
  } else {
    mma_ss_w(tmem_d, w0, x0, idesc, 0);
    mma_ss_w(tmem_d, w1, x1, idesc, 1);
  }
  if (wl_img) {
    const uint32_t wlc = wl_img + (uint32_t)c * kGC * 64;
    const uint64_t l0 = sdesc(wlc, 16, 512, kSw64), l1 = sdesc(wlc + 32, 16, 512, kSw64);
    if (point_major) {
      mma_ss_w(tmem_d, x0, l0, idesc, 1);
      mma_ss_w(tmem_d, x1, l1, idesc, 1);
    } else {
      mma_ss_w(tmem_d, l0, x0, idesc, 1);
      mma_ss_w(tmem_d, l1, x1, idesc, 1);
    }
  }
  if (xr_s) {
    const uint64_t r0 = sdesc(xr_s, 16, 512, kSw64), r1 = sdesc(xr_s + 32, 16, 512, kSw64);
    if (point_major) {
      mma_ss_w(tmem_d, r0, w0, idesc, 1);
      mma_ss_w(tmem_d, r1, w1, idesc, 1);
    } else {
      mma_ss_w(tmem_d, w0, r0, idesc, 1);
      mma_ss_w(tmem_d, w1, r1, idesc, 1);
    }
  }
  if (point_major)
    mma_ss_w(tmem_d, xe, we, idesc, 1);
  else
    mma_ss_w(tmem_d, we, xe, idesc, 1);
}

// fp32 point tensors -> bf16 hi and residual lo tensors of the same layout (v = hi + lo
// to ~2^-16 relative): the tensor-core path's operands for fp32 inputs.
__global__ void k_split_bf16(const float* __restrict__ v, __nv_bfloat16* __restrict__ hi,
                             __nv_bfloat16* __restrict__ lo, int64_t n) {
  const int64_t i = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) * 4;
  if (i >= n) return;
  const float4 a = *reinterpret_cast<const float4*>(v + i);
  const float e[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
  for (int k = 0; k < 4; k++) {
    const __nv_bfloat16 h = __float2bfloat16_rn(e[k]);
    hi[i + k] = h;
    lo[i + k] = __float2bfloat16_rn(e[k] - __bfloat162float(h));
  }
}

// Producer-side bulk loads of an image into smem (pieces of at most 32 KB).
__device__ __forceinline__ void load_images(uint8_t* dst, const uint8_t* src, uint32_t bytes, uint64_t* bar) {
  constexpr uint32_t kPiece = 32768;
  for (uint32_t off = 0; off < bytes; off += kPiece) {
    const uint32_t n = (bytes - off) < kPiece ? (bytes - off) : kPiece;
    bulk_load(dst + off, src + off, n, bar);
  }
}

// 2^t for 32 log2-weights -> 16 bf16x2 words.
__device__ __forceinline__ void weights32(const uint32_t (&v)[32], uint32_t (&p)[16]) {
#pragma unroll
  for (int k = 0; k < 16; k++) p[k] = pack_bf16(ex2(__uint_as_float(v[2 * k])), ex2(__uint_as_float(v[2 * k + 1])));
}

// 2^t for 32 log2-weights -> the bf16 pairs (hi) and the bf16 pairs of the
// residuals w - hi (lo): w = hi + lo to ~2^-16 relative.
__device__ __forceinline__ void weights32_hilo(const uint32_t (&v)[32], uint32_t (&hi)[16], uint32_t (&lo)[16]) {
#pragma unroll
  for (int k = 0; k < 16; k++) {
    const float w0 = ex2(__uint_as_float(v[2 * k])), w1 = ex2(__uint_as_float(v[2 * k + 1]));
    const uint32_t p = pack_bf16(w0, w1);
    const float h0 = __uint_as_float(p << 16), h1 = __uint_as_float(p & 0xFFFF0000u);
    hi[k] = p;
    lo[k] = pack_bf16(w0 - h0, w1 - h1);
  }
}

// The 128 log2-weights of one TMEM lane of an S buffer -> bf16 weights written back
// in place, packed in pairs, into the first 64 columns, in two halves: columns
// [64 h, 64 h + 64) -> packed weights in columns [32 h, 32 h + 32), which this
// thread has already read.
__device__ __forceinline__ void weights_in_halves(uint32_t tS) {
#pragma unroll 1
  for (int half = 0; half < 2; half++) {
    uint32_t v0[32], v1[32];
    tmem_ld32(tS + half * 64, v0);
    tmem_ld32(tS + half * 64 + 32, v1);
    tmem_wait_ld2(v0, v1);
    uint32_t pk0[16], pk1[16];
    weights32(v0, pk0);
    weights32(v1, pk1);
    tmem_st16(tS + half * 32, pk0);
    tmem_st16(tS + half * 32 + 16, pk1);
  }
}

// One 64-slot half of the row: the log2-weights in columns [0, 64) from tS -> bf16
// weights packed in pairs into columns [0, 32) from tS, which this thread has read.
__device__ __forceinline__ void weights_half(uint32_t tS) {
  uint32_t v0[32], v1[32];
  tmem_ld32(tS, v0);
  tmem_ld32(tS + 32, v1);
  tmem_wait_ld2(v0, v1);
  uint32_t pk0[16], pk1[16];
  weights32(v0, pk0);
  weights32(v1, pk1);
  tmem_st16(tS, pk0);
  tmem_st16(tS + 16, pk1);
}

// One 64-column half with split products: the log2-weights in columns [0, 64) from tS
// -> the bf16 weights packed in pairs into columns [0, 32) and the bf16 pairs of
// their residuals into [32, 64).  The whole half is in registers before the first
// store, so the stores may land on columns not yet converted.
__device__ __forceinline__ void weights_hilo_half(uint32_t tS) {
  uint32_t v0[32], v1[32];
  tmem_ld32(tS, v0);
  tmem_ld32(tS + 32, v1);
  tmem_wait_ld2(v0, v1);
  uint32_t hi[16], lo[16];
  weights32_hilo(v0, hi, lo);
  tmem_st16(tS, hi);
  tmem_st16(tS + 32, lo);
  weights32_hilo(v1, hi, lo);
  tmem_st16(tS + 16, hi);
  tmem_st16(tS + 48, lo);
}

// The weight helpers above, plus acc += sum over the block's 128 slots of w_g ds[g]
// (ds: the block's slice of a per-slot array in shared memory; every lane reads
// the same address, a broadcast).  The backward of the slice needs this sum for
// its delta (the dS term).
__device__ __forceinline__ void weights32_ds(const uint32_t (&v)[32], uint32_t (&p)[16], const float* ds,
                                             float& acc) {
  const float4* d4 = reinterpret_cast<const float4*>(ds);
#pragma unroll
  for (int k = 0; k < 8; k++) {
    const float4 q = d4[k];
    const float w0 = ex2(__uint_as_float(v[4 * k])), w1 = ex2(__uint_as_float(v[4 * k + 1]));
    const float w2 = ex2(__uint_as_float(v[4 * k + 2])), w3 = ex2(__uint_as_float(v[4 * k + 3]));
    acc = fmaf(w0, q.x, acc);
    acc = fmaf(w1, q.y, acc);
    acc = fmaf(w2, q.z, acc);
    acc = fmaf(w3, q.w, acc);
    p[2 * k] = pack_bf16(w0, w1);
    p[2 * k + 1] = pack_bf16(w2, w3);
  }
}
__device__ __forceinline__ void weights32_hilo_ds(const uint32_t (&v)[32], uint32_t (&hi)[16], uint32_t (&lo)[16],
                                                  const float* ds, float& acc) {
  const float4* d4 = reinterpret_cast<const float4*>(ds);
#pragma unroll
  for (int k = 0; k < 8; k++) {
    const float4 q = d4[k];
    float w[4];
#pragma unroll
    for (int e = 0; e < 4; e++) w[e] = ex2(__uint_as_float(v[4 * k + e]));
    acc = fmaf(w[0], q.x, acc);
    acc = fmaf(w[1], q.y, acc);
    acc = fmaf(w[2], q.z, acc);
    acc = fmaf(w[3], q.w, acc);
#pragma unroll
    for (int e = 0; e < 2; e++) {
      const uint32_t pk = pack_bf16(w[2 * e], w[2 * e + 1]);
      hi[2 * k + e] = pk;
      lo[2 * k + e] = pack_bf16(w[2 * e] - __uint_as_float(pk << 16), w[2 * e + 1] - __uint_as_float(pk & 0xFFFF0000u));
    }
  }
}
__device__ __forceinline__ void weights_in_halves_ds(uint32_t tS, const float* ds, float& acc) {
#pragma unroll 1
  for (int half = 0; half < 2; half++) {
    uint32_t v0[32], v1[32];
    tmem_ld32(tS + half * 64, v0);
    tmem_ld32(tS + half * 64 + 32, v1);
    tmem_wait_ld2(v0, v1);
    uint32_t pk0[16], pk1[16];
    weights32_ds(v0, pk0, ds + half * 64, acc);
    weights32_ds(v1, pk1, ds + half * 64 + 32, acc);
    tmem_st16(tS + half * 32, pk0);
    tmem_st16(tS + half * 32 + 16, pk1);
  }
}
// weights_hilo_half with the sum over the half's 64 slots.
__device__ __forceinline__ void weights_hilo_half_ds(uint32_t tS, const float* ds, float& acc) {
  uint32_t v0[32], v1[32];
  tmem_ld32(tS, v0);
  tmem_ld32(tS + 32, v1);
  tmem_wait_ld2(v0, v1);
  uint32_t hi[16], lo[16];
  weights32_hilo_ds(v0, hi, lo, ds, acc);
  tmem_st16(tS, hi);
  tmem_st16(tS + 32, lo);
  weights32_hilo_ds(v1, hi, lo, ds + 32, acc);
  tmem_st16(tS + 16, hi);
  tmem_st16(tS + 48, lo);
}

// A point-extra row [1, 1, -v_1, -v_2, -v_3, 0, 0, 0] (bf16): v = v_1 + v_2 + v_3 in
// three bf16 parts, which hold v's 24 significant bits, so that the row adds -v to
// fp32 precision against a slot side [.., .., 1, 1, 1, 0 ...].  (Two parts would
// leave an error of ~2^-17 |v|: as -lse2, a per-point error of the weights'
// normalisation, which the softmax backward's cancellation amplifies in dtau.)
__device__ __forceinline__ uint4 extra_row3(float nv) {
  const __nv_bfloat16 p1 = __float2bfloat16_rn(nv);
  const float r1 = nv - __bfloat162float(p1);
  const __nv_bfloat16 p2 = __float2bfloat16_rn(r1);
  const __nv_bfloat16 p3 = __float2bfloat16_rn(r1 - __bfloat162float(p2));
  return make_uint4(0x3F803F80u, (uint32_t)__bfloat16_as_ushort(p1) | ((uint32_t)__bfloat16_as_ushort(p2) << 16),
                    (uint32_t)__bfloat16_as_ushort(p3), 0u);
}

// Point-extra rows [1, 1, -lse2 in three parts, 0, 0, 0] from lse [B,H,N] (natural
// log) into px [B*H, Np, 8]; padded points (n >= N) get -1e30 so that their weights
// vanish.
__global__ void k_prep_px(const float* __restrict__ lse, uint4* __restrict__ px, int64_t BH, int64_t N, int64_t Np) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= BH * Np) return;
  const int64_t bh = i / Np, n = i % Np;
  px[i] = extra_row3(n < N ? -lse[bh * N + n] * kLog2e : -1e30f);
}

// ---- host side -------------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// 3-D view of a [B, N, C] bf16 tensor; box = (box_c channels, 128 points, 1).
bool make_point_map(CUtensorMap* map, const void* ptr, const Shape& s, int box_c, CUtensorMapSwizzle sw) {
  auto fn = encode_fn();
  if (!fn) return false;
  const uint64_t C = (uint64_t)s.H * s.d;
  cuuint64_t dims[3] = {C, (cuuint64_t)s.N, (cuuint64_t)s.B};
  cuuint64_t strides[2] = {C * 2, (cuuint64_t)s.N * C * 2};
  cuuint32_t box[3] = {(cuuint32_t)box_c, (cuuint32_t)kTile, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 2-D view of the point-extra rows [B*H*Np, 8] bf16; box = (8, 128 points).
bool make_px_map(CUtensorMap* map, const void* ptr, int64_t BH, int64_t Np) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {8, (cuuint64_t)(BH * Np)};
  cuuint64_t strides[1] = {16};
  cuuint32_t box[2] = {8, (cuuint32_t)kTile};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The tensor-core kernels see G rounded up to whole 128-slot blocks (padding slots
// carry weight 0); outputs keep the caller's G.
Shape tc_padded(const Shape& s) {
  Shape r = s;
  r.G = (s.G + kGC - 1) / kGC * kGC;
  return r;
}

size_t w_image_bytes(const Shape& s) { return (size_t)s.H * s.G * kWRow; }
// Z' image of the forward's deslice; fp32 inputs carry z' as hi and residual halves.
size_t z_image_bytes(const Shape& s) { return (size_t)s.BH() * s.G * (s.dtype == FS_F32 ? 128 : 64); }
int64_t padded_n(const Shape& s) { return (s.N + kTile - 1) / kTile * kTile; }
size_t px_bytes(const Shape& s) { return (size_t)s.BH() * padded_n(s) * 16; }

// Point splits per work unit for one-CTA-per-SM kernels: the split count P that
// minimises the makespan in units of one unit's work, ceil(units * P / SMs) / P
// (whole waves of CTAs), smallest P on ties; at most one split per point tile.
int point_splits(const Shape& s, int units) {
  const int64_t tiles = (s.N + kTile - 1) / kTile;
  const int64_t sms = num_sms();
  if (units < 1) units = 1;
  int64_t best = 1;
  double best_t = 1e30;
  for (int64_t p = 1; p <= 2 * sms && p <= tiles; p++) {
    const double t = (double)((units * p + sms - 1) / sms) / (double)p;
    if (t < best_t - 1e-12) {
      best_t = t;
      best = p;
    }
  }
  return (int)best;
}

// rows x cols floats from src (row pitch spitch floats) to dst (row pitch dpitch
// floats): a slot range's slice of W [H, d, G], bias [H, G] or a per-slot tensor.
cudaError_t copy_rows(float* dst, int64_t dpitch, const float* src, int64_t spitch, int64_t cols, int64_t rows,
                      cudaStream_t st) {
  return cudaMemcpy2DAsync(dst, (size_t)dpitch * sizeof(float), src, (size_t)spitch * sizeof(float),
                           (size_t)cols * sizeof(float), (size_t)rows, cudaMemcpyDeviceToDevice, st);
}

constexpr size_t kMaxSmem = 232448;  // opt-in shared memory per block on sm_103
template <typename K>
cudaError_t set_smem(K kernel, size_t bytes) {
  return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

// W image of the padded shape sp (sp.G = G rounded up) from W [H, d, G].
cudaError_t prep_w(const Shape& sp, int G, const float* W, const float* bias, const float* tau, uint8_t* img,
                   uint32_t* status, cudaStream_t st) {
  const int64_t n = (int64_t)sp.H * 5 * sp.G;
  k_prep_w<<<(unsigned)((n + 127) / 128), 128, 0, st>>>(W, bias, tau, img, sp.H, G, sp.G, status);
  return cudaGetLastError();
}

}  // namespace
}  // namespace fs
