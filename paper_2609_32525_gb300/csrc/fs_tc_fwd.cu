// Tensor-core forward path for bf16 inputs on sm_103a (tcgen05 + TMEM + TMA).
//
// The three streaming passes of the paper's G-blocked family (Appendix G.1):
//   k_stats   : per point and head, lse_n = log sum_g exp(a_ng)        (point-owned)
//   k_slice   : per slot, U_g = sum_n w_ng f_n and S_g = sum_n w_ng     (slot-owned,
//               split over points; the partials are summed in a fixed order after)
//   k_deslice : per point, out_n = sum_g w_ng z'_g                      (point-owned)
// w is recomputed tile by tile in every pass and never leaves the SM.
//
// Every pass forms the logits of a 128-point tile against a chunk of GC slots
// with one tcgen05.mma chain (M = 128 points, N = GC slots, K = 48):
//   A = [ x (32 bf16) | 1, 1, -lse_hi, -lse_lo, 0.. ]     (per point)
//   B = [ W*log2e/tau (32) | beta'_hi, beta'_lo, 1, 1, 0.. ]  (per slot)
// so the accumulator already holds a2 - lse2 = log2 of the slice weight (the
// bias and the normaliser ride on the tensor core; lse2 and beta' are split
// into two bf16 halves to keep them near fp32 accurate).  The stats pass uses
// A = [x | 1, 1, 0, 0] and keeps a running max / sum in registers.
//
// CTA layout (384 threads): warp 0 issues TMA / bulk copies, warp 1 owns the
// TMEM allocation and issues every tcgen05.mma from one lane, warps 4..11 form
// two softmax warpgroups that split the columns of every chunk: thread r of a
// warpgroup owns TMEM lane r = point r of the tile (tcgen05.ld 32x32b), so
// every SM sub-partition runs two softmax warps.  Warps 2, 3 idle.  All waits are bounded (2 s): a wait
// that gives up flags FS_ERR_TIMEOUT in the status word and the CTA drains its
// in-flight copies and MMAs, frees TMEM and exits.
//
// Shared-memory operand layouts (all bases 1024-byte aligned):
//   x tile      K-major, 64 B rows, 64B swizzle (TMA)          128 x 32
//   A extra     K-major, 32 B rows, 32B swizzle (threads)      128 x 16
//   W' chunk    K-major, 64 B rows, 64B swizzle (prep image)    GC x 32
//   B extra     K-major, 32 B rows, 32B swizzle (prep image)    GC x 16
//   Z' (deslice B)  K-major rows = channels, 128 B rows, 128B swizzle
//   E (slice A)     MN-major (slots contiguous), 128B swizzle
//   [F | 1] (slice B)  MN-major, three 16-channel blocks, 32B swizzle (TMA)
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
constexpr int kD = 32;            // head width of the tensor-core path
constexpr int kSoftmaxWarp0 = 4;  // warps 4..11: two softmax warpgroups
constexpr int kStages = 3;        // x-tile pipeline depth (stats / deslice)
constexpr int kSliceStages = 3;   // slice pipeline depth
constexpr uint32_t kXBytes = kTile * 64;    // 128 points x 32 bf16
constexpr uint32_t kXeBytes = kTile * 32;   // 128 points x 16 bf16
constexpr uint32_t kFBlock = kTile * 32;    // 128 points x 16 channels
constexpr int kSliceRange = 512;            // slots per slice CTA at most

// ---- operand images written by the prep kernel -------------------------------------------
// W image for head h: G rows (slots) x 64 B of W*log2e/tau (64B swizzle), then
// G rows x 32 B of [beta'_hi, beta'_lo, 1, 1, 0...] (32B swizzle).
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

__global__ void k_prep_w(const float* __restrict__ W, const float* __restrict__ bias, const float* __restrict__ tau,
                         uint8_t* __restrict__ img, int H, int G, uint32_t* status) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t total = (int64_t)H * G;
  if (i >= total) return;
  const int h = (int)(i / G), g = (int)(i % G);
  const float t = tau[h];
  if (!(t > 0.f && t < INFINITY)) {
    atomicCAS(status, 0u, 5u);
    return;
  }
  const float scale = kLog2e / t;
  uint8_t* base = img + (size_t)h * G * 96;
  __nv_bfloat16* wp = reinterpret_cast<__nv_bfloat16*>(base);
  for (int k = 0; k < kD; k++)
    wp[off_sw64(g, k) / 2] = __float2bfloat16_rn(W[((int64_t)h * kD + k) * G + g] * scale);
  __nv_bfloat16* ep = reinterpret_cast<__nv_bfloat16*>(base + (size_t)G * 64);
  const float b2 = bias[(int64_t)h * G + g] * scale;
  const __nv_bfloat16 hi = __float2bfloat16_rn(b2);
  const __nv_bfloat16 lo = __float2bfloat16_rn(b2 - __bfloat162float(hi));
  const __nv_bfloat16 one = __float2bfloat16_rn(1.f), zero = __float2bfloat16_rn(0.f);
  for (int k = 0; k < 16; k++) {
    __nv_bfloat16 v = zero;
    if (k == 0) v = hi;
    else if (k == 1) v = lo;
    else if (k == 2 || k == 3) v = one;
    ep[off_sw32(g, k) / 2] = v;
  }
}

__global__ void k_prep_z(const float* __restrict__ zp, uint8_t* __restrict__ img, int64_t BH, int G) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t total = BH * G * kD;
  if (i >= total) return;
  const int c = (int)(i % kD);
  const int g = (int)((i / kD) % G);
  const int64_t bh = i / ((int64_t)kD * G);
  __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(img + (size_t)bh * G * 64);
  out[off_z(c, g) / 2] = __float2bfloat16_rn(zp[i]);
}

// ---- shared pieces of the three streaming kernels ----------------------------------------------
struct Work {
  int64_t bh;      // batch * H + head
  int64_t tile0;   // first point tile of this CTA
  int64_t ntiles;  // number of point tiles
};

// CTA (split p of unit bh) processes a contiguous range of point tiles.
__device__ __forceinline__ Work work_of(int64_t N, int splits) {
  Work w;
  w.bh = blockIdx.y;
  const int64_t tiles = (N + kTile - 1) / kTile;
  const int p = blockIdx.x;
  w.tile0 = tiles * p / splits;
  w.ntiles = tiles * (p + 1) / splits - w.tile0;
  return w;
}

// Row r of the per-tile A extra block: [1, 1, -l_hi, -l_lo, 0 x 12] (32B swizzle).
__device__ __forceinline__ void write_a_extra(uint8_t* xe, int r, float l2) {
  const __nv_bfloat16 hi = __float2bfloat16_rn(l2);
  const __nv_bfloat16 lo = __float2bfloat16_rn(l2 - __bfloat162float(hi));
  const uint32_t one = 0x3F80u;
  const uint32_t w0 = one | (one << 16);
  const uint32_t nhi = (uint32_t)__bfloat16_as_ushort(__hneg(hi));
  const uint32_t nlo = (uint32_t)__bfloat16_as_ushort(__hneg(lo));
  const uint32_t w1 = nhi | (nlo << 16);
  const uint32_t base = smem_u32(xe) + (uint32_t)((r >> 3) * 256 + (r & 7) * 32);
  const uint32_t sw = (uint32_t)((r & 7) >> 2);
  st_shared_v4(base + ((0u ^ sw) << 4), w0, w1, 0u, 0u);
  st_shared_v4(base + ((1u ^ sw) << 4), 0u, 0u, 0u, 0u);
}

// Issues the K = 48 logits MMA chain for chunk `c` into TMEM column `d_col`.
template <int GC>
__device__ __forceinline__ void issue_logits(uint32_t tmem_d, uint32_t x_s, uint32_t xe_s, uint32_t w_img,
                                             uint32_t we_img, int c) {
  constexpr uint32_t idesc = idesc_bf16(128, GC, false, false);
  const uint32_t wc = w_img + (uint32_t)c * GC * 64;
  const uint32_t wec = we_img + (uint32_t)c * GC * 32;
  mma_ss(tmem_d, sdesc(x_s, 16, 512, kSw64), sdesc(wc, 16, 512, kSw64), idesc, 0);
  mma_ss(tmem_d, sdesc(x_s + 32, 16, 512, kSw64), sdesc(wc + 32, 16, 512, kSw64), idesc, 1);
  mma_ss(tmem_d, sdesc(xe_s, 16, 256, kSw32), sdesc(wec, 16, 256, kSw32), idesc, 1);
}

// Producer-side loads of one W image (and optionally a Z' image) into smem.
__device__ __forceinline__ void load_images(uint8_t* dst, const uint8_t* src, uint32_t bytes, uint64_t* bar) {
  constexpr uint32_t kPiece = 32768;
  for (uint32_t off = 0; off < bytes; off += kPiece) {
    const uint32_t n = (bytes - off) < kPiece ? (bytes - off) : kPiece;
    bulk_load(dst + off, src + off, n, bar);
  }
}

// =========================================================================================
// Deslice: out_n = sum_g w_ng z'_g.
// smem: [W img G*96][Z' img G*64][x stages][xe stages][barriers]
// TMEM: three S buffers [0, 3*GC), O buffers [3*GC, 3*GC + 64).  The logits run
// two chunks ahead of the softmax.  The two softmax warpgroups split every
// chunk's columns: warpgroup wg reads S columns [64 wg, 64 wg + 64) and writes
// their bf16 weights back, packed in pairs, into columns [64 wg, 64 wg + 32) of
// the same buffer, which the P x Z' MMA reads as its A operand.
// =========================================================================================
constexpr int kSBuf = 3;

template <int GC>
__global__ void __launch_bounds__(kThreads, 1)
    k_deslice(const __grid_constant__ CUtensorMap xmap, const uint8_t* __restrict__ wimg,
              const uint8_t* __restrict__ zimg, const float* __restrict__ lse, __nv_bfloat16* __restrict__ out,
              int64_t N, int H, int G, int splits, uint32_t* status) {
  static_assert(GC == 128, "chunk width");
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t wbytes = (uint32_t)G * 96, zbytes = (uint32_t)G * 64;
  uint8_t* s_w = smem;
  uint8_t* s_z = s_w + wbytes;
  uint8_t* s_x = s_z + zbytes;
  uint8_t* s_xe = s_x + kStages * kXBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(s_xe + kStages * kXeBytes);
  uint64_t* wz_full = bars;
  uint64_t* x_full = bars + 1;
  uint64_t* x_empty = x_full + kStages;
  uint64_t* xe_ready = x_empty + kStages;
  uint64_t* s_full = xe_ready + kStages;
  uint64_t* p_ready = s_full + kSBuf;
  uint64_t* o_full = p_ready + kSBuf;
  uint64_t* o_free = o_full + 2;
  uint64_t* drain = o_free + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  Abort* ab = reinterpret_cast<Abort*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const Work wk = work_of(N, splits);
  const int64_t b = wk.bh / H;
  const int h = (int)(wk.bh % H);
  const int nch = G / GC;
  constexpr uint32_t kO = kSBuf * GC;  // TMEM column base of the O buffers

  if (threadIdx.x == 0) {
    mbar_init(wz_full, 1);
    for (int s = 0; s < kStages; s++) {
      mbar_init(&x_full[s], 1);
      mbar_init(&x_empty[s], 1);
      mbar_init(&xe_ready[s], 4);
    }
    for (int i = 0; i < kSBuf; i++) {
      mbar_init(&s_full[i], 1);
      mbar_init(&p_ready[i], 8);
    }
    for (int i = 0; i < 2; i++) {
      mbar_init(&o_full[i], 1);
      mbar_init(&o_free[i], 8);
    }
    mbar_init(drain, 1);
    ab->flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ------------------------------ producer ------------------------------
    if (lane == 0 && wk.ntiles > 0) {
      prefetch_tmap(&xmap);
      mbar_expect_tx(wz_full, wbytes + zbytes);
      load_images(s_w, wimg + (size_t)h * wbytes, wbytes, wz_full);
      load_images(s_z, zimg + (size_t)wk.bh * zbytes, zbytes, wz_full);
      int64_t i = 0;
      for (; i < wk.ntiles; i++) {
        const int s = (int)(i % kStages);
        if (i >= kStages && !mbar_wait(&x_empty[s], (uint32_t)(((i / kStages) - 1) & 1), ab, status)) break;
        mbar_expect_tx(&x_full[s], kXBytes);
        tma_load_3d(s_x + s * kXBytes, &xmap, h * kD, (int)((wk.tile0 + i) * kTile), (int)b, &x_full[s]);
      }
      // Drain: the newest load of each stage has landed before the CTA exits.
      for (int64_t j = (i > kStages ? i - kStages : 0); j < i; j++)
        mbar_wait(&x_full[j % kStages], (uint32_t)((j / kStages) & 1), ab, nullptr, 2000000000ull);
      mbar_wait(wz_full, 0, ab, nullptr, 2000000000ull);
    }
  } else if (warp == 1) {
    // ------------------------------ MMA issuer ------------------------------
    // One flattened sequence q = tile * nch + chunk; the logits of q+2 are issued
    // before waiting for the softmax of q, across tile boundaries.  A buffer is
    // rewritten only by an MMA issued after the P x Z' MMA that last read it, and
    // tcgen05.mma executes in issue order.
    if (lane == 0 && wk.ntiles > 0) {
      constexpr uint32_t idesc_pv = idesc_bf16(128, kD, false, false);
      const uint32_t sw = smem_u32(s_w), swe = sw + (uint32_t)G * 64, sz = smem_u32(s_z);
      const int64_t total = wk.ntiles * nch;
      auto logits = [&](int64_t qq) -> bool {
        const int64_t i = qq / nch;
        const int c = (int)(qq % nch);
        const int s = (int)(i % kStages);
        if (c == 0) {
          const uint32_t par = (uint32_t)((i / kStages) & 1);
          if (!mbar_wait(&x_full[s], par, ab, status) || !mbar_wait(&xe_ready[s], par, ab, status)) return false;
          tc_fence_after();
        }
        const int bb = (int)(qq % kSBuf);
        issue_logits<GC>(tmem + (uint32_t)bb * GC, smem_u32(s_x + s * kXBytes), smem_u32(s_xe + s * kXeBytes), sw,
                         swe, c);
        mma_commit(&s_full[bb]);
        if (c == nch - 1) mma_commit(&x_empty[s]);
        return true;
      };
      bool ok = mbar_wait(wz_full, 0, ab, status) && logits(0) && (total < 2 || logits(1));
      for (int64_t q = 0; ok && q < total; q++) {
        const int64_t i = q / nch;
        const int c = (int)(q % nch);
        const int ob = (int)(i & 1);
        const int bb = (int)(q % kSBuf);
        if (q + 2 < total && !(ok = logits(q + 2))) break;
        if (c == 0 && i >= 2 && !(ok = mbar_wait(&o_free[ob], (uint32_t)(((i >> 1) - 1) & 1), ab, status))) break;
        if (!(ok = mbar_wait(&p_ready[bb], (uint32_t)((q / kSBuf) & 1), ab, status))) break;
        tc_fence_after();
        const uint32_t tS = tmem + (uint32_t)bb * GC;
        const uint32_t tO = tmem + kO + (uint32_t)ob * kD;
#pragma unroll
        for (int k = 0; k < GC / 16; k++) {
          const int g0 = c * GC + k * 16;
          const uint32_t zaddr = sz + (uint32_t)((g0 >> 6) * 4096 + (g0 & 63) * 2);
          const uint32_t tP = tS + (uint32_t)((k >> 2) * 64 + (k & 3) * 8);
          mma_ts(tO, tP, sdesc(zaddr, 16, 1024, kSw128), idesc_pv, (c > 0 || k > 0) ? 1u : 0u);
        }
        if (c == nch - 1) mma_commit(&o_full[ob]);
      }
      // Drain every MMA issued by this thread before TMEM is freed.
      mma_commit(drain);
      mbar_wait(drain, 0, ab, nullptr, 2000000000ull);
    }
  } else if (warp >= kSoftmaxWarp0) {
    // ------------------------------ softmax warpgroups ------------------------------
    const int wg = (warp - kSoftmaxWarp0) >> 2;
    const int wq = warp & 3;  // TMEM sub-partition of this warp
    const int r = wq * 32 + lane;
    const uint32_t lane_addr = (uint32_t)(wq * 32) << 16;
    int64_t q = 0;
    bool ok = true;
    // lse of tile j, loaded two tiles ahead of its use.
    auto load_l2 = [&](int64_t j) -> float {
      const int64_t nn = (wk.tile0 + j) * kTile + r;
      return (j < wk.ntiles && nn < N) ? lse[wk.bh * N + nn] * kLog2e : 0.f;
    };
    // The A extra block of tile j carries -lse of its points; warpgroup 0 writes
    // it one tile ahead so the MMA warp can run the next tile's logits early.
    auto put_extra = [&](int64_t j, float l2) -> bool {
      const int s = (int)(j % kStages);
      if (j >= kStages && !mbar_wait(&x_empty[s], (uint32_t)(((j / kStages) - 1) & 1), ab, status)) return false;
      write_a_extra(s_xe + s * kXeBytes, r, l2);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&xe_ready[s]);
      return true;
    };
    // Output of tile t: this warpgroup's 16 channels of O -> bf16 -> global.
    auto epilogue = [&](int64_t t) -> bool {
      const int ob = (int)(t & 1);
      if (!mbar_wait(&o_full[ob], (uint32_t)((t >> 1) & 1), ab, status)) return false;
      tc_fence_after();
      uint32_t o[16];
      tmem_ld16(tmem + lane_addr + kO + (uint32_t)ob * kD + (uint32_t)wg * 16, o);
      tmem_wait_ld(o);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&o_free[ob]);
      const int64_t n = (wk.tile0 + t) * kTile + r;
      if (n < N) {
        uint4* dst = reinterpret_cast<uint4*>(out + ((b * N + n) * H + h) * kD + wg * 16);
#pragma unroll
        for (int j = 0; j < 2; j++)
          dst[j] = make_uint4(pack_bf16(__uint_as_float(o[8 * j]), __uint_as_float(o[8 * j + 1])),
                              pack_bf16(__uint_as_float(o[8 * j + 2]), __uint_as_float(o[8 * j + 3])),
                              pack_bf16(__uint_as_float(o[8 * j + 4]), __uint_as_float(o[8 * j + 5])),
                              pack_bf16(__uint_as_float(o[8 * j + 6]), __uint_as_float(o[8 * j + 7])));
      }
      return true;
    };
    float l2_next = 0.f;
    if (wg == 0 && wk.ntiles > 0) {
      const float l2_0 = load_l2(0);
      l2_next = load_l2(1);
      ok = put_extra(0, l2_0);
    }
    for (int64_t i = 0; ok && i < wk.ntiles; i++) {
      if (wg == 0 && i + 1 < wk.ntiles) {
        const float l2 = l2_next;
        l2_next = load_l2(i + 2);
        if (!(ok = put_extra(i + 1, l2))) break;
      }
      for (int c = 0; c < nch; c++, q++) {
        const int bb = (int)(q % kSBuf);
        if (!(ok = mbar_wait(&s_full[bb], (uint32_t)((q / kSBuf) & 1), ab, status))) break;
        tc_fence_after();
        const uint32_t tS = tmem + lane_addr + (uint32_t)bb * GC + (uint32_t)wg * 64;
        uint32_t v0[32], v1[32];
        tmem_ld32(tS, v0);
        tmem_ld32(tS + 32, v1);
        tmem_wait_ld2(v0, v1);
        uint32_t pk0[16], pk1[16];
#pragma unroll
        for (int j = 0; j < 16; j++) {
          pk0[j] = pack_bf16(ex2(__uint_as_float(v0[2 * j])), ex2(__uint_as_float(v0[2 * j + 1])));
          pk1[j] = pack_bf16(ex2(__uint_as_float(v1[2 * j])), ex2(__uint_as_float(v1[2 * j + 1])));
        }
        tmem_st16(tS, pk0);
        tmem_st16(tS + 16, pk1);
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&p_ready[bb]);
        // The output of the previous tile is drained after this tile's first chunk,
        // when its last P x Z' MMA has long finished.
        if (c == 0 && i > 0 && !(ok = epilogue(i - 1))) break;
      }
    }
    if (ok && wk.ntiles > 0) epilogue(wk.ntiles - 1);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

// =========================================================================================
// Statistics: lse_n = log sum_g exp(a_ng)  (natural log), written to lse[bh*N + n].
// Same logits pipeline as the deslice with A extra = [1, 1, 0, 0].  Each
// softmax warpgroup keeps a running (max, sum) over its half of every chunk;
// the halves are combined through shared memory at the end of a tile.
// =========================================================================================
template <int GC>
__global__ void __launch_bounds__(kThreads, 1)
    k_stats(const __grid_constant__ CUtensorMap xmap, const uint8_t* __restrict__ wimg, float* __restrict__ lse,
            int64_t N, int H, int G, int splits, uint32_t* status) {
  static_assert(GC == 128, "chunk width");
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t wbytes = (uint32_t)G * 96;
  uint8_t* s_w = smem;
  uint8_t* s_x = s_w + wbytes;
  uint8_t* s_xe = s_x + kStages * kXBytes;
  float2* s_ml = reinterpret_cast<float2*>(s_xe + kStages * kXeBytes);  // [2][128] warpgroup-1 partials
  uint64_t* bars = reinterpret_cast<uint64_t*>(s_ml + 2 * kTile);
  uint64_t* w_full = bars;
  uint64_t* x_full = bars + 1;
  uint64_t* x_empty = x_full + kStages;
  uint64_t* s_full = x_empty + kStages;
  uint64_t* s_free = s_full + 2;
  uint64_t* ml_full = s_free + 2;   // warpgroup 1 partials written   (per tile parity)
  uint64_t* ml_empty = ml_full + 2; // warpgroup 0 has read them
  uint64_t* drain = ml_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  Abort* ab = reinterpret_cast<Abort*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const Work wk = work_of(N, splits);
  const int64_t b = wk.bh / H;
  const int h = (int)(wk.bh % H);
  const int nch = G / GC;

  if (threadIdx.x == 0) {
    mbar_init(w_full, 1);
    for (int s = 0; s < kStages; s++) {
      mbar_init(&x_full[s], 1);
      mbar_init(&x_empty[s], 1);
    }
    for (int i = 0; i < 2; i++) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_free[i], 8);
      mbar_init(&ml_full[i], 4);
      mbar_init(&ml_empty[i], 4);
    }
    mbar_init(drain, 1);
    ab->flag = 0;
    fence_mbar_init();
  }
  // The A extra block is constant here: [1, 1, 0, 0, ...] for every row and stage.
  for (int idx = threadIdx.x; idx < kStages * kTile; idx += kThreads)
    write_a_extra(s_xe + (idx / kTile) * kXeBytes, idx % kTile, 0.f);
  fence_proxy_async_smem();
  if (warp == 1) tmem_alloc(tmem_slot, 256);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0 && wk.ntiles > 0) {
      prefetch_tmap(&xmap);
      mbar_expect_tx(w_full, wbytes);
      load_images(s_w, wimg + (size_t)h * wbytes, wbytes, w_full);
      int64_t i = 0;
      for (; i < wk.ntiles; i++) {
        const int s = (int)(i % kStages);
        if (i >= kStages && !mbar_wait(&x_empty[s], (uint32_t)(((i / kStages) - 1) & 1), ab, status)) break;
        mbar_expect_tx(&x_full[s], kXBytes);
        tma_load_3d(s_x + s * kXBytes, &xmap, h * kD, (int)((wk.tile0 + i) * kTile), (int)b, &x_full[s]);
      }
      for (int64_t j = (i > kStages ? i - kStages : 0); j < i; j++)
        mbar_wait(&x_full[j % kStages], (uint32_t)((j / kStages) & 1), ab, nullptr, 2000000000ull);
      mbar_wait(w_full, 0, ab, nullptr, 2000000000ull);
    }
  } else if (warp == 1) {
    if (lane == 0 && wk.ntiles > 0) {
      const uint32_t sw = smem_u32(s_w), swe = sw + (uint32_t)G * 64;
      bool ok = mbar_wait(w_full, 0, ab, status);
      int64_t q = 0;
      for (int64_t i = 0; ok && i < wk.ntiles; i++) {
        const int s = (int)(i % kStages);
        if (!(ok = mbar_wait(&x_full[s], (uint32_t)((i / kStages) & 1), ab, status))) break;
        tc_fence_after();
        const uint32_t xs = smem_u32(s_x + s * kXBytes), xes = smem_u32(s_xe + s * kXeBytes);
        for (int c = 0; c < nch; c++, q++) {
          if (q >= 2 && !(ok = mbar_wait(&s_free[q & 1], (uint32_t)(((q >> 1) - 1) & 1), ab, status))) break;
          tc_fence_after();
          issue_logits<GC>(tmem + (uint32_t)(q & 1) * GC, xs, xes, sw, swe, c);
          mma_commit(&s_full[q & 1]);
        }
        if (!ok) break;
        mma_commit(&x_empty[s]);
      }
      mma_commit(drain);
      mbar_wait(drain, 0, ab, nullptr, 2000000000ull);
    }
  } else if (warp >= kSoftmaxWarp0) {
    const int wg = (warp - kSoftmaxWarp0) >> 2;
    const int wq = warp & 3;
    const int r = wq * 32 + lane;
    const uint32_t lane_addr = (uint32_t)(wq * 32) << 16;
    int64_t q = 0;
    bool ok = true;
    for (int64_t i = 0; ok && i < wk.ntiles; i++) {
      const int64_t n = (wk.tile0 + i) * kTile + r;
      float m = -INFINITY, l = 0.f;
      for (int c = 0; c < nch; c++, q++) {
        if (!(ok = mbar_wait(&s_full[q & 1], (uint32_t)((q >> 1) & 1), ab, status))) break;
        tc_fence_after();
        const uint32_t tS = tmem + lane_addr + (uint32_t)(q & 1) * GC + (uint32_t)wg * (GC / 2);
        uint32_t v0[32], v1[32];
        tmem_ld32(tS, v0);
        tmem_ld32(tS + 32, v1);
        tmem_wait_ld2(v0, v1);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&s_free[q & 1]);
        // Chunk maximum as a tree of three-input maxima (short dependency chains).
        float t[22];
#pragma unroll
        for (int j = 0; j < 10; j++) {
          t[j] = max3(__uint_as_float(v0[3 * j]), __uint_as_float(v0[3 * j + 1]), __uint_as_float(v0[3 * j + 2]));
          t[10 + j] = max3(__uint_as_float(v1[3 * j]), __uint_as_float(v1[3 * j + 1]), __uint_as_float(v1[3 * j + 2]));
        }
        t[20] = max3(__uint_as_float(v0[30]), __uint_as_float(v0[31]), __uint_as_float(v1[30]));
        t[21] = fmaxf(__uint_as_float(v1[31]), m);
#pragma unroll
        for (int j = 0; j < 7; j++) t[j] = max3(t[3 * j], t[3 * j + 1], t[3 * j + 2]);
        const float mn = max3(max3(t[0], t[1], t[2]), max3(t[3], t[4], t[5]), fmaxf(t[6], t[21]));
        float acc[8];
#pragma unroll
        for (int j = 0; j < 8; j++) acc[j] = 0.f;
#pragma unroll
        for (int j = 0; j < 32; j++) {
          acc[j & 7] += ex2(__uint_as_float(v0[j]) - mn);
          acc[(j + 4) & 7] += ex2(__uint_as_float(v1[j]) - mn);
        }
        const float sum = ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
        l = l * ex2(m - mn) + sum;
        m = mn;
      }
      if (!ok) break;
      const int pb = (int)(i & 1);
      if (wg == 1) {
        if (i >= 2 && !(ok = mbar_wait(&ml_empty[pb], (uint32_t)(((i >> 1) - 1) & 1), ab, status))) break;
        s_ml[pb * kTile + r] = make_float2(m, l);
        __syncwarp();
        if (lane == 0) mbar_arrive(&ml_full[pb]);
      } else {
        if (!(ok = mbar_wait(&ml_full[pb], (uint32_t)((i >> 1) & 1), ab, status))) break;
        const float2 o = s_ml[pb * kTile + r];
        __syncwarp();
        if (lane == 0) mbar_arrive(&ml_empty[pb]);
        const float M = fmaxf(m, o.x);
        const float L = l * ex2(m - M) + o.y * ex2(o.x - M);
        if (n < N) lse[wk.bh * N + n] = (M + log2f(L)) * kLn2;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 256);
}

// =========================================================================================
// Slice (slot-owned, split over points): the G/128 slot chunks of a head are cut
// into `ranges` balanced ranges of at most 4 chunks; CTA (p, bh, r) owns range r
// and point split p: U_g = sum_n w_ng f_n, S_g = sum_n w_ng with w from lse.
// Writes part[p][bh][g][0..32] = (U_g, S_g).
// smem: [W img of the range, up to 512*96][stages: x | xe | F_lo F_hi ones][E buffers 2 x 32 KB][bars]
// TMEM: S buffers [0, 256), accumulators [256 + 48 j, ...) for M-tile j.
// Warpgroup wg writes the E rows of slots [64 wg, 64 wg + 64) of every chunk.
// =========================================================================================
constexpr uint32_t kStageBytes = kXBytes + kXeBytes + 3 * kFBlock;  // 8 + 4 + 12 KB
constexpr uint32_t kEBytes = 128 * kTile * 2;                       // 128 slots x 128 points bf16

__global__ void __launch_bounds__(kThreads, 1)
    k_slice(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ CUtensorMap fmap,
            const uint8_t* __restrict__ wimg, const float* __restrict__ lse, float* __restrict__ part, int64_t N,
            int H, int G, int splits, int ranges, uint32_t* status) {
  constexpr int GC = 128;
  const int nchunks = G / GC;
  const int rng = blockIdx.z;  // slot range
  const int c_lo = rng * nchunks / ranges, c_hi = (rng + 1) * nchunks / ranges;
  const int NCH = c_hi - c_lo;  // chunks of this CTA, 1..4
  const int GS = NCH * GC;
  const int g_base = c_lo * GC;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  constexpr uint32_t wbytes = (uint32_t)kSliceRange * 96;
  uint8_t* s_w = smem;
  uint8_t* s_st = s_w + wbytes;
  uint8_t* s_e = s_st + kSliceStages * kStageBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(s_e + 2 * kEBytes);
  uint64_t* w_full = bars;
  uint64_t* x_full = bars + 1;
  uint64_t* xe_ready = x_full + kSliceStages;
  uint64_t* st_empty = xe_ready + kSliceStages;
  uint64_t* s_full = st_empty + kSliceStages;
  uint64_t* s_free = s_full + 2;
  uint64_t* e_ready = s_free + 2;
  uint64_t* e_free = e_ready + 2;
  uint64_t* acc_full = e_free + 2;
  uint64_t* drain = acc_full + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  Abort* ab = reinterpret_cast<Abort*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const Work wk = work_of(N, splits);
  const int64_t b = wk.bh / H;
  const int h = (int)(wk.bh % H);

  if (threadIdx.x == 0) {
    mbar_init(w_full, 1);
    for (int s = 0; s < kSliceStages; s++) {
      mbar_init(&x_full[s], 1);
      mbar_init(&xe_ready[s], 4);
      mbar_init(&st_empty[s], 1);
    }
    for (int i = 0; i < 2; i++) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_free[i], 8);
      mbar_init(&e_ready[i], 8);
      mbar_init(&e_free[i], 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(drain, 1);
    ab->flag = 0;
    fence_mbar_init();
  }
  // Constant "ones" block of every stage: row n = [1, 0 x 15] (32B swizzle).
  for (int idx = threadIdx.x; idx < kSliceStages * kTile; idx += kThreads) {
    const int s = idx / kTile, r = idx % kTile;
    const uint32_t base = smem_u32(s_st + s * kStageBytes + kXBytes + kXeBytes + 2 * kFBlock) +
                          (uint32_t)((r >> 3) * 256 + (r & 7) * 32);
    const uint32_t sw = (uint32_t)((r & 7) >> 2);
    st_shared_v4(base + ((0u ^ sw) << 4), 0x3F80u, 0u, 0u, 0u);
    st_shared_v4(base + ((1u ^ sw) << 4), 0u, 0u, 0u, 0u);
  }
  fence_proxy_async_smem();
  if (warp == 1) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      prefetch_tmap(&xmap);
      prefetch_tmap(&fmap);
      // W image rows g_base .. g_base+GS of head h: the W' part and the extra part are
      // separate row arrays in the global image (G rows each).
      mbar_expect_tx(w_full, (uint32_t)GS * 96);
      const uint8_t* src = wimg + (size_t)h * G * 96;
      load_images(s_w, src + (size_t)g_base * 64, GS * 64, w_full);
      load_images(s_w + GS * 64, src + (size_t)G * 64 + (size_t)g_base * 32, GS * 32, w_full);
      int64_t i = 0;
      for (; i < wk.ntiles; i++) {
        const int s = (int)(i % kSliceStages);
        if (i >= kSliceStages &&
            !mbar_wait(&st_empty[s], (uint32_t)(((i / kSliceStages) - 1) & 1), ab, status))
          break;
        uint8_t* st = s_st + s * kStageBytes;
        const int n0 = (int)((wk.tile0 + i) * kTile);
        mbar_expect_tx(&x_full[s], kXBytes + 2 * kFBlock);
        tma_load_3d(st, &xmap, h * kD, n0, (int)b, &x_full[s]);
        tma_load_3d(st + kXBytes + kXeBytes, &fmap, h * kD, n0, (int)b, &x_full[s]);
        tma_load_3d(st + kXBytes + kXeBytes + kFBlock, &fmap, h * kD + 16, n0, (int)b, &x_full[s]);
      }
      for (int64_t j = (i > kSliceStages ? i - kSliceStages : 0); j < i; j++)
        mbar_wait(&x_full[j % kSliceStages], (uint32_t)((j / kSliceStages) & 1), ab, nullptr, 2000000000ull);
      mbar_wait(w_full, 0, ab, nullptr, 2000000000ull);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc_sl = idesc_bf16(128, 48, true, true);
      const uint32_t sw = smem_u32(s_w), swe = sw + GS * 64;
      const int64_t total = wk.ntiles * NCH;
      auto logits = [&](int64_t qq) -> bool {
        const int64_t i = qq / NCH;
        const int c = (int)(qq % NCH);
        const int s = (int)(i % kSliceStages);
        if (c == 0) {
          const uint32_t par = (uint32_t)((i / kSliceStages) & 1);
          if (!mbar_wait(&x_full[s], par, ab, status) || !mbar_wait(&xe_ready[s], par, ab, status)) return false;
        }
        if (qq >= 2 && !mbar_wait(&s_free[qq & 1], (uint32_t)(((qq >> 1) - 1) & 1), ab, status)) return false;
        tc_fence_after();
        const uint32_t st = smem_u32(s_st + s * kStageBytes);
        issue_logits<GC>(tmem + (uint32_t)(qq & 1) * GC, st, st + kXBytes, sw, swe, c);
        mma_commit(&s_full[qq & 1]);
        return true;
      };
      bool ok = mbar_wait(w_full, 0, ab, status) && (total == 0 || logits(0));
      for (int64_t q = 0; ok && q < total; q++) {
        const int64_t i = q / NCH;
        const int c = (int)(q % NCH);
        const int s = (int)(i % kSliceStages);
        if (q + 1 < total && !(ok = logits(q + 1))) break;
        if (!(ok = mbar_wait(&e_ready[q & 1], (uint32_t)((q >> 1) & 1), ab, status))) break;
        tc_fence_after();
        const uint32_t ebase = smem_u32(s_e + (q & 1) * kEBytes);
        const uint32_t fs = smem_u32(s_st + s * kStageBytes) + kXBytes + kXeBytes;
        const uint32_t tacc = tmem + 256 + (uint32_t)c * 48;
#pragma unroll
        for (int k = 0; k < kTile / 16; k++)
          mma_ss(tacc, sdesc(ebase + (uint32_t)k * 2048, 16384, 1024, kSw128),
                 sdesc(fs + (uint32_t)k * 512, kFBlock, 256, kSw32), idesc_sl, (i > 0 || k > 0) ? 1u : 0u);
        mma_commit(&e_free[q & 1]);
        if (c == NCH - 1) mma_commit(&st_empty[s]);
      }
      if (ok) mma_commit(acc_full);
      mma_commit(drain);
      mbar_wait(drain, 0, ab, nullptr, 2000000000ull);
    }
  } else if (warp >= kSoftmaxWarp0) {
    const int wg = (warp - kSoftmaxWarp0) >> 2;
    const int wq = warp & 3;
    const int r = wq * 32 + lane;
    const uint32_t lane_addr = (uint32_t)(wq * 32) << 16;
    int64_t q = 0;
    bool ok = true;
    auto load_l2 = [&](int64_t j) -> float {
      const int64_t nn = (wk.tile0 + j) * kTile + r;
      return (j < wk.ntiles && nn < N) ? lse[wk.bh * N + nn] * kLog2e : 0.f;
    };
    auto put_extra = [&](int64_t j, float l2) -> bool {
      const int s = (int)(j % kSliceStages);
      if (j >= kSliceStages && !mbar_wait(&st_empty[s], (uint32_t)(((j / kSliceStages) - 1) & 1), ab, status))
        return false;
      write_a_extra(s_st + s * kStageBytes + kXBytes, r, l2);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&xe_ready[s]);
      return true;
    };
    float l2_next = 0.f;
    if (wg == 0 && wk.ntiles > 0) {
      const float l2_0 = load_l2(0);
      l2_next = load_l2(1);
      ok = put_extra(0, l2_0);
    }
    for (int64_t i = 0; ok && i < wk.ntiles; i++) {
      const int64_t n = (wk.tile0 + i) * kTile + r;
      const bool valid = n < N;
      if (wg == 0 && i + 1 < wk.ntiles) {
        const float l2 = l2_next;
        l2_next = load_l2(i + 2);
        if (!(ok = put_extra(i + 1, l2))) break;
      }
      for (int c = 0; c < NCH; c++, q++) {
        if (!(ok = mbar_wait(&s_full[q & 1], (uint32_t)((q >> 1) & 1), ab, status))) break;
        tc_fence_after();
        const uint32_t tS = tmem + lane_addr + (uint32_t)(q & 1) * GC + (uint32_t)wg * 64;
        uint32_t v0[32], v1[32];
        tmem_ld32(tS, v0);
        tmem_ld32(tS + 32, v1);
        tmem_wait_ld2(v0, v1);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&s_free[q & 1]);
        // w = 2^(a2 - lse2); padded points contribute nothing.
        uint32_t pk[32];
#pragma unroll
        for (int j = 0; j < 16; j++) {
          pk[j] = valid ? pack_bf16(ex2(__uint_as_float(v0[2 * j])), ex2(__uint_as_float(v0[2 * j + 1]))) : 0u;
          pk[16 + j] = valid ? pack_bf16(ex2(__uint_as_float(v1[2 * j])), ex2(__uint_as_float(v1[2 * j + 1]))) : 0u;
        }
        if (q >= 2 && !(ok = mbar_wait(&e_free[q & 1], (uint32_t)(((q >> 1) - 1) & 1), ab, status))) break;
        // E[r][g], g in this warpgroup's 64 slots: MN-major m-block wg (16 KB apart), k-group r/8.
        const uint32_t eb = smem_u32(s_e + (q & 1) * kEBytes) + (uint32_t)wg * 16384 +
                            (uint32_t)((r >> 3) * 1024 + (r & 7) * 128);
#pragma unroll
        for (int j = 0; j < 8; j++)
          st_shared_v4(eb + (((uint32_t)j ^ (uint32_t)(r & 7)) << 4), pk[4 * j], pk[4 * j + 1], pk[4 * j + 2],
                       pk[4 * j + 3]);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&e_ready[q & 1]);
      }
    }
    // Epilogue: the accumulators of this CTA's slot range -> partials
    // (warpgroup 0 the numerators U, warpgroup 1 the weight sums S).
    const int64_t BH = gridDim.y;
    if (ok && wk.ntiles > 0 && mbar_wait(acc_full, 0, ab, status)) {
      tc_fence_after();
      for (int j = 0; j < NCH; j++) {
        const int g = g_base + j * GC + r;
        float* o = part + (((int64_t)blockIdx.x * BH + wk.bh) * G + g) * (kD + 1);
        if (wg == 0) {
          uint32_t u[32];
          tmem_ld32(tmem + lane_addr + 256 + j * 48, u);
          tmem_wait_ld(u);
#pragma unroll
          for (int k = 0; k < kD; k++) o[k] = __uint_as_float(u[k]);
        } else {
          uint32_t sv[16];
          tmem_ld16(tmem + lane_addr + 256 + j * 48 + 32, sv);
          tmem_wait_ld(sv);
          o[kD] = __uint_as_float(sv[0]);
        }
      }
    } else if (ok && wk.ntiles == 0) {
      for (int j = 0; j < NCH; j++) {
        const int g = g_base + j * GC + r;
        float* o = part + (((int64_t)blockIdx.x * BH + wk.bh) * G + g) * (kD + 1);
        if (wg == 0)
          for (int k = 0; k < kD; k++) o[k] = 0.f;
        else
          o[kD] = 0.f;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
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

size_t w_image_bytes(const Shape& s) { return (size_t)s.H * s.G * 96; }
size_t z_image_bytes(const Shape& s) { return (size_t)s.BH() * s.G * 64; }

int point_splits(const Shape& s, int units) {
  const int64_t tiles = (s.N + kTile - 1) / kTile;
  int64_t p = num_sms() / (units < 1 ? 1 : units);
  if (p < 1) p = 1;
  if (p > tiles) p = tiles;
  if (p > 65535) p = 65535;
  return (int)p;
}

// Balanced ranges of at most kSliceRange/128 whole 128-slot chunks per head.
int slice_ranges(const Shape& s) {
  const int chunks = s.G / 128, per = kSliceRange / 128;
  const int r = (chunks + per - 1) / per;
  return r < 1 ? 1 : r;
}
int slice_splits(const Shape& s) { return point_splits(s, (int)(s.BH() * slice_ranges(s))); }

size_t smem_deslice(int G) { return 1024 + (size_t)G * 160 + kStages * (kXBytes + kXeBytes) + 256; }
size_t smem_stats(int G) { return 1024 + (size_t)G * 96 + kStages * (kXBytes + kXeBytes) + 2 * kTile * 8 + 256; }
size_t smem_slice() { return 1024 + (size_t)kSliceRange * 96 + kSliceStages * kStageBytes + 2 * kEBytes + 256; }

template <typename K>
cudaError_t set_smem(K kernel, size_t bytes) {
  return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

cudaError_t prep_w(const Shape& s, const float* W, const float* bias, const float* tau, uint8_t* img,
                   uint32_t* status, cudaStream_t st) {
  const int64_t n = (int64_t)s.H * s.G;
  k_prep_w<<<(unsigned)((n + 127) / 128), 128, 0, st>>>(W, bias, tau, img, s.H, s.G, status);
  return cudaGetLastError();
}

}  // namespace

bool tc_forward_supported(const Shape& s) {
  return s.dtype == FS_BF16 && s.d == kD && s.G % 128 == 0 && s.G <= 1024 && s.N >= 1 && encode_fn() != nullptr;
}

int tc_forward_launch_count(const Shape&) { return 4 /*prep_w, stats, slice, reduce*/ + 3 /*prep_w, prep_z, deslice*/; }

size_t tc_slice_partials_bytes(const Shape& s) {
  if (!tc_forward_supported(s)) return 0;
  return (size_t)slice_splits(s) * s.BH() * s.G * (kD + 1) * sizeof(float);
}
size_t tc_slice_prep_bytes(const Shape& s) { return tc_forward_supported(s) ? w_image_bytes(s) : 0; }
size_t tc_deslice_prep_bytes(const Shape& s) {
  return tc_forward_supported(s) ? align_up(w_image_bytes(s), 256) + z_image_bytes(s) : 0;
}

cudaError_t tc_stats(const Shape& s, const void* x, const float* W, const float* bias, const float* tau, float* lse,
                     void* prep, uint32_t* status, cudaStream_t st) {
  uint8_t* wimg = static_cast<uint8_t*>(prep);
  cudaError_t e = prep_w(s, W, bias, tau, wimg, status, st);
  if (e != cudaSuccess) return e;
  CUtensorMap xmap;
  if (!make_point_map(&xmap, x, s, kD, CU_TENSOR_MAP_SWIZZLE_64B)) return cudaErrorInvalidValue;
  const int P = point_splits(s, (int)s.BH());
  const size_t sm = smem_stats(s.G);
  dim3 grid((unsigned)P, (unsigned)s.BH());
  if (s.G % 128 == 0) {
    if ((e = set_smem(k_stats<128>, sm)) != cudaSuccess) return e;
    k_stats<128><<<grid, kThreads, sm, st>>>(xmap, wimg, lse, s.N, s.H, s.G, P, status);
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

cudaError_t tc_slice_fwd(const Shape& s, const void* x, const void* f, const float* W, const float* bias,
                         const float* tau, float* tokens, float* wsum, float* lse, int finalize, float* part,
                         void* prep, uint32_t* status, cudaStream_t st) {
  cudaError_t e = tc_stats(s, x, W, bias, tau, lse, prep, status, st);
  if (e != cudaSuccess) return e;
  uint8_t* wimg = static_cast<uint8_t*>(prep);
  CUtensorMap xmap, fmap;
  if (!make_point_map(&xmap, x, s, kD, CU_TENSOR_MAP_SWIZZLE_64B)) return cudaErrorInvalidValue;
  if (!make_point_map(&fmap, f, s, 16, CU_TENSOR_MAP_SWIZZLE_32B)) return cudaErrorInvalidValue;
  const int R = slice_ranges(s), P = slice_splits(s);
  dim3 grid((unsigned)P, (unsigned)s.BH(), (unsigned)R);
  const size_t sm = smem_slice();
  if ((e = set_smem(k_slice, sm)) != cudaSuccess) return e;
  k_slice<<<grid, kThreads, sm, st>>>(xmap, fmap, wimg, lse, part, s.N, s.H, s.G, P, R, status);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  return simt_reduce_tokens(s, P, part, tokens, wsum, finalize, st);
}

cudaError_t tc_deslice_fwd(const Shape& s, const void* x, const float* W, const float* bias, const float* tau,
                           const float* zp, const float* lse, void* out, void* prep, uint32_t* status,
                           cudaStream_t st) {
  uint8_t* wimg = static_cast<uint8_t*>(prep);
  uint8_t* zimg = wimg + align_up(w_image_bytes(s), 256);
  cudaError_t e = prep_w(s, W, bias, tau, wimg, status, st);
  if (e != cudaSuccess) return e;
  const int64_t nz = s.BH() * s.G * kD;
  k_prep_z<<<(unsigned)((nz + 255) / 256), 256, 0, st>>>(zp, zimg, s.BH(), s.G);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  CUtensorMap xmap;
  if (!make_point_map(&xmap, x, s, kD, CU_TENSOR_MAP_SWIZZLE_64B)) return cudaErrorInvalidValue;
  const int P = point_splits(s, (int)s.BH());
  const size_t sm = smem_deslice(s.G);
  dim3 grid((unsigned)P, (unsigned)s.BH());
  if ((e = set_smem(k_deslice<128>, sm)) != cudaSuccess) return e;
  k_deslice<128><<<grid, kThreads, sm, st>>>(xmap, wimg, zimg, lse, static_cast<__nv_bfloat16*>(out), s.N, s.H,
                                             s.G, P, status);
  return cudaGetLastError();
}

}  // namespace fs
