// SIMT fp32 kernels: every step of the coupling with fp32 FMA products and fp32
// accumulation (the paper's "ieee" dot level, Appendix G.2).  They serve every
// shape the tensor-core kernels do not cover (d != 32, G above their limits, small
// fp32 problems, the backward of fp32 inputs), and the small steps every path
// shares: the fixed-order reductions, the mixes and their backward.
//
// Ownership follows the paper's G-blocked family (Appendix G.1): a statistics
// pass per point; slot-owned split-N partial numerators and weight sums with a
// fixed-order reduction afterwards; point-owned deslice; backward as
// point-owned (input gradients, two sweeps over slots) plus slot-owned
// (parameter and token gradients) kernels.  No float atomics anywhere.
//
// Logits are formed as a2 = x . (W * log2e/tau) + beta * log2e/tau, i.e. the
// temperature-scaled logit in base-2 units, so that w = exp2(a2 - lse*log2e).
#include "fs_internal.h"

#include <cuda_bf16.h>
#include <math_constants.h>

namespace fs {
namespace {

constexpr int kThreads = 128;

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(__nv_bfloat16 v) { return __bfloat162float(v); }
// Row of D contiguous elements -> floats (16-byte vector loads).
template <int D>
__device__ __forceinline__ void load_row(const float* p, float (&v)[D]) {
  const float4* q = reinterpret_cast<const float4*>(p);
#pragma unroll
  for (int i = 0; i < D / 4; i++) {
    float4 t = q[i];
    v[4 * i] = t.x; v[4 * i + 1] = t.y; v[4 * i + 2] = t.z; v[4 * i + 3] = t.w;
  }
}
template <int D>
__device__ __forceinline__ void load_row(const __nv_bfloat16* p, float (&v)[D]) {
  const uint4* q = reinterpret_cast<const uint4*>(p);
#pragma unroll
  for (int i = 0; i < D / 8; i++) {
    uint4 t = q[i];
    const uint32_t w[4] = {t.x, t.y, t.z, t.w};
#pragma unroll
    for (int j = 0; j < 4; j++) {
      v[8 * i + 2 * j] = __uint_as_float(w[j] << 16);
      v[8 * i + 2 * j + 1] = __uint_as_float(w[j] & 0xffff0000u);
    }
  }
}
template <int D>
__device__ __forceinline__ void store_row(float* p, const float (&v)[D]) {
  float4* q = reinterpret_cast<float4*>(p);
#pragma unroll
  for (int i = 0; i < D / 4; i++) q[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
}
template <int D>
__device__ __forceinline__ void store_row(__nv_bfloat16* p, const float (&v)[D]) {
  uint4* q = reinterpret_cast<uint4*>(p);
#pragma unroll
  for (int i = 0; i < D / 8; i++) {
    uint32_t w[4];
#pragma unroll
    for (int j = 0; j < 4; j++) {
      __nv_bfloat162 t = __floats2bfloat162_rn(v[8 * i + 2 * j], v[8 * i + 2 * j + 1]);
      w[j] = *reinterpret_cast<uint32_t*>(&t);
    }
    q[i] = make_uint4(w[0], w[1], w[2], w[3]);
  }
}

__device__ __forceinline__ void set_status(uint32_t* status, uint32_t code) {
  if (status) atomicCAS(status, 0u, code);
}

// tau must be positive and finite; returns false (and flags the status word) otherwise.
__device__ __forceinline__ bool tau_ok(float t, uint32_t* status) {
  if (t > 0.f && t < CUDART_INF_F) return true;
  if (threadIdx.x == 0) set_status(status, kDevBadTau);
  return false;
}

__device__ __forceinline__ int64_t row_index(int64_t b, int64_t n, int h, int64_t N, int H) {
  return (b * N + n) * H + h;
}

// Stage GC slots of W[h] (scaled by `scale`) as sW[g][k] plus the scaled bias.  The
// rows are unpadded (16-byte aligned), so that the compute loops, in which every lane
// reads the same row, take them four floats at a time; the staging stores are then
// bank-conflicted, which costs little against the compute on each chunk.
template <int D, int GC>
__device__ __forceinline__ void stage_w(float (*sW)[D], float* sB, const float* W,
                                        const float* bias, int h, int G, int g0, float scale) {
  for (int i = threadIdx.x; i < GC * D; i += kThreads) {
    const int g = i % GC, k = i / GC;
    sW[g][k] = (g0 + g < G) ? W[((int64_t)h * D + k) * G + g0 + g] * scale : 0.f;
  }
  for (int i = threadIdx.x; i < GC; i += kThreads)
    sB[i] = (g0 + i < G) ? bias[(int64_t)h * G + g0 + i] * scale : 0.f;
}

// ---- statistics: lse per (point, head) ------------------------------------------
template <int D, typename T>
__global__ void __launch_bounds__(kThreads) k_stats(const T* __restrict__ x, const float* __restrict__ W,
                                                     const float* __restrict__ bias,
                                                     const float* __restrict__ tau, float* __restrict__ lse,
                                                     int64_t N, int H, int G, uint32_t* status) {
  constexpr int GC = 32;
  __shared__ __align__(16) float sW[GC][D];
  __shared__ float sB[GC];
  const int64_t bh = blockIdx.y;
  const int64_t b = bh / H;
  const int h = (int)(bh % H);
  if (!tau_ok(tau[h], status)) return;
  const float scale = kLog2e / tau[h];
  const int64_t n = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  const bool valid = n < N;
  float xr[D];
  if (valid) load_row<D>(x + row_index(b, n, h, N, H) * D, xr);
  else {
#pragma unroll
    for (int k = 0; k < D; k++) xr[k] = 0.f;
  }
  float m = -CUDART_INF_F, l = 0.f;
  for (int g0 = 0; g0 < G; g0 += GC) {
    __syncthreads();
    stage_w<D, GC>(sW, sB, W, bias, h, G, g0, scale);
    __syncthreads();
    const int gn = min(GC, G - g0);
    float a[GC];
    float cm = -CUDART_INF_F;
#pragma unroll
    for (int g = 0; g < GC; g++) {
      float s = sB[g];
#pragma unroll
      for (int k = 0; k < D; k++) s = fmaf(xr[k], sW[g][k], s);
      a[g] = (g < gn) ? s : -CUDART_INF_F;
      cm = fmaxf(cm, a[g]);
    }
    const float mn = fmaxf(m, cm);
    float acc = 0.f;
#pragma unroll
    for (int g = 0; g < GC; g++) acc += exp2f(a[g] - mn);
    l = l * exp2f(m - mn) + acc;
    m = mn;
  }
  if (valid) lse[bh * N + n] = (m + log2f(l)) * kLn2;
}

// ---- slice: slot-owned split-N partials ------------------------------------------
// grid (ceil(G/128), B*H, P); thread = slot.  part[p][bh][g][0..D] = (U, S).
template <int D, typename T>
__global__ void __launch_bounds__(kThreads) k_slice_partial(
    const T* __restrict__ x, const T* __restrict__ f, const float* __restrict__ W,
    const float* __restrict__ bias, const float* __restrict__ tau, const float* __restrict__ lse,
    float* __restrict__ part, int64_t B, int64_t N, int H, int G, int64_t per_split, uint32_t* status) {
  constexpr int PT = 32;
  __shared__ __align__(16) float sx[PT][D];
  __shared__ float sf[PT][D];
  __shared__ float sl[PT];
  const int g = blockIdx.x * kThreads + threadIdx.x;
  const int64_t bh = blockIdx.y;
  const int64_t b = bh / H;
  const int h = (int)(bh % H);
  const int p = blockIdx.z;
  if (!tau_ok(tau[h], status)) return;
  const float scale = kLog2e / tau[h];
  float wc[D], U[D];
  float bb = 0.f, S = 0.f;
#pragma unroll
  for (int k = 0; k < D; k++) {
    wc[k] = (g < G) ? W[((int64_t)h * D + k) * G + g] * scale : 0.f;
    U[k] = 0.f;
  }
  if (g < G) bb = bias[(int64_t)h * G + g] * scale;
  const int64_t n_begin = (int64_t)p * per_split;
  const int64_t n_end = min(N, n_begin + per_split);
  for (int64_t n0 = n_begin; n0 < n_end; n0 += PT) {
    __syncthreads();
    for (int i = threadIdx.x; i < PT * D; i += kThreads) {
      const int j = i / D, k = i % D;
      const int64_t n = n0 + j;
      float xv = 0.f, fv = 0.f;
      if (n < n_end) {
        const int64_t idx = row_index(b, n, h, N, H) * D + k;
        xv = to_f(x[idx]);
        fv = to_f(f[idx]);
      }
      sx[j][k] = xv;
      sf[j][k] = fv;
    }
    for (int i = threadIdx.x; i < PT; i += kThreads) {
      const int64_t n = n0 + i;
      sl[i] = (n < n_end) ? lse[bh * N + n] * kLog2e : CUDART_INF_F;
    }
    __syncthreads();
    // Four points at a time: their logits are independent chains; the sums take
    // the points in order.
#pragma unroll 1
    for (int j = 0; j < PT; j += 4) {
      float a[4] = {bb, bb, bb, bb};
#pragma unroll
      for (int k = 0; k < D; k++)
#pragma unroll
        for (int q = 0; q < 4; q++) a[q] = fmaf(sx[j + q][k], wc[k], a[q]);
      float w[4];
#pragma unroll
      for (int q = 0; q < 4; q++) w[q] = exp2f(a[q] - sl[j + q]);
#pragma unroll
      for (int q = 0; q < 4; q++) {
        S += w[q];
#pragma unroll
        for (int k = 0; k < D; k++) U[k] = fmaf(w[q], sf[j + q][k], U[k]);
      }
    }
  }
  if (g < G) {
    float* o = part + (((int64_t)p * B * H + bh) * G + g) * (D + 1);
#pragma unroll
    for (int k = 0; k < D; k++) o[k] = U[k];
    o[D] = S;
  }
}

// Fixed-order sum of the P partials [P, BHG, D+1], then (optionally) the
// normalisation.  The sum over splits runs in split order.  Partials hold Gs >= G
// slot rows per (b, h) (the tensor-core path pads G to whole 128-slot blocks);
// only the first G are reduced.
__global__ void k_reduce_tokens(const float* __restrict__ part, int P, int64_t BH, int G, int Gs, int D,
                                float* __restrict__ tokens, float* __restrict__ wsum, int finalize,
                                float eps) {
  // One warp per output row bh * G + g; lane l sums columns l, l + 32, l + 64 (<= D)
  // of its partial row over the splits, loads four splits ahead.
  const int64_t i = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (i >= BH * G) return;  // whole warps
  const int64_t row = (i / G) * Gs + i % G;  // its partial row
  const int64_t stride = BH * Gs * (D + 1);
  const float* src = part + row * (D + 1);
  float v[3] = {0.f, 0.f, 0.f};
#pragma unroll
  for (int j = 0; j < 3; j++) {
    const int c = lane + 32 * j;
    if (c > D) continue;
    int p = 0;
    for (; p + 4 <= P; p += 4) {
      const float a0 = src[(int64_t)p * stride + c], a1 = src[(int64_t)(p + 1) * stride + c];
      const float a2 = src[(int64_t)(p + 2) * stride + c], a3 = src[(int64_t)(p + 3) * stride + c];
      v[j] = (((v[j] + a0) + a1) + a2) + a3;
    }
    for (; p < P; p++) v[j] += src[(int64_t)p * stride + c];
  }
  const int jS = D >> 5;  // column D (the weight sum) is lane D % 32's entry jS
  const float S = __shfl_sync(0xffffffffu, jS == 0 ? v[0] : (jS == 1 ? v[1] : v[2]), D & 31);
#pragma unroll
  for (int j = 0; j < 3; j++) {
    const int c = lane + 32 * j;
    if (c < D)
      tokens[i * D + c] = finalize ? v[j] / (S + eps) : v[j];
    else if (c == D)
      wsum[i] = v[j];
  }
}

__global__ void k_finalize(float* __restrict__ tokens, const float* __restrict__ wsum, int64_t BHG,
                           int D, float eps) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= BHG * D) return;
  tokens[i] = tokens[i] / (wsum[i / D] + eps);
}

// ---- mix and its backward ------------------------------------------------------------
// out[bh][g][c] = sum_k A_h(g, k) in[bh][k][c] per (b, h), with A_h = M[h] (the mix,
// z' = M z) or A_h = M[h]^T (its backward, dz = M^T dz').
//
// A block of 8 warps owns a tile of 16 rows g x 32 channels and sweeps k in chunks of
// 64.  A and `in` chunks are staged in shared memory by cp.async, three chunks deep,
// so that two chunks' loads are in flight while one is multiplied.  Warp w takes k
// = 8w .. 8w + 7 of every chunk; each lane keeps a 4 x 4 register tile (4 rows g, 4
// channels), so that two 16-byte shared loads feed 16 FMAs.  The eight warps'
// partial sums are added at the end in warp order: the sum over k has a fixed order.
// kVec: G % 4 == 0, so rows of M move as 16-byte pieces; otherwise as 4-byte words.
constexpr int kMixTG = 16, kMixTC = 32, kMixKC = 64, kMixStages = 3;
// A tile: g-major [16][64 + 4] for the mix (the pad puts the four rows a lane reads,
// g = q, q + 4, q + 8, q + 12, on different banks); k-major [64][16] for the transpose,
// as M[k][g] lies in memory.
template <bool kTrans>
__host__ __device__ constexpr int mix_a_words() { return kTrans ? kMixKC * kMixTG : kMixTG * (kMixKC + 4); }

__device__ __forceinline__ void cp_async16(float* dst, const float* src, bool valid) {
  const unsigned d = static_cast<unsigned>(__cvta_generic_to_shared(dst));
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(d), "l"(src), "r"(valid ? 16 : 0) : "memory");
}
__device__ __forceinline__ void cp_async4(float* dst, const float* src, bool valid) {
  const unsigned d = static_cast<unsigned>(__cvta_generic_to_shared(dst));
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(d), "l"(src), "r"(valid ? 4 : 0) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

template <bool kTrans, bool kVec>
__global__ void __launch_bounds__(256) k_mix_tiled(const float* __restrict__ M, const float* __restrict__ in,
                                                   float* __restrict__ out, int H, int G, int D) {
  constexpr int TG = kMixTG, TC = kMixTC, KC = kMixKC, S = kMixStages;
  constexpr int AW = mix_a_words<kTrans>(), BW = KC * TC, SW = AW + BW;
  __shared__ __align__(16) float sm[S * SW];
  const int64_t bh = blockIdx.y;
  const int h = (int)(bh % H);
  const int g0 = blockIdx.x * TG, c0 = blockIdx.z * TC;
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const float* Mh = M + (int64_t)h * G * G;
  const float* X = in + bh * (int64_t)G * D;
  const int nch = (G + KC - 1) / KC;

  // Stage chunk `ch` (k = ch * KC ...) into buffer `buf`; out-of-range words are zero-filled.
  auto issue = [&](int ch, int buf) {
    if (ch < nch) {
      const int k0 = ch * KC;
      float* sa = sm + buf * SW;
      float* sb = sa + AW;
      if (kVec) {
        if (kTrans) {  // A(g, k) = M[k][g]: row k, 4 consecutive g
          const int k = t >> 2, gg = (t & 3) * 4;
          const bool v = k0 + k < G && g0 + gg < G;
          cp_async16(sa + k * TG + gg, v ? Mh + (int64_t)(k0 + k) * G + g0 + gg : Mh, v);
        } else {  // A(g, k) = M[g][k]: row g, 4 consecutive k
          const int g = t >> 4, kk = (t & 15) * 4;
          const bool v = g0 + g < G && k0 + kk < G;
          cp_async16(sa + g * (KC + 4) + kk, v ? Mh + (int64_t)(g0 + g) * G + k0 + kk : Mh, v);
        }
      } else {
#pragma unroll
        for (int r = 0; r < 4; r++) {
          const int e = t + 256 * r;
          if (kTrans) {
            const int k = e / TG, gg = e % TG;
            const bool v = k0 + k < G && g0 + gg < G;
            cp_async4(sa + k * TG + gg, v ? Mh + (int64_t)(k0 + k) * G + g0 + gg : Mh, v);
          } else {
            const int g = e / KC, kk = e % KC;
            const bool v = g0 + g < G && k0 + kk < G;
            cp_async4(sa + g * (KC + 4) + kk, v ? Mh + (int64_t)(g0 + g) * G + k0 + kk : Mh, v);
          }
        }
      }
#pragma unroll
      for (int r = 0; r < 2; r++) {  // `in` rows k, 4 consecutive channels (D % 4 == 0)
        const int e = t + 256 * r, k = e >> 3, cc = (e & 7) * 4;
        const bool v = k0 + k < G && c0 + cc < D;
        cp_async16(sb + k * TC + cc, v ? X + (int64_t)(k0 + k) * D + c0 + cc : X, v);
      }
    }
    cp_async_commit();
  };

  // Lane (gq, cq): channels 4cq .. 4cq + 3; rows g = gq + 4i (mix) or 4gq + i (transpose).
  const int gq = lane >> 3, cq = lane & 7;
  float acc[4][4] = {};
#pragma unroll
  for (int st = 0; st < S - 1; st++) issue(st, st);
  for (int ch = 0; ch < nch; ch++) {
    cp_async_wait<S - 2>();
    __syncthreads();  // chunk ch is visible; every warp is done with chunk ch - 1's buffer
    issue(ch + S - 1, (ch + S - 1) % S);
    const float* sa = sm + (ch % S) * SW;
    const float* sb = sa + AW;
    if (kTrans) {
#pragma unroll
      for (int kk = 0; kk < 8; kk++) {
        const int k = warp * 8 + kk;
        const float4 a = *reinterpret_cast<const float4*>(sa + k * TG + 4 * gq);
        const float4 b = *reinterpret_cast<const float4*>(sb + k * TC + 4 * cq);
        const float av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
        for (int i = 0; i < 4; i++)
#pragma unroll
          for (int j = 0; j < 4; j++) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
      }
    } else {
#pragma unroll
      for (int half = 0; half < 2; half++) {
        const int kb = warp * 8 + half * 4;
        float av[4][4], bv[4][4];
#pragma unroll
        for (int i = 0; i < 4; i++) {
          const float4 a = *reinterpret_cast<const float4*>(sa + (gq + 4 * i) * (KC + 4) + kb);
          av[i][0] = a.x; av[i][1] = a.y; av[i][2] = a.z; av[i][3] = a.w;
        }
#pragma unroll
        for (int kk = 0; kk < 4; kk++) {
          const float4 b = *reinterpret_cast<const float4*>(sb + (kb + kk) * TC + 4 * cq);
          bv[kk][0] = b.x; bv[kk][1] = b.y; bv[kk][2] = b.z; bv[kk][3] = b.w;
        }
#pragma unroll
        for (int kk = 0; kk < 4; kk++)
#pragma unroll
          for (int i = 0; i < 4; i++)
#pragma unroll
            for (int j = 0; j < 4; j++) acc[i][j] = fmaf(av[i][kk], bv[kk][j], acc[i][j]);
      }
    }
  }
  cp_async_wait<0>();
  __syncthreads();  // the staging buffers become the eight warps' partial tiles
  float* red = sm;  // [8][TG][TC]
#pragma unroll
  for (int i = 0; i < 4; i++) {
    const int g = kTrans ? 4 * gq + i : gq + 4 * i;
    *reinterpret_cast<float4*>(red + (warp * TG + g) * TC + 4 * cq) = make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
  }
  __syncthreads();
#pragma unroll
  for (int r = 0; r < 2; r++) {
    const int o = t + 256 * r, g = o / TC, c = o % TC;
    float v = 0.f;
#pragma unroll
    for (int w = 0; w < 8; w++) v += red[(w * TG + g) * TC + c];
    if (g0 + g < G && c0 + c < D) out[(bh * G + g0 + g) * (int64_t)D + c0 + c] = v;
  }
}
static_assert(8 * kMixTG * kMixTC <= kMixStages * (kMixKC * kMixTC + kMixTG * (kMixKC + 4)),
              "the partial tiles fit in the staging buffers");

// Per-token channel map (the attention-free core): out[bh][g][c] = sum_k A(c, k)
// in[bh][g][k], with A = Wc[h] (forward) or Wc[h]^T (its token backward); one
// thread per output word, the sum over k in a fixed order.
template <bool kTrans>
__global__ void k_mix_channels(const float* __restrict__ Wc, const float* __restrict__ in, float* __restrict__ out,
                               int64_t BHG, int H, int G, int D) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= BHG * D) return;
  const int c = (int)(idx % D);
  const int64_t t = idx / D;  // token bh * G + g
  const int h = (int)((t / G) % H);
  const float* A = Wc + (int64_t)h * D * D;
  const float* z = in + t * D;
  float acc = 0.f;
  for (int k = 0; k < D; k++) acc = fmaf(kTrans ? A[(int64_t)k * D + c] : A[(int64_t)c * D + k], z[k], acc);
  out[idx] = acc;
}

// dWc[h][c][k] = sum over b and g of dzp[b,h,g,c] z[b,h,g,k] (fixed order: b, then g).
__global__ void k_mix_channels_dW(const float* __restrict__ z, const float* __restrict__ dzp, float* __restrict__ dWc,
                                  int64_t B, int H, int G, int D) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)H * D * D) return;
  const int k = (int)(idx % D), c = (int)((idx / D) % D), h = (int)(idx / ((int64_t)D * D));
  float acc = 0.f;
  for (int64_t b = 0; b < B; b++) {
    const int64_t base = (b * H + h) * (int64_t)G * D;
    for (int g = 0; g < G; g++) acc = fmaf(dzp[base + (int64_t)g * D + c], z[base + (int64_t)g * D + k], acc);
  }
  dWc[idx] = acc;
}

// dM[h][g][k] = sum_b sum_c dzp[b,h,g,c] z[b,h,k,c]: per head a G x G product with
// K = B*D, tiled 64 x 64 per block (16 x 16 threads, 4 x 4 outputs each), the two
// operand tiles staged in shared memory 16 channels at a time; the sum runs over
// b, then c, in a fixed order.
__global__ void __launch_bounds__(256) k_mix_bwd_dM(const float* __restrict__ z, const float* __restrict__ dzp,
                                                    float* __restrict__ dM, int64_t B, int H, int G, int D) {
  constexpr int T = 64, KC = 16;
  __shared__ float sa[KC][T + 1];
  __shared__ float sb[KC][T + 1];
  const int h = blockIdx.z;
  const int g0 = blockIdx.y * T, k0 = blockIdx.x * T;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};
  for (int64_t b = 0; b < B; b++) {
    const float* A = dzp + (b * H + h) * (int64_t)G * D;
    const float* Z = z + (b * H + h) * (int64_t)G * D;
    for (int c0 = 0; c0 < D; c0 += KC) {
      __syncthreads();
      for (int i = threadIdx.x; i < T * KC; i += 256) {
        const int r = i / KC, c = i % KC;
        sa[c][r] = (g0 + r < G && c0 + c < D) ? A[(int64_t)(g0 + r) * D + c0 + c] : 0.f;
        sb[c][r] = (k0 + r < G && c0 + c < D) ? Z[(int64_t)(k0 + r) * D + c0 + c] : 0.f;
      }
      __syncthreads();
#pragma unroll
      for (int c = 0; c < KC; c++) {
        float av[4], bv[4];
#pragma unroll
        for (int i = 0; i < 4; i++) {
          av[i] = sa[c][ty + 16 * i];
          bv[i] = sb[c][tx + 16 * i];
        }
#pragma unroll
        for (int i = 0; i < 4; i++)
#pragma unroll
          for (int j = 0; j < 4; j++) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
      }
    }
  }
#pragma unroll
  for (int i = 0; i < 4; i++) {
    const int g = g0 + ty + 16 * i;
    if (g >= G) continue;
#pragma unroll
    for (int j = 0; j < 4; j++) {
      const int k = k0 + tx + 16 * j;
      if (k < G) dM[((int64_t)h * G + g) * G + k] = acc[i][j];
    }
  }
}

// ---- deslice: point-owned ----------------------------------------------------------
template <int D, typename T>
__global__ void __launch_bounds__(kThreads) k_deslice(const T* __restrict__ x, const float* __restrict__ W,
                                                       const float* __restrict__ bias,
                                                       const float* __restrict__ tau,
                                                       const float* __restrict__ zp,
                                                       const float* __restrict__ lse, T* __restrict__ out,
                                                       int64_t N, int H, int G, uint32_t* status) {
  constexpr int GC = 32;
  __shared__ __align__(16) float sW[GC][D];
  __shared__ __align__(16) float sZ[GC][D];
  __shared__ float sB[GC];
  const int64_t bh = blockIdx.y;
  const int64_t b = bh / H;
  const int h = (int)(bh % H);
  if (!tau_ok(tau[h], status)) return;
  const float scale = kLog2e / tau[h];
  const int64_t n = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  const bool valid = n < N;
  float xr[D], acc[D];
#pragma unroll
  for (int k = 0; k < D; k++) { xr[k] = 0.f; acc[k] = 0.f; }
  float l2 = CUDART_INF_F;
  if (valid) {
    load_row<D>(x + row_index(b, n, h, N, H) * D, xr);
    l2 = lse[bh * N + n] * kLog2e;
  }
  const float* zb = zp + bh * G * D;
  for (int g0 = 0; g0 < G; g0 += GC) {
    __syncthreads();
    stage_w<D, GC>(sW, sB, W, bias, h, G, g0, scale);
    for (int i = threadIdx.x; i < GC * D; i += kThreads) {
      const int g = i / D, k = i % D;
      sZ[g][k] = (g0 + g < G) ? zb[(int64_t)(g0 + g) * D + k] : 0.f;
    }
    __syncthreads();
    const int gn = min(GC, G - g0);
    // Four slots at a time (independent logit chains); the output sums the slots in
    // order.  Slots past gn have zero z' rows and add exact zeros.
#pragma unroll 1
    for (int g = 0; g < gn; g += 4) {
      float a[4];
#pragma unroll
      for (int q = 0; q < 4; q++) a[q] = sB[g + q];
#pragma unroll
      for (int k = 0; k < D; k++)
#pragma unroll
        for (int q = 0; q < 4; q++) a[q] = fmaf(xr[k], sW[g + q][k], a[q]);
#pragma unroll
      for (int q = 0; q < 4; q++) {
        if (g + q >= gn) break;
        const float w = exp2f(a[q] - l2);
#pragma unroll
        for (int k = 0; k < D; k++) acc[k] = fmaf(w, sZ[g + q][k], acc[k]);
      }
    }
  }
  if (valid) store_row<D>(out + row_index(b, n, h, N, H) * D, acc);
}

// ---- backward, point-owned -------------------------------------------------------------
// Gradient w.r.t. the weights of point n at slot g:
//   MODE 0 (deslice): dw_g = dO . z'_g
//   MODE 1 (slice)  : dw_g = f . dU_g + dS_g      (dUS[bh][g] = (dU_g, dS_g))
// Sweep 1 forms delta = sum_g w_g dw_g (and, for the slice, dfx = sum_g w_g dU_g);
// sweep 2 forms dx = (1/tau) sum_g w_g (dw_g - delta) W[:,g].
template <int D, typename T, int MODE>
__global__ void __launch_bounds__(kThreads) k_bwd_point(
    const T* __restrict__ x, const T* __restrict__ v /* dout (MODE 0) or fx (MODE 1) */,
    const float* __restrict__ W, const float* __restrict__ bias, const float* __restrict__ tau,
    const float* __restrict__ tok /* z' (MODE 0) or (dU,dS) (MODE 1) */, const float* __restrict__ lse,
    T* __restrict__ dx, T* __restrict__ dfx, float* __restrict__ delta, float* __restrict__ dt_part,
    int accumulate, int64_t N, int H, int G, uint32_t* status) {
  constexpr int GC = 16;
  __shared__ float s_dt[kThreads];
  constexpr int TS = (MODE == 0) ? D : D + 1;  // token row stride in memory
  __shared__ __align__(16) float sW[GC][D];
  __shared__ __align__(16) float sT[GC][D];  // t_g (z' or dU)
  __shared__ float sS[GC];                    // MODE 1: dS_g
  __shared__ float sB[GC];
  const int64_t bh = blockIdx.y;
  const int64_t b = bh / H;
  const int h = (int)(bh % H);
  if (!tau_ok(tau[h], status)) return;
  const float scale = kLog2e / tau[h];
  const int64_t n = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  const bool valid = n < N;
  float xr[D], vr[D], acc[D];
#pragma unroll
  for (int k = 0; k < D; k++) { xr[k] = 0.f; vr[k] = 0.f; acc[k] = 0.f; }
  float l2 = CUDART_INF_F;
  const int64_t row = row_index(b, n, h, N, H);
  if (valid) {
    load_row<D>(x + row * D, xr);
    load_row<D>(v + row * D, vr);
    l2 = lse[bh * N + n] * kLog2e;
  }
  const float* tb = tok + bh * G * TS;
  float dl = 0.f;
  // The point's term of the temperature gradient, sum_g da_g (a_g - lse) in base-2
  // units: with the logits centred on lse (exact, since sum_g da_g = 0) the row
  // sum carries no large cancelling parts (App. G.2).
  float dtn = 0.f;
  for (int sweep = 0; sweep < 2; sweep++) {
    for (int g0 = 0; g0 < G; g0 += GC) {
      __syncthreads();
      stage_w<D, GC>(sW, sB, W, bias, h, G, g0, scale);
      for (int i = threadIdx.x; i < GC * TS; i += kThreads) {
        const int g = i / TS, k = i % TS;
        const float t = (g0 + g < G) ? tb[(int64_t)(g0 + g) * TS + k] : 0.f;
        if (k < D)
          sT[g][k] = t;
        else
          sS[g] = t;
      }
      __syncthreads();
      const int gn = min(GC, G - g0);
      // Four slots at a time: their logit and dw dot products are independent chains
      // (one 32-long chain per slot would leave the FMA pipe waiting on each result).
      // The per-slot updates below run in slot order, as one slot at a time would.
#pragma unroll 1
      for (int g = 0; g < gn; g += 4) {
        float a[4], dwq[4];
#pragma unroll
        for (int q = 0; q < 4; q++) {
          a[q] = sB[g + q];
          dwq[q] = (MODE == 0) ? 0.f : sS[g + q];
        }
#pragma unroll
        for (int k = 0; k < D; k++)
#pragma unroll
          for (int q = 0; q < 4; q++) {
            a[q] = fmaf(xr[k], sW[g + q][k], a[q]);
            dwq[q] = fmaf(vr[k], sT[g + q][k], dwq[q]);
          }
#pragma unroll
        for (int q = 0; q < 4; q++) {
          if (g + q >= gn) break;
          const float w = exp2f(a[q] - l2);
          const float dw = dwq[q];
          if (sweep == 0) {
            dl = fmaf(w, dw, dl);
            if (MODE == 1) {
#pragma unroll
              for (int k = 0; k < D; k++) acc[k] = fmaf(w, sT[g + q][k], acc[k]);
            }
          } else {
            const float da = w * (dw - dl);
#pragma unroll
            for (int k = 0; k < D; k++) acc[k] = fmaf(da, sW[g + q][k], acc[k]);
            if (valid) dtn = fmaf(da, a[q] - l2, dtn);
          }
        }
      }
    }
    if (sweep == 0) {
      if (MODE == 1 && valid) store_row<D>(dfx + row * D, acc);
#pragma unroll
      for (int k = 0; k < D; k++) acc[k] = 0.f;
    }
  }
  // Block sum of the temperature terms (fixed tree order) -> dt_part[bh][block].
  s_dt[threadIdx.x] = dtn;
  __syncthreads();
  for (int w = kThreads / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) s_dt[threadIdx.x] += s_dt[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) dt_part[bh * gridDim.x + blockIdx.x] = s_dt[0] * kLn2;
  if (!valid) return;
  delta[bh * N + n] = dl;
  // acc = sum_g da_g W[:,g] * log2e/tau ; dx = sum_g da_g W[:,g] / tau = acc * ln2.
#pragma unroll
  for (int k = 0; k < D; k++) acc[k] *= kLn2;
  if (accumulate) {
    float old[D];
    load_row<D>(dx + row * D, old);
#pragma unroll
    for (int k = 0; k < D; k++) acc[k] += old[k];
  }
  store_row<D>(dx + row * D, acc);
}

// ---- backward, slot-owned ---------------------------------------------------------------
// grid (ceil(G/128), B*H, P); thread = slot g.  For every point n of the split:
//   da = w (dw - delta_n);  dWa += da x_n;  dba += da;  dta += da * a_n
//   MODE 0 also accumulates dz'_g += w dO_n.
// part[p][bh][g][...] = (MODE 0: dz'(D)) , dWa(D), dba, dta   (un-scaled by 1/tau)
template <int D, typename T, int MODE>
__global__ void __launch_bounds__(kThreads) k_bwd_slot(
    const T* __restrict__ x, const T* __restrict__ v, const float* __restrict__ W,
    const float* __restrict__ bias, const float* __restrict__ tau, const float* __restrict__ tok,
    const float* __restrict__ lse, const float* __restrict__ delta, float* __restrict__ part, int64_t B,
    int64_t N, int H, int G, int64_t per_split, uint32_t* status) {
  constexpr int PT = 32;
  constexpr int TS = (MODE == 0) ? D : D + 1;
  constexpr int PS = (MODE == 0) ? 2 * D + 2 : D + 2;
  __shared__ __align__(16) float sx[PT][D];
  __shared__ __align__(16) float sv[PT][D];
  __shared__ float sl[PT];
  __shared__ float sd[PT];
  const int g = blockIdx.x * kThreads + threadIdx.x;
  const int64_t bh = blockIdx.y;
  const int64_t b = bh / H;
  const int h = (int)(bh % H);
  const int p = blockIdx.z;
  if (!tau_ok(tau[h], status)) return;
  const float scale = kLog2e / tau[h];
  float wc[D], tg[D], dzp[D], dWa[D];
  float bb = 0.f, dSg = 0.f, dba = 0.f;
#pragma unroll
  for (int k = 0; k < D; k++) {
    wc[k] = (g < G) ? W[((int64_t)h * D + k) * G + g] * scale : 0.f;
    tg[k] = (g < G) ? tok[(bh * G + g) * TS + k] : 0.f;
    dzp[k] = 0.f;
    dWa[k] = 0.f;
  }
  if (g < G) {
    bb = bias[(int64_t)h * G + g] * scale;
    if (MODE == 1) dSg = tok[(bh * G + g) * TS + D];
  }
  const int64_t n_begin = (int64_t)p * per_split;
  const int64_t n_end = min(N, n_begin + per_split);
  for (int64_t n0 = n_begin; n0 < n_end; n0 += PT) {
    __syncthreads();
    for (int i = threadIdx.x; i < PT * D; i += kThreads) {
      const int j = i / D, k = i % D;
      const int64_t n = n0 + j;
      float xv = 0.f, vv = 0.f;
      if (n < n_end) {
        const int64_t idx = row_index(b, n, h, N, H) * D + k;
        xv = to_f(x[idx]);
        vv = to_f(v[idx]);
      }
      sx[j][k] = xv;
      sv[j][k] = vv;
    }
    for (int i = threadIdx.x; i < PT; i += kThreads) {
      const int64_t n = n0 + i;
      const bool ok = n < n_end;
      sl[i] = ok ? lse[bh * N + n] * kLog2e : CUDART_INF_F;
      sd[i] = ok ? delta[bh * N + n] : 0.f;
    }
    __syncthreads();
    // Four points at a time: independent logit and dw chains; the updates below run
    // in point order, as one point at a time would.
#pragma unroll 1
    for (int j = 0; j < PT; j += 4) {
      float a[4], dwq[4];
#pragma unroll
      for (int q = 0; q < 4; q++) {
        a[q] = bb;
        dwq[q] = dSg;
      }
#pragma unroll
      for (int k = 0; k < D; k++)
#pragma unroll
        for (int q = 0; q < 4; q++) {
          a[q] = fmaf(sx[j + q][k], wc[k], a[q]);
          dwq[q] = fmaf(sv[j + q][k], tg[k], dwq[q]);
        }
#pragma unroll
      for (int q = 0; q < 4; q++) {
        const float w = exp2f(a[q] - sl[j + q]);
        const float da = w * (dwq[q] - sd[j + q]);
        if (MODE == 0) {
#pragma unroll
          for (int k = 0; k < D; k++) dzp[k] = fmaf(w, sv[j + q][k], dzp[k]);
        }
#pragma unroll
        for (int k = 0; k < D; k++) dWa[k] = fmaf(da, sx[j + q][k], dWa[k]);
        dba += da;
      }
    }
  }
  if (g < G) {
    float* o = part + (((int64_t)p * B * H + bh) * G + g) * PS;
    int off = 0;
    if (MODE == 0) {
#pragma unroll
      for (int k = 0; k < D; k++) o[k] = dzp[k];
      off = D;
    }
#pragma unroll
    for (int k = 0; k < D; k++) o[off + k] = dWa[k];
    o[off + D] = dba;
    o[off + D + 1] = 0.f;  // (the temperature gradient is formed per point, see k_bwd_point)
  }
}

// ---- the coupling's whole backward, fused -------------------------------------------------
// The deslice's and the slice's weight gradients share the weights, so their softmax
// backward adds up: da = w (dw - delta) with dw_g = dO . z'_g + fx . dU_g + dS_g and
// delta = sum_g w_g dw_g.  One point pass and one slot pass then serve both (the
// separate calls make two of each).
// Point pass: sweep 1 forms delta and dfx = sum_g w_g dU_g, sweep 2 dx = (1/tau) sum_g
// da_g W[:,g] (added to dx when accumulate) and the points' temperature terms.
template <int D, typename T>
__global__ void __launch_bounds__(kThreads) k_bwd_point_comb(
    const T* __restrict__ x, const T* __restrict__ dO, const T* __restrict__ fx, const float* __restrict__ W,
    const float* __restrict__ bias, const float* __restrict__ tau, const float* __restrict__ zp,
    const float* __restrict__ dUS, const float* __restrict__ lse, T* __restrict__ dx, T* __restrict__ dfx,
    float* __restrict__ delta, float* __restrict__ dt_part, int accumulate, int64_t N, int H, int G,
    uint32_t* status) {
  constexpr int GC = 16;
  __shared__ float s_dt[kThreads];
  __shared__ __align__(16) float sW[GC][D];
  __shared__ __align__(16) float sZ[GC][D];  // z'_g
  __shared__ __align__(16) float sU[GC][D];  // dU_g
  __shared__ float sS[GC];                    // dS_g
  __shared__ float sB[GC];
  const int64_t bh = blockIdx.y;
  const int64_t b = bh / H;
  const int h = (int)(bh % H);
  if (!tau_ok(tau[h], status)) return;
  const float scale = kLog2e / tau[h];
  const int64_t n = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  const bool valid = n < N;
  float xr[D], dr[D], fr[D], acc[D];
#pragma unroll
  for (int k = 0; k < D; k++) { xr[k] = 0.f; dr[k] = 0.f; fr[k] = 0.f; acc[k] = 0.f; }
  float l2 = CUDART_INF_F;
  const int64_t row = row_index(b, n, h, N, H);
  if (valid) {
    load_row<D>(x + row * D, xr);
    load_row<D>(dO + row * D, dr);
    load_row<D>(fx + row * D, fr);
    l2 = lse[bh * N + n] * kLog2e;
  }
  const float* zb = zp + bh * G * D;
  const float* ub = dUS + bh * G * (D + 1);
  auto stage = [&](int g0) {
    __syncthreads();
    stage_w<D, GC>(sW, sB, W, bias, h, G, g0, scale);
    for (int i = threadIdx.x; i < GC * D; i += kThreads) {
      const int g = i / D, k = i % D;
      sZ[g][k] = (g0 + g < G) ? zb[(int64_t)(g0 + g) * D + k] : 0.f;
    }
    for (int i = threadIdx.x; i < GC * (D + 1); i += kThreads) {
      const int g = i / (D + 1), k = i % (D + 1);
      const float t = (g0 + g < G) ? ub[(int64_t)(g0 + g) * (D + 1) + k] : 0.f;
      if (k < D)
        sU[g][k] = t;
      else
        sS[g] = t;
    }
    __syncthreads();
  };
  // Logits and dw of kQ slots at a time (independent chains; the point's x, dO, fx and
  // accumulator rows already hold 128 registers, so two rather than four).
  constexpr int kQ = 2;
  auto chains = [&](int g, float (&a)[kQ], float (&dwq)[kQ]) {
#pragma unroll
    for (int q = 0; q < kQ; q++) {
      a[q] = sB[g + q];
      dwq[q] = sS[g + q];
    }
#pragma unroll
    for (int k = 0; k < D; k++)
#pragma unroll
      for (int q = 0; q < kQ; q++) {
        a[q] = fmaf(xr[k], sW[g + q][k], a[q]);
        dwq[q] = fmaf(dr[k], sZ[g + q][k], dwq[q]);
        dwq[q] = fmaf(fr[k], sU[g + q][k], dwq[q]);
      }
  };
  // Sweep 1: delta and dfx (updates in slot order).
  float dl = 0.f;
  for (int g0 = 0; g0 < G; g0 += GC) {
    stage(g0);
    const int gn = min(GC, G - g0);
#pragma unroll 1
    for (int g = 0; g < gn; g += kQ) {
      float a[kQ], dwq[kQ];
      chains(g, a, dwq);
#pragma unroll
      for (int q = 0; q < kQ; q++) {
        if (g + q < gn) {
          const float w = exp2f(a[q] - l2);
          dl = fmaf(w, dwq[q], dl);
#pragma unroll
          for (int k = 0; k < D; k++) acc[k] = fmaf(w, sU[g + q][k], acc[k]);
        }
      }
    }
  }
  if (valid) store_row<D>(dfx + row * D, acc);
#pragma unroll
  for (int k = 0; k < D; k++) acc[k] = 0.f;
  // Sweep 2: dx and the temperature terms.
  float dtn = 0.f;
  for (int g0 = 0; g0 < G; g0 += GC) {
    stage(g0);
    const int gn = min(GC, G - g0);
#pragma unroll 1
    for (int g = 0; g < gn; g += kQ) {
      float a[kQ], dwq[kQ];
      chains(g, a, dwq);
#pragma unroll
      for (int q = 0; q < kQ; q++) {
        if (g + q < gn) {
          const float da = exp2f(a[q] - l2) * (dwq[q] - dl);
#pragma unroll
          for (int k = 0; k < D; k++) acc[k] = fmaf(da, sW[g + q][k], acc[k]);
          if (valid) dtn = fmaf(da, a[q] - l2, dtn);
        }
      }
    }
  }
  // Block sum of the temperature terms (fixed tree order) -> dt_part[bh][block].
  s_dt[threadIdx.x] = dtn;
  __syncthreads();
  for (int w = kThreads / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) s_dt[threadIdx.x] += s_dt[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) dt_part[bh * gridDim.x + blockIdx.x] = s_dt[0] * kLn2;
  if (!valid) return;
  delta[bh * N + n] = dl;
#pragma unroll
  for (int k = 0; k < D; k++) acc[k] *= kLn2;
  if (accumulate) {
    float old[D];
    load_row<D>(dx + row * D, old);
#pragma unroll
    for (int k = 0; k < D; k++) acc[k] += old[k];
  }
  store_row<D>(dx + row * D, acc);
}

// Slot pass of the fused backward: thread = slot g; for every point n of the split,
// da = w (dw - delta_n) with dw as above; dWa += da x_n; dba += da.
// part[p][bh][g] = (dWa (D), dba, 0), un-scaled by 1/tau.
template <int D, typename T>
__global__ void __launch_bounds__(kThreads) k_bwd_slot_comb(
    const T* __restrict__ x, const T* __restrict__ dO, const T* __restrict__ fx, const float* __restrict__ W,
    const float* __restrict__ bias, const float* __restrict__ tau, const float* __restrict__ zp,
    const float* __restrict__ dUS, const float* __restrict__ lse, const float* __restrict__ delta,
    float* __restrict__ part, int64_t B, int64_t N, int H, int G, int64_t per_split, uint32_t* status) {
  constexpr int PT = 32;
  constexpr int PS = D + 2;
  __shared__ __align__(16) float sx[PT][D];
  __shared__ __align__(16) float sd[PT][D];  // dO
  __shared__ __align__(16) float sf[PT][D];  // fx
  __shared__ float sl[PT];
  __shared__ float sdl[PT];
  const int g = blockIdx.x * kThreads + threadIdx.x;
  const int64_t bh = blockIdx.y;
  const int64_t b = bh / H;
  const int h = (int)(bh % H);
  const int p = blockIdx.z;
  if (!tau_ok(tau[h], status)) return;
  const float scale = kLog2e / tau[h];
  float wc[D], zg[D], ug[D], dWa[D];
  float bb = 0.f, dSg = 0.f, dba = 0.f;
#pragma unroll
  for (int k = 0; k < D; k++) {
    wc[k] = (g < G) ? W[((int64_t)h * D + k) * G + g] * scale : 0.f;
    zg[k] = (g < G) ? zp[(bh * G + g) * D + k] : 0.f;
    ug[k] = (g < G) ? dUS[(bh * G + g) * (D + 1) + k] : 0.f;
    dWa[k] = 0.f;
  }
  if (g < G) {
    bb = bias[(int64_t)h * G + g] * scale;
    dSg = dUS[(bh * G + g) * (D + 1) + D];
  }
  const int64_t n_begin = (int64_t)p * per_split;
  const int64_t n_end = min(N, n_begin + per_split);
  for (int64_t n0 = n_begin; n0 < n_end; n0 += PT) {
    __syncthreads();
    for (int i = threadIdx.x; i < PT * D; i += kThreads) {
      const int j = i / D, k = i % D;
      const int64_t n = n0 + j;
      float xv = 0.f, dv = 0.f, fv = 0.f;
      if (n < n_end) {
        const int64_t idx = row_index(b, n, h, N, H) * D + k;
        xv = to_f(x[idx]);
        dv = to_f(dO[idx]);
        fv = to_f(fx[idx]);
      }
      sx[j][k] = xv;
      sd[j][k] = dv;
      sf[j][k] = fv;
    }
    for (int i = threadIdx.x; i < PT; i += kThreads) {
      const int64_t n = n0 + i;
      const bool ok = n < n_end;
      sl[i] = ok ? lse[bh * N + n] * kLog2e : CUDART_INF_F;
      sdl[i] = ok ? delta[bh * N + n] : 0.f;
    }
    __syncthreads();
    // Four points at a time (independent chains), updates in point order.
#pragma unroll 1
    for (int j = 0; j < PT; j += 4) {
      float a[4], dwq[4];
#pragma unroll
      for (int q = 0; q < 4; q++) {
        a[q] = bb;
        dwq[q] = dSg;
      }
#pragma unroll
      for (int k = 0; k < D; k++)
#pragma unroll
        for (int q = 0; q < 4; q++) {
          a[q] = fmaf(sx[j + q][k], wc[k], a[q]);
          dwq[q] = fmaf(sd[j + q][k], zg[k], dwq[q]);
          dwq[q] = fmaf(sf[j + q][k], ug[k], dwq[q]);
        }
#pragma unroll
      for (int q = 0; q < 4; q++) {
        const float w = exp2f(a[q] - sl[j + q]);
        const float da = w * (dwq[q] - sdl[j + q]);
#pragma unroll
        for (int k = 0; k < D; k++) dWa[k] = fmaf(da, sx[j + q][k], dWa[k]);
        dba += da;
      }
    }
  }
  if (g < G) {
    float* o = part + (((int64_t)p * B * H + bh) * G + g) * PS;
#pragma unroll
    for (int k = 0; k < D; k++) o[k] = dWa[k];
    o[D] = dba;
    o[D + 1] = 0.f;  // (the temperature gradient is formed per point, in the point pass)
  }
}

// Token-gradient prep for the slice backward: dUS[bh][g] = (dz_g/(S_g+eps), -(dz_g.z_g)/(S_g+eps)).
__global__ void k_slice_bwd_prep(const float* __restrict__ z, const float* __restrict__ wsum,
                                 const float* __restrict__ dz, float* __restrict__ dUS, int64_t BHG, int D,
                                 float eps) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= BHG) return;
  const float den = wsum[i] + eps;
  float s = 0.f;
  for (int c = 0; c < D; c++) {
    const float g = dz[i * D + c];
    dUS[i * (D + 1) + c] = g / den;
    s = fmaf(g, z[i * D + c], s);
  }
  dUS[i * (D + 1) + D] = -s / den;
}

// Fixed-order reduction of slot-owned backward partials over (b, p), one thread
// per output word (consecutive threads read consecutive words of a partial row):
//   k_reduce_bwd_params: dW[h][k][g], db[h][g] (written, or added), sums over b then p;
//   k_reduce_bwd_tokens: d_tokens_mixed[b][h][g][c], sums over p.
// The temperature gradient is reduced separately, from its own partials.
__global__ void k_reduce_bwd_params(const float* __restrict__ part, int P, int64_t B, int H, int G, int Gs, int D,
                                    int PS, int off, const float* __restrict__ tau, float* __restrict__ dW,
                                    float* __restrict__ db, int accumulate) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)H * G * (D + 1)) return;
  const int k = (int)(idx % (D + 1));
  const int64_t hg = idx / (D + 1);
  const int h = (int)(hg / G), g = (int)(hg % G);
  const int64_t BH = B * H;
  float s = 0.f;
  for (int64_t b = 0; b < B; b++)
    for (int p = 0; p < P; p++) s += part[(((int64_t)p * BH + b * H + h) * Gs + g) * PS + off + k];
  s *= 1.f / tau[h];
  if (k < D) {
    const int64_t o = ((int64_t)h * D + k) * G + g;
    dW[o] = (accumulate ? dW[o] : 0.f) + s;
  } else {
    db[hg] = (accumulate ? db[hg] : 0.f) + s;
  }
}
__global__ void k_reduce_bwd_tokens(const float* __restrict__ part, int P, int64_t BH, int G, int Gs, int D, int PS,
                                    float* __restrict__ dzp) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= BH * G * D) return;
  const int c = (int)(idx % D);
  const int64_t i = idx / D;                  // output row bh * G + g
  const int64_t row = (i / G) * Gs + i % G;  // its partial row
  float s = 0.f;
  for (int p = 0; p < P; p++) s += part[((int64_t)p * BH * Gs + row) * PS + c];
  dzp[idx] = s;
}

// dtau[h] (+)= -(1/tau_h) * sum over batches and point blocks of the block sums of
// sum_g da (a - lse) (fixed order: strided per thread, then a tree).
__global__ void k_reduce_dtau(const float* __restrict__ dt_part, int64_t B, int H, int64_t nblk,
                              const float* __restrict__ tau, float* __restrict__ dtau, int accumulate) {
  __shared__ float s[256];
  const int h = blockIdx.x;
  float v = 0.f;
  for (int64_t b = 0; b < B; b++)
    for (int64_t i = threadIdx.x; i < nblk; i += 256) v += dt_part[(b * H + h) * nblk + i];
  s[threadIdx.x] = v;
  __syncthreads();
  for (int w = 128; w > 0; w >>= 1) {
    if (threadIdx.x < w) s[threadIdx.x] += s[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) dtau[h] = (accumulate ? dtau[h] : 0.f) - s[0] / tau[h];
}

inline dim3 point_grid(const Shape& s) {
  return dim3((unsigned)((s.N + kThreads - 1) / kThreads), (unsigned)s.BH());
}
inline dim3 slot_grid(const Shape& s, int P) {
  return dim3((unsigned)((s.G + kThreads - 1) / kThreads), (unsigned)s.BH(), (unsigned)P);
}
inline int64_t per_split(const Shape& s, int P) { return (s.N + P - 1) / P; }

template <int D, typename T>
cudaError_t launch_stats(const Shape& s, const void* x, const float* W, const float* bias, const float* tau,
                         float* lse, uint32_t* status, cudaStream_t st) {
  k_stats<D, T><<<point_grid(s), kThreads, 0, st>>>((const T*)x, W, bias, tau, lse, s.N, s.H, s.G, status);
  return cudaGetLastError();
}

template <int D, typename T>
cudaError_t launch_slice_partials(const Shape& s, int P, const void* x, const void* f, const float* W,
                                  const float* bias, const float* tau, const float* lse, float* part,
                                  uint32_t* status, cudaStream_t st) {
  k_slice_partial<D, T><<<slot_grid(s, P), kThreads, 0, st>>>((const T*)x, (const T*)f, W, bias, tau, lse,
                                                               part, s.B, s.N, s.H, s.G, per_split(s, P),
                                                               status);
  return cudaGetLastError();
}

template <int D, typename T>
cudaError_t launch_deslice(const Shape& s, const void* x, const float* W, const float* bias, const float* tau,
                           const float* zp, const float* lse, void* out, uint32_t* status, cudaStream_t st) {
  k_deslice<D, T><<<point_grid(s), kThreads, 0, st>>>((const T*)x, W, bias, tau, zp, lse, (T*)out, s.N, s.H,
                                                       s.G, status);
  return cudaGetLastError();
}

template <int D, typename T, int MODE>
cudaError_t launch_bwd(const Shape& s, int P, const void* x, const void* v, const float* W, const float* bias,
                       const float* tau, const float* tok, const float* lse, void* dx, void* dfx, float* delta,
                       float* dt_part, float* part, int accumulate, uint32_t* status, cudaStream_t st) {
  k_bwd_point<D, T, MODE><<<point_grid(s), kThreads, 0, st>>>((const T*)x, (const T*)v, W, bias, tau, tok, lse,
                                                               (T*)dx, (T*)dfx, delta, dt_part, accumulate, s.N,
                                                               s.H, s.G, status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_bwd_slot<D, T, MODE><<<slot_grid(s, P), kThreads, 0, st>>>((const T*)x, (const T*)v, W, bias, tau, tok,
                                                                lse, delta, part, s.B, s.N, s.H, s.G,
                                                                per_split(s, P), status);
  return cudaGetLastError();
}

template <int D, typename T>
cudaError_t launch_bwd_comb(const Shape& s, int P, const void* x, const void* dO, const void* fx, const float* W,
                            const float* bias, const float* tau, const float* zp, const float* dUS,
                            const float* lse, void* dx, void* dfx, float* delta, float* dt_part, float* part,
                            int accumulate, uint32_t* status, cudaStream_t st) {
  k_bwd_point_comb<D, T><<<point_grid(s), kThreads, 0, st>>>((const T*)x, (const T*)dO, (const T*)fx, W, bias, tau,
                                                              zp, dUS, lse, (T*)dx, (T*)dfx, delta, dt_part,
                                                              accumulate, s.N, s.H, s.G, status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_bwd_slot_comb<D, T><<<slot_grid(s, P), kThreads, 0, st>>>((const T*)x, (const T*)dO, (const T*)fx, W, bias, tau,
                                                               zp, dUS, lse, delta, part, s.B, s.N, s.H, s.G,
                                                               per_split(s, P), status);
  return cudaGetLastError();
}

// Dispatch over (d, dtype).// Dispatch over (d, dtype).
#define FS_DISPATCH(s, FN, ...)                                                        \
  do {                                                                                 \
    const bool bf = (s).dtype == FS_BF16;                                              \
    switch ((s).d) {                                                                   \
      case 16: return bf ? FN<16, __nv_bfloat16>(__VA_ARGS__) : FN<16, float>(__VA_ARGS__); \
      case 32: return bf ? FN<32, __nv_bfloat16>(__VA_ARGS__) : FN<32, float>(__VA_ARGS__); \
      case 64: return bf ? FN<64, __nv_bfloat16>(__VA_ARGS__) : FN<64, float>(__VA_ARGS__); \
      default: return cudaErrorInvalidValue;                                           \
    }                                                                                  \
  } while (0)

template <int D, typename T>
cudaError_t launch_bwd_deslice(const Shape& s, int P, const void* x, const void* v, const float* W,
                               const float* bias, const float* tau, const float* tok, const float* lse,
                               void* dx, float* delta, float* dt_part, float* part, int accumulate,
                               uint32_t* status, cudaStream_t st) {
  return launch_bwd<D, T, 0>(s, P, x, v, W, bias, tau, tok, lse, dx, nullptr, delta, dt_part, part, accumulate,
                             status, st);
}
template <int D, typename T>
cudaError_t launch_bwd_slice(const Shape& s, int P, const void* x, const void* v, const float* W,
                             const float* bias, const float* tau, const float* tok, const float* lse, void* dx,
                             void* dfx, float* delta, float* dt_part, float* part, int accumulate,
                             uint32_t* status, cudaStream_t st) {
  return launch_bwd<D, T, 1>(s, P, x, v, W, bias, tau, tok, lse, dx, dfx, delta, dt_part, part, accumulate,
                             status, st);
}

}  // namespace

cudaError_t simt_reduce_bwd(const Shape& s, int P, const float* part, int Gs, int PS, int has_dzp, const float* tau,
                            float* dzp, float* dW, float* db, float* dtau, const float* dt_part, int64_t nblk,
                            int accumulate, cudaStream_t st) {
  const int64_t nw = (int64_t)s.H * s.G * (s.d + 1);
  k_reduce_bwd_params<<<(unsigned)((nw + 255) / 256), 256, 0, st>>>(part, P, s.B, s.H, s.G, Gs, s.d, PS,
                                                                     has_dzp ? s.d : 0, tau, dW, db, accumulate);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (has_dzp) {
    const int64_t BHG = s.BH() * s.G;
    k_reduce_bwd_tokens<<<(unsigned)((BHG * s.d + 255) / 256), 256, 0, st>>>(part, P, s.BH(), s.G, Gs, s.d, PS,
                                                                              dzp);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  k_reduce_dtau<<<s.H, 256, 0, st>>>(dt_part, s.B, s.H, nblk, tau, dtau, accumulate);
  return cudaGetLastError();
}

cudaError_t simt_reduce_dzp(const Shape& s, int P, const float* part, int Gs, int PS, float* dzp, cudaStream_t st) {
  const int64_t BHG = s.BH() * s.G;
  k_reduce_bwd_tokens<<<(unsigned)((BHG * s.d + 255) / 256), 256, 0, st>>>(part, P, s.BH(), s.G, Gs, s.d, PS, dzp);
  return cudaGetLastError();
}

cudaError_t simt_slice_bwd_prep(const Shape& s, const float* z, const float* wsum, const float* dz, float* dUS,
                                cudaStream_t st) {
  const int64_t BHG = s.BH() * s.G;
  k_slice_bwd_prep<<<(unsigned)((BHG + 255) / 256), 256, 0, st>>>(z, wsum, dz, dUS, BHG, s.d, s.eps);
  return cudaGetLastError();
}

int64_t simt_point_blocks(const Shape& s) { return (s.N + kThreads - 1) / kThreads; }

cudaError_t simt_stats(const Shape& s, const void* x, const float* W, const float* bias, const float* tau,
                       float* lse, uint32_t* status, cudaStream_t st) {
  FS_DISPATCH(s, launch_stats, s, x, W, bias, tau, lse, status, st);
}

cudaError_t simt_slice_partials(const Shape& s, int P, const void* x, const void* f, const float* W,
                                const float* bias, const float* tau, const float* lse, float* part,
                                uint32_t* status, cudaStream_t st) {
  FS_DISPATCH(s, launch_slice_partials, s, P, x, f, W, bias, tau, lse, part, status, st);
}

cudaError_t simt_reduce_tokens(const Shape& s, int P, const float* part, int Gs, float* tokens, float* wsum,
                               int finalize, cudaStream_t st) {
  const int64_t n = s.BH() * s.G * 32;  // a warp per output row
  k_reduce_tokens<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(part, P, s.BH(), s.G, Gs, s.d, tokens, wsum, finalize,
                                                               s.eps);
  return cudaGetLastError();
}

cudaError_t simt_finalize(const Shape& s, float* tokens, const float* wsum, cudaStream_t st) {
  const int64_t BHG = s.BH() * s.G;
  k_finalize<<<(unsigned)((BHG * s.d + 255) / 256), 256, 0, st>>>(tokens, wsum, BHG, s.d, s.eps);
  return cudaGetLastError();
}

cudaError_t simt_mix(const Shape& s, const float* M, const float* z, float* zp, cudaStream_t st) {
  const dim3 grid((unsigned)((s.G + kMixTG - 1) / kMixTG), (unsigned)s.BH(), (unsigned)((s.d + kMixTC - 1) / kMixTC));
  if (s.G % 4 == 0)
    k_mix_tiled<false, true><<<grid, 256, 0, st>>>(M, z, zp, s.H, s.G, s.d);
  else
    k_mix_tiled<false, false><<<grid, 256, 0, st>>>(M, z, zp, s.H, s.G, s.d);
  return cudaGetLastError();
}

cudaError_t simt_mix_bwd(const Shape& s, const float* M, const float* z, const float* dzp, float* dz, float* dM,
                         cudaStream_t st) {
  const dim3 grid((unsigned)((s.G + kMixTG - 1) / kMixTG), (unsigned)s.BH(), (unsigned)((s.d + kMixTC - 1) / kMixTC));
  if (s.G % 4 == 0)
    k_mix_tiled<true, true><<<grid, 256, 0, st>>>(M, dzp, dz, s.H, s.G, s.d);
  else
    k_mix_tiled<true, false><<<grid, 256, 0, st>>>(M, dzp, dz, s.H, s.G, s.d);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const dim3 tiles((unsigned)((s.G + 63) / 64), (unsigned)((s.G + 63) / 64), (unsigned)s.H);
  k_mix_bwd_dM<<<tiles, 256, 0, st>>>(z, dzp, dM, s.B, s.H, s.G, s.d);
  return cudaGetLastError();
}

cudaError_t simt_mix_channels(const Shape& s, const float* Wc, const float* z, float* zp, cudaStream_t st) {
  const int64_t BHG = s.BH() * s.G;
  k_mix_channels<false><<<(unsigned)((BHG * s.d + 255) / 256), 256, 0, st>>>(Wc, z, zp, BHG, s.H, s.G, s.d);
  return cudaGetLastError();
}

cudaError_t simt_mix_channels_bwd(const Shape& s, const float* Wc, const float* z, const float* dzp, float* dz,
                                  float* dWc, cudaStream_t st) {
  const int64_t BHG = s.BH() * s.G;
  k_mix_channels<true><<<(unsigned)((BHG * s.d + 255) / 256), 256, 0, st>>>(Wc, dzp, dz, BHG, s.H, s.G, s.d);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int64_t n = (int64_t)s.H * s.d * s.d;
  k_mix_channels_dW<<<(unsigned)((n + 127) / 128), 128, 0, st>>>(z, dzp, dWc, s.B, s.H, s.G, s.d);
  return cudaGetLastError();
}

cudaError_t simt_deslice(const Shape& s, const void* x, const float* W, const float* bias, const float* tau,
                         const float* zp, const float* lse, void* out, uint32_t* status, cudaStream_t st) {
  FS_DISPATCH(s, launch_deslice, s, x, W, bias, tau, zp, lse, out, status, st);
}

cudaError_t simt_deslice_bwd(const Shape& s, int P, const void* x, const float* W, const float* bias,
                             const float* tau, const float* zp, const float* lse, const void* dout, float* dzp,
                             void* dx, float* dW, float* db, float* dtau, int accumulate, float* delta,
                             float* part, float* dt_part, uint32_t* status, cudaStream_t st) {
  cudaError_t e = [&]() -> cudaError_t {
    FS_DISPATCH(s, launch_bwd_deslice, s, P, x, dout, W, bias, tau, zp, lse, dx, delta, dt_part, part,
                accumulate, status, st);
  }();
  if (e != cudaSuccess) return e;
  return simt_reduce_bwd(s, P, part, s.G, 2 * s.d + 2, 1, tau, dzp, dW, db, dtau, dt_part, simt_point_blocks(s),
                         accumulate, st);
}

cudaError_t simt_slice_bwd(const Shape& s, int P, const void* x, const void* f, const float* W,
                           const float* bias, const float* tau, const float* z, const float* wsum,
                           const float* lse, const float* dz, void* dx, void* dfx, float* dW, float* db,
                           float* dtau, int accumulate, float* delta, float* dUS, float* part, float* dt_part,
                           uint32_t* status, cudaStream_t st) {
  cudaError_t e = simt_slice_bwd_prep(s, z, wsum, dz, dUS, st);
  if (e != cudaSuccess) return e;
  e = [&]() -> cudaError_t {
    FS_DISPATCH(s, launch_bwd_slice, s, P, x, f, W, bias, tau, dUS, lse, dx, dfx, delta, dt_part, part,
                accumulate, status, st);
  }();
  if (e != cudaSuccess) return e;
  return simt_reduce_bwd(s, P, part, s.G, s.d + 2, 0, tau, nullptr, dW, db, dtau, dt_part, simt_point_blocks(s),
                         accumulate, st);
}

// The coupling's whole backward on the SIMT kernels: d z' as the forward slice's
// unnormalised numerators with dO for fx, the mix backward, the slice's dU, dS, then
// one point pass and one slot pass for da_D + da_S (k_bwd_point_comb, k_bwd_slot_comb)
// and the parameter reductions.  `part` holds the larger of the two partial sets;
// the d z' reduction's weight sums go to dUS, which the prologue then overwrites.
cudaError_t simt_coupling_bwd(const Shape& s, int P, const void* x, const void* fx, const void* dout,
                              const float* W, const float* bias, const float* tau, const float* M, const float* z,
                              const float* wsum, const float* zp, const float* lse, float* dzp, float* dz,
                              float* dM, void* dx, void* dfx, float* dW, float* db, float* dtau, int accumulate,
                              float* delta, float* dUS, float* part, float* dt_part, uint32_t* status,
                              cudaStream_t st) {
  cudaError_t e = simt_slice_partials(s, P, x, dout, W, bias, tau, lse, part, status, st);
  if (e != cudaSuccess) return e;
  if ((e = simt_reduce_tokens(s, P, part, s.G, dzp, dUS, 0, st)) != cudaSuccess) return e;
  if ((e = simt_mix_bwd(s, M, z, dzp, dz, dM, st)) != cudaSuccess) return e;
  if ((e = simt_slice_bwd_prep(s, z, wsum, dz, dUS, st)) != cudaSuccess) return e;
  e = [&]() -> cudaError_t {
    FS_DISPATCH(s, launch_bwd_comb, s, P, x, dout, fx, W, bias, tau, zp, dUS, lse, dx, dfx, delta, dt_part, part,
                accumulate, status, st);
  }();
  if (e != cudaSuccess) return e;
  return simt_reduce_bwd(s, P, part, s.G, s.d + 2, 0, tau, nullptr, dW, db, dtau, dt_part, simt_point_blocks(s),
                         accumulate, st);
}
// Kernels it launches (the statistics, when needed, are counted by the caller).
int simt_coupling_bwd_launch_count() { return 2 /*partials, reduce*/ + 2 /*mix backward*/ + 1 /*prologue*/ +
                                              2 /*point, slot*/ + 2 /*reductions*/; }

}  // namespace fs
