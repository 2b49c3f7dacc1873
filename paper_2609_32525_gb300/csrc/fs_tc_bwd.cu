// Tensor-core backward (tcgen05 / TMEM / TMA) for bf16 inputs on sm_103a.
//
// The gradients of the slice and of the deslice (Sec. 3.3) share one form.  With
// w_ng = softmax_g(a_ng), a per-point vector v_n and per-slot t_g, c_g:
//   dw_ng = v_n . t_g + c_g,   delta_n = sum_g w_ng dw_ng,   da_ng = w_ng (dw_ng - delta_n)
//   deslice: v = dO, t = z', c = 0;   slice: v = fx, t = dU = dz/(S+eps), c = dS = -dz.z/(S+eps)
// and then
//   dx_n = (1/tau) sum_g da_ng W[:,g],   dW[:,g] = (1/tau) sum_n da_ng x_n,
//   dbias_g = (1/tau) sum_n da_ng,       dtau = -(1/tau) sum_n sum_g da_ng (a_ng - lse_n),
//   deslice also d z'_g = sum_n w_ng dO_n;  slice also dfx_n = sum_g w_ng dU_g.
// Three passes, w recomputed in each and never written to memory:
//   rows  (point-owned; the deslice kernel in a backward mode): delta_n (and dfx_n);
//   slot  (slot-owned, split over points): dW, dbias, dtau (and d z') partials;
//   point (point-owned): dx.
// dw - delta is one more MMA chain of the logits' shape: the slot side carries
// [t_g | c_g halves, 1, 1, 1] (the T image, laid out as the W image) and the point
// side [v_n | 1, 1, -delta_n in three bf16 parts] (delta's point-extra rows).
#include "fs_tc_common.cuh"

namespace fs {
namespace {

using namespace tc;

constexpr int kBStages = 6;                            // slot pass pipeline depth (point tiles)
constexpr int kDxStages = 3;                           // point pass pipeline depth
constexpr uint32_t kBStage = 2 * kXBytes + 2 * kPxBytes;  // x | v | lse rows | delta rows (TMA halves)
constexpr uint32_t kPxZero = 2 * kPxBytes;             // one zero block for the k = 8..15 halves
constexpr uint32_t kWBlockB = kGC * kWRow;             // one 128-slot block of a W or T image

// ---- prep kernels ------------------------------------------------------------------------------

// T image of (b,h), in the W image's layout (kWRow bytes per slot): t_g rounded to
// bf16, the extra rows [c_hi, c_lo, 1, 1, 1, 0...] (k = 2..4 meet -delta's three
// parts), the residual t_g - bf16(t_g).
// t: [BH][G][tstride] fp32, c_g = t[..][32] when has_c.  Also writes c_g to c_out
// [BH][Gp].  Padding slots [G, Gp) get t = 0 and c = 0 (their weights are 0).
__global__ void k_prep_t(const float* __restrict__ t, int tstride, int has_c, uint8_t* __restrict__ img,
                         float* __restrict__ c_out, int64_t BH, int G, int Gp) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= BH * Gp) return;
  const int64_t bh = i / Gp;
  const int g = (int)(i % Gp);
  const bool real = g < G;
  const float* src = t + (bh * G + (real ? g : 0)) * tstride;
  uint8_t* base = img + (size_t)bh * Gp * kWRow;
  __nv_bfloat16* hp = reinterpret_cast<__nv_bfloat16*>(base);
  __nv_bfloat16* lp = reinterpret_cast<__nv_bfloat16*>(base + (size_t)Gp * 96);
  for (int k = 0; k < kD; k++) {
    const float v = real ? src[k] : 0.f;
    const __nv_bfloat16 hi = __float2bfloat16_rn(v);
    hp[off_sw64(g, k) / 2] = hi;
    lp[off_sw64(g, k) / 2] = __float2bfloat16_rn(v - __bfloat162float(hi));
  }
  const float c = (has_c && real) ? src[kD] : 0.f;
  if (c_out) c_out[i] = c;
  const __nv_bfloat16 chi = __float2bfloat16_rn(c);
  const __nv_bfloat16 clo = __float2bfloat16_rn(c - __bfloat162float(chi));
  __nv_bfloat16* ep = reinterpret_cast<__nv_bfloat16*>(base + (size_t)Gp * 64);
  for (int k = 0; k < 16; k++)
    ep[off_sw32(g, k) / 2] = k == 0 ? chi : (k == 1 ? clo : __float2bfloat16_rn((k >= 2 && k <= 4) ? 1.f : 0.f));
}

// W'^T image of head h in the Z layout (channel rows, slots along K), W' =
// W log2(e)/tau: the bf16 half, then the residual half (Gp*128 bytes per head;
// padding slots zero).  It is the B operand of dx += da W'^T.
__global__ void k_prep_wt(const float* __restrict__ W, const float* __restrict__ tau, uint8_t* __restrict__ img,
                          int H, int G, int Gp, uint32_t* status) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (int64_t)H * kD * Gp) return;
  const int g = (int)(i % Gp);
  const int c = (int)((i / Gp) % kD);
  const int h = (int)(i / ((int64_t)kD * Gp));
  const float tv = tau[h];
  if (!(tv > 0.f && tv < INFINITY)) {
    atomicCAS(status, 0u, (uint32_t)FS_ERR_BAD_TAU);
    return;
  }
  const float v = g < G ? W[((int64_t)h * kD + c) * G + g] * (kLog2e / tv) : 0.f;
  __nv_bfloat16* hp = reinterpret_cast<__nv_bfloat16*>(img + (size_t)h * Gp * 128);
  __nv_bfloat16* lp = reinterpret_cast<__nv_bfloat16*>(img + (size_t)h * Gp * 128 + (size_t)Gp * 64);
  const __nv_bfloat16 hi = __float2bfloat16_rn(v);
  hp[off_z(c, g) / 2] = hi;
  lp[off_z(c, g) / 2] = __float2bfloat16_rn(v - __bfloat162float(hi));
}

// delta's point-extra rows [1, 1, -delta in three bf16 parts, 0, 0, 0] into dpx [BH, Np, 8];
// delta_n = delta[bh][n] (+ delta2[bh][n] when given, + wds[0][bh][n] + wds[1][bh][n]
// when wds is given).
__global__ void k_prep_dpx(const float* __restrict__ delta, const float* __restrict__ delta2,
                           const float* __restrict__ wds, uint4* __restrict__ dpx, int64_t BH, int64_t N, int64_t Np) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= BH * Np) return;
  const int64_t bh = i / Np, n = i % Np;
  float d = 0.f;
  if (n < N) {
    d = delta[bh * N + n];
    if (delta2) d += delta2[bh * N + n];
    if (wds) d += wds[bh * N + n] + wds[(BH + bh) * N + n];
  }
  dpx[i] = extra_row3(-d);
}

// ---- device pieces -----------------------------------------------------------------------------

// M = 128 x N = 64 product with K = 48 (80 with the residual half, lo_a or lo_b):
// a0/b0 are the K-major 64B-swizzled 32-channel blocks, ae/be the extra blocks
// (kExtra = false: K = 32 / 64, no extra block).
// acc0: add to what d holds (a second chain into the same accumulator).
template <bool kLoA, bool kExtra = true>
__device__ __forceinline__ void issue_dot64(uint32_t d, uint32_t a, uint32_t b, uint64_t ae, uint64_t be,
                                            uint32_t lo, uint32_t acc0 = 0) {
  constexpr uint32_t idesc = idesc_bf16(128, 64, false, false);
  mma_ss_w(d, sdesc(a, 16, 512, kSw64), sdesc(b, 16, 512, kSw64), idesc, acc0);
  mma_ss_w(d, sdesc(a + 32, 16, 512, kSw64), sdesc(b + 32, 16, 512, kSw64), idesc, 1);
  if (lo) {
    if (kLoA) {
      mma_ss_w(d, sdesc(lo, 16, 512, kSw64), sdesc(b, 16, 512, kSw64), idesc, 1);
      mma_ss_w(d, sdesc(lo + 32, 16, 512, kSw64), sdesc(b + 32, 16, 512, kSw64), idesc, 1);
    } else {
      mma_ss_w(d, sdesc(a, 16, 512, kSw64), sdesc(lo, 16, 512, kSw64), idesc, 1);
      mma_ss_w(d, sdesc(a + 32, 16, 512, kSw64), sdesc(lo + 32, 16, 512, kSw64), idesc, 1);
    }
  }
  if (kExtra) mma_ss_w(d, ae, be, idesc, 1);
}

// The same logits product with the slot side (A) in TMEM: tW holds a slot block's W'
// image as packed bf16 pairs, K steps of 8 columns: W' (2 steps), its residual (2), the
// extra block (1).  Only the point side (B) is read from shared memory.
__device__ __forceinline__ void issue_logits64_ts(uint32_t d, uint32_t tW, uint32_t b, uint64_t be, bool lo) {
  constexpr uint32_t idesc = idesc_bf16(128, 64, false, false);
  mma_ts_w(d, tW, sdesc(b, 16, 512, kSw64), idesc, 0u);
  mma_ts_w(d, tW + 8, sdesc(b + 32, 16, 512, kSw64), idesc, 1u);
  if (lo) {
    mma_ts_w(d, tW + 16, sdesc(b, 16, 512, kSw64), idesc, 1u);
    mma_ts_w(d, tW + 24, sdesc(b + 32, 16, 512, kSw64), idesc, 1u);
  }
  mma_ts_w(d, tW + 32, be, idesc, 1u);
}

// Point-extra descriptor (no swizzle, 16-byte rows) whose k = 8..15 half is the shared zero block.
__device__ __forceinline__ uint64_t px_desc(uint32_t px_s, uint32_t zero_s) { return sdesc(px_s, zero_s - px_s, 128, 0); }

// One 64-column unit of a TMEM lane: L (log2 weights) at tL, dw - delta at tD.
// da = 2^L (dw - delta) goes back in place into the L columns as bf16 pairs: columns
// [32 h, 32 h + 16) the hi halves of entries [32 h, 32 h + 32), [32 h + 16, 32 h + 32)
// their lo halves (kSplit).  kW: the weights too, into the dw columns, same layout.
// kSums: dt += sum da L, db += sum da.
template <bool kSplit, bool kW, bool kSums>
__device__ __forceinline__ void da_unit(uint32_t tL, uint32_t tD, float& dt, float& db) {
  // Pairs of entries go through the packed f32x2 forms (one instruction for both).
  const uint64_t neg1 = pack2(__float_as_uint(-1.f), __float_as_uint(-1.f));
#pragma unroll 1
  for (int h2 = 0; h2 < 2; h2++) {
    uint32_t l[32], dw[32];
    tmem_ld32(tL + 32 * h2, l);
    tmem_ld32(tD + 32 * h2, dw);
    tmem_wait_ld2(l, dw);
    uint32_t dh[16], dl[16], wh[16], wl[16];
    uint64_t t2 = 0, sb2 = 0;  // (+0, +0)
#pragma unroll
    for (int k = 0; k < 16; k++) {
      const uint64_t L2 = pack2(l[2 * k], l[2 * k + 1]);
      const uint64_t w2 = pack2(__float_as_uint(ex2(__uint_as_float(l[2 * k]))),
                                __float_as_uint(ex2(__uint_as_float(l[2 * k + 1]))));
      const uint64_t a2 = mul2(w2, pack2(dw[2 * k], dw[2 * k + 1]));
      if (kSums) {
        t2 = fma2(a2, L2, t2);
        sb2 = add2(sb2, a2);
      }
      const uint32_t p = pack_bf16(lo_f(a2), hi_f(a2));
      dh[k] = p;
      if (kSplit) {
        const uint64_t r2 = fma2(pack2(p << 16, p & 0xFFFF0000u), neg1, a2);  // a - bf16(a)
        dl[k] = pack_bf16(lo_f(r2), hi_f(r2));
      }
      if (kW) {
        const uint32_t q = pack_bf16(lo_f(w2), hi_f(w2));
        wh[k] = q;
        if (kSplit) {
          const uint64_t r2 = fma2(pack2(q << 16, q & 0xFFFF0000u), neg1, w2);
          wl[k] = pack_bf16(lo_f(r2), hi_f(r2));
        }
      }
    }
    tmem_st16(tL + 32 * h2, dh);
    if (kSplit) tmem_st16(tL + 32 * h2 + 16, dl);
    if (kW) {
      tmem_st16(tD + 32 * h2, wh);
      if (kSplit) tmem_st16(tD + 32 * h2 + 16, wl);
    }
    if (kSums) {
      dt += lo_f(t2) + hi_f(t2);
      db += lo_f(sb2) + hi_f(sb2);
    }
  }
}
// TMEM column (within a unit) of the hi pairs of K-step kk (16 entries).
__device__ __forceinline__ uint32_t da_col(int kk) { return (uint32_t)(32 * (kk >> 1) + 8 * (kk & 1)); }

// One 64-column unit of a TMEM lane: L (log2 weights) -> w = 2^L in place, as bf16
// pairs in da_unit's layout (hi pairs, then their residuals with kSplit).
template <bool kSplit>
__device__ __forceinline__ void w_unit(uint32_t tL) {
  const uint64_t neg1 = pack2(__float_as_uint(-1.f), __float_as_uint(-1.f));
#pragma unroll 1
  for (int h2 = 0; h2 < 2; h2++) {
    uint32_t l[32];
    tmem_ld32(tL + 32 * h2, l);
    tmem_wait_ld(l);
    uint32_t wh[16], wl[16];
#pragma unroll
    for (int k = 0; k < 16; k++) {
      const uint64_t w2 = pack2(__float_as_uint(ex2(__uint_as_float(l[2 * k]))),
                                __float_as_uint(ex2(__uint_as_float(l[2 * k + 1]))));
      const uint32_t q = pack_bf16(lo_f(w2), hi_f(w2));
      wh[k] = q;
      if (kSplit) {
        const uint64_t r2 = fma2(pack2(q << 16, q & 0xFFFF0000u), neg1, w2);
        wl[k] = pack_bf16(lo_f(r2), hi_f(r2));
      }
    }
    tmem_st16(tL + 32 * h2, wh);
    if (kSplit) tmem_st16(tL + 32 * h2 + 16, wl);
  }
}

// The slot pass's accumulators are flushed into registers every kSlotFlush of an
// issuer's units (64 points each), for the reason the slice's are: the tensor cores'
// fp32 accumulation drifts towards zero over a long chain of K steps.
constexpr int kSlotFlush = 8;
__device__ __forceinline__ bool slot_flush_at(int u) { return ((u >> 1) % kSlotFlush) == 0; }

// =========================================================================================
// Slot pass: CTA (slot block, point split p, bh) owns 128 slots.  Unit u is half
// u & 1 (64 points) of point tile u >> 1.  Per unit, warp 1 forms, transposed
// (M = 128 slots, N = 64 points, TMEM lane = slot),
//   L = a2 - lse2 (W block vs [x | 1, 1, -lse2]) and dw - delta (T block vs [v | 1, 1, -delta]);
// softmax warpgroup u % 2 turns them into da (and, MODE 1, w) in place and sums
// da (a2 - lse2) and da per slot in registers; warp 2 + u % 2 issues
//   dWx += da^T x   (K = points; x's 64B-swizzled tile read as an MN-major B operand)
//   MODE 1: dZ += w^T dO (the token gradient), from dO's tile the same way.
// Writes part[p][bh][g] = MODE 1: (dZ(32), dWx(32), sum da, 0); MODE 2: (dWx, sum da, 0)
// and dt_part[bh][p * R + block] = ln2 * sum over the block's slots of sum da (a2 - lse2).
// Two more modes serve fs_coupling_bwd:
//   MODE 0: the token gradient alone, dZ += w^T dO (no dw chain, no da): part = dZ(32);
//   MODE 3: da = da_D + da_S as in the combined point pass (dw - delta as two chains:
//     the deslice's T block against dO, the slice's T2 block against [fx | 1, 1, -delta]
//     (its extra block [dS_hi, dS_lo, 1, 1, 1] meets delta's rows), delta = delta_D +
//     delta_S), written like MODE 2.
// smem: [W block: hi 8K | extra 4K | lo 8K][T block: same][stages][zero 2K][red 1.5K][bars]
// TMEM: unit u uses set u % 3: L [128 s, +64), dw [128 s + 64, +64); accumulators
// dWx_j [384 + 32 j), dZ_j [448 + 32 j).
// =========================================================================================
template <int MODE, bool split>
__global__ void __launch_bounds__(kThreads, 1)
    k_bwd_slot_tc(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ CUtensorMap vmap,
                  const __grid_constant__ CUtensorMap pmap, const __grid_constant__ CUtensorMap dmap,
                  const __grid_constant__ CUtensorMap fmap, const uint8_t* __restrict__ wimg,
                  const uint8_t* __restrict__ timg, const uint8_t* __restrict__ timg2, float* __restrict__ part,
                  float* __restrict__ dt_part, int64_t N, int64_t Np, int H, int G, int splits,
                  uint32_t* status) {
  constexpr int kNSt = MODE == 3 ? kBStages - 1 : kBStages;    // stages (MODE 3's are larger)
  constexpr uint32_t kStgS = kBStage + (MODE == 3 ? kXBytes : 0u);  // x | v | px | dpx [| fx]
  const int g_base = blockIdx.x * kGC;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* s_w = smem;               // W block
  uint8_t* s_t = s_w + kWBlockB;     // T block
  uint8_t* s_t2 = s_t + kWBlockB;    // MODE 3: the slice's T block
  uint8_t* s_st = s_t2 + (MODE == 3 ? kWBlockB : 0u);  // stages
  uint8_t* s_zero = s_st + kNSt * kStgS;  // above the stages' point rows (positive LBO)
  float* s_red = reinterpret_cast<float*>(s_zero + kPxZero);  // 3 x 128 floats
  uint64_t* bars = reinterpret_cast<uint64_t*>(s_red + 3 * kGC);
  uint64_t* w_full = bars;
  uint64_t* x_full = bars + 1;
  uint64_t* st_empty = x_full + kNSt;
  uint64_t* s_full = st_empty + kNSt;
  uint64_t* p_ready = s_full + kSBuf;  // [issuer][set]
  uint64_t* pv_done = p_ready + 2 * kSBuf;
  uint64_t* acc_full = pv_done + kSBuf;
  uint64_t* acc_done = acc_full + 1;  // [issuer]: products of each of its units complete
  uint64_t* wt_ready = acc_done + 2;  // MODES 2, 3: the W' image is in TMEM
  uint64_t* drain = wt_ready + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 3);
  Abort* ab = reinterpret_cast<Abort*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const Work wk = work_of(N, splits, blockIdx.y, blockIdx.z);
  const int64_t b = wk.bh / H;
  const int h = (int)(wk.bh % H);
  const int units = 2 * wk.ntiles;
  // Accumulator flushes (as in the slice): issuer j's chain restarts every
  // kSlotFlush of its units after warpgroup j has added the accumulator into
  // registers.  MODE 1 keeps two accumulators per issuer (dW, dZ) and no flushes.
  constexpr bool kFl = MODE != 1;
  // MODES 2 and 3 keep no dZ accumulator, so its 64 TMEM columns hold slot-side images
  // and those MMAs read only their point side from shared memory: MODE 2 the W' image
  // (W', its residual, the extra block: 40 columns); MODE 3 W' and its residual (32)
  // and the deslice's T image and its residual (32), the two extra blocks staying in
  // shared memory.
  constexpr bool kWT = MODE == 2 || MODE == 3;
  constexpr bool kTT = MODE == 3;
  constexpr uint32_t kAccW = kSBuf * kGC, kAccZ = kAccW + 64;
  constexpr uint32_t kAccF = MODE == 0 ? kAccZ : kAccW;  // the flushed accumulator
  constexpr uint32_t kVOff = kXBytes, kPOff = 2 * kXBytes, kDOff = 2 * kXBytes + kPxBytes;

  if (threadIdx.x == 0) {
    mbar_init(w_full, 1);
    for (int s = 0; s < kNSt; s++) {
      mbar_init(&x_full[s], 1);
      mbar_init(&st_empty[s], 3);  // the logits issuer and both product issuers
    }
    for (int i = 0; i < kSBuf; i++) {
      mbar_init(&s_full[i], 1);
      mbar_init(&p_ready[i], 4);
      mbar_init(&p_ready[kSBuf + i], 4);
      mbar_init(&pv_done[i], 1);
    }
    mbar_init(acc_full, 2);
    mbar_init(&acc_done[0], 1);
    mbar_init(&acc_done[1], 1);
    mbar_init(wt_ready, 4);
    for (int i = 0; i < 3; i++) mbar_init(&drain[i], 1);
    ab->flag = 0;
    fence_mbar_init();
  }
  zero_smem(s_zero, kPxZero);
  fence_proxy_async_smem();
  if (warp == 1) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ------------------------------ producer ------------------------------
    if (lane == 0) {
      prefetch_tmap(&xmap);
      prefetch_tmap(&vmap);
      prefetch_tmap(&pmap);
      if (MODE != 0) prefetch_tmap(&dmap);
      if (MODE == 3) prefetch_tmap(&fmap);
      constexpr int kImages = MODE == 0 ? 1 : (MODE == 3 ? 3 : 2);  // W [, T [, T2]]
      mbar_expect_tx(w_full, kImages * kWBlockB);
      const uint8_t* ws = wimg + (size_t)h * G * kWRow;
      const uint8_t* ts = timg + (size_t)wk.bh * G * kWRow;
      const uint8_t* ts2 = MODE == 3 ? timg2 + (size_t)wk.bh * G * kWRow : nullptr;
      for (int im = 0; im < kImages; im++) {
        const uint8_t* src = im == 0 ? ws : (im == 1 ? ts : ts2);
        uint8_t* dst = im == 0 ? s_w : (im == 1 ? s_t : s_t2);
        load_images(dst, src + (size_t)g_base * 64, kGC * 64, w_full);
        load_images(dst + kGC * 64, src + (size_t)G * 64 + (size_t)g_base * 32, kGC * 32, w_full);
        load_images(dst + kGC * 96, src + (size_t)G * 96 + (size_t)g_base * 64, kGC * 64, w_full);
      }
      int i = 0;
      for (; i < wk.ntiles; i++) {
        const int s = i % kNSt;
        if (i >= kNSt && !mbar_wait(&st_empty[s], (uint32_t)(((i / kNSt) - 1) & 1), ab, status)) break;
        uint8_t* st = s_st + s * kStgS;
        const int n0 = (int)((wk.tile0 + i) * kTile);
        mbar_expect_tx(&x_full[s], MODE == 0 ? kBStage - kPxBytes : kStgS);
        tma_load_3d(st, &xmap, h * kD, n0, (int)b, &x_full[s]);
        tma_load_3d(st + kVOff, &vmap, h * kD, n0, (int)b, &x_full[s]);
        tma_load_2d(st + kPOff, &pmap, 0, (int)(wk.bh * Np + n0), &x_full[s]);
        if (MODE != 0) tma_load_2d(st + kDOff, &dmap, 0, (int)(wk.bh * Np + n0), &x_full[s]);
        if (MODE == 3) tma_load_3d(st + kBStage, &fmap, h * kD, n0, (int)b, &x_full[s]);
      }
      for (int j = (i > kNSt ? i - kNSt : 0); j < i; j++)
        mbar_wait(&x_full[j % kNSt], (uint32_t)((j / kNSt) & 1), ab, nullptr, kWaitNs);
      mbar_wait(w_full, 0, ab, nullptr, kWaitNs);
    }
  } else if (warp == 1) {
    // ------------------------------ logits and dw issuer ------------------------------
    const uint32_t sw = smem_u32(s_w), stt = smem_u32(s_t), stt2 = smem_u32(s_t2), sz = smem_u32(s_zero);
    bool ok = mbar_wait_w(w_full, 0, ab, status);
    if (kWT && ok) {
      ok = mbar_wait_w(wt_ready, 0, ab, status);
      tc_fence_after();
    }
    for (int u = 0; ok && u < units; u++) {
      const int i = u >> 1, half = u & 1;
      const int s = i % kNSt;
      const int bb = u % kSBuf;
      if (half == 0 && !(ok = mbar_wait_w(&x_full[s], (uint32_t)((i / kNSt) & 1), ab, status))) break;
      if (u >= kSBuf && !(ok = mbar_wait_w(&pv_done[bb], (uint32_t)(((u / kSBuf) - 1) & 1), ab, status))) break;
      tc_fence_after();
      const uint32_t st = smem_u32(s_st + s * kStgS);
      const uint32_t rows = (uint32_t)half * 64 * 64;     // the unit's 64 points in the 64-byte-row tiles
      const uint32_t prow = (uint32_t)half * 64 * 16;     // ... and in the 16-byte extra rows
      const uint32_t tL = tmem + (uint32_t)bb * kGC;
      if (kTT) {
        constexpr uint32_t idesc = idesc_bf16(128, 64, false, false);
        const uint32_t tW = tmem + kAccZ, tT = tW + 32;
        const uint32_t xb = st + rows, vb = st + kVOff + rows;
        mma_ts_w(tL, tW, sdesc(xb, 16, 512, kSw64), idesc, 0u);
        mma_ts_w(tL, tW + 8, sdesc(xb + 32, 16, 512, kSw64), idesc, 1u);
        if (split) {
          mma_ts_w(tL, tW + 16, sdesc(xb, 16, 512, kSw64), idesc, 1u);
          mma_ts_w(tL, tW + 24, sdesc(xb + 32, 16, 512, kSw64), idesc, 1u);
        }
        mma_ss_w(tL, sdesc(sw + kGC * 64, 16, 256, kSw32), px_desc(st + kPOff + prow, sz), idesc, 1u);
        // the deslice's chain: T (and its residual) from TMEM against dO, no extra block
        mma_ts_w(tL + 64, tT, sdesc(vb, 16, 512, kSw64), idesc, 0u);
        mma_ts_w(tL + 64, tT + 8, sdesc(vb + 32, 16, 512, kSw64), idesc, 1u);
        if (split) {
          mma_ts_w(tL + 64, tT + 16, sdesc(vb, 16, 512, kSw64), idesc, 1u);
          mma_ts_w(tL + 64, tT + 24, sdesc(vb + 32, 16, 512, kSw64), idesc, 1u);
        }
      } else if (kWT)
        issue_logits64_ts(tL, tmem + kAccZ, st + rows, px_desc(st + kPOff + prow, sz), split);
      else
        issue_dot64<true>(tL, sw, st + rows, sdesc(sw + kGC * 64, 16, 256, kSw32), px_desc(st + kPOff + prow, sz),
                          split ? sw + kGC * 96 : 0u);
      if (MODE == 1 || MODE == 2)
        issue_dot64<true>(tL + 64, stt, st + kVOff + rows, sdesc(stt + kGC * 64, 16, 256, kSw32),
                          px_desc(st + kDOff + prow, sz), split ? stt + kGC * 96 : 0u);
      if (MODE == 3) {
        // The deslice's T has c = 0, so its chain (issued above from TMEM) needs no extra
        // block: the slice's extra block [dS_hi, dS_lo, 1, 1, 1] against delta's rows
        // [1, 1, -delta parts] adds dS - delta in one K step.
        issue_dot64<true>(tL + 64, stt2, st + kBStage + rows, sdesc(stt2 + kGC * 64, 16, 256, kSw32),
                          px_desc(st + kDOff + prow, sz), split ? stt2 + kGC * 96 : 0u, 1u);
      }
      mma_commit_w(&s_full[bb]);
      if (half == 1) mma_commit_w(&st_empty[s]);
    }
    mma_commit_w(&drain[0]);
    mbar_wait_w(&drain[0], 0, ab, nullptr, kWaitNs);
  } else if (warp == 2 || warp == 3) {
    // ------------------------------ product issuers ------------------------------
    const int j = warp - 2;  // units u with u % 2 == j (half j of every tile)
    constexpr uint32_t idesc = idesc_bf16(128, kD, false, true);
    bool ok = true;
    for (int u = j; ok && u < units; u += 2) {
      const int i = u >> 1;
      const int s = i % kNSt;
      const int bb = u % kSBuf;
      // This issuer's units on set bb are 2 kSBuf apart.
      if (!(ok = mbar_wait_w(&p_ready[j * kSBuf + bb], (uint32_t)((u / (2 * kSBuf)) & 1), ab, status))) break;
      tc_fence_after();
      const uint32_t st = smem_u32(s_st + s * kStgS) + (uint32_t)j * 64 * 64;
      const uint32_t tL = tmem + (uint32_t)bb * kGC, tD = tL + 64;
#pragma unroll
      for (int kk = 0; kk < 4; kk++) {
        // 16 points: two 8-row groups of the 64B-swizzled tile (MN-major: channels contiguous).
        const uint64_t xd = sdesc(st + (uint32_t)kk * 1024, 4096, 512, kSw64);
        const bool fresh = u < 2 || (kFl && slot_flush_at(u));
        const uint32_t acc = (!fresh || kk > 0) ? 1u : 0u;
        if (MODE == 0) {  // the weights are in the L columns: dZ += w^T dO
          const uint64_t vd = sdesc(st + kVOff + (uint32_t)kk * 1024, 4096, 512, kSw64);
          mma_ts_w(tmem + kAccZ + (uint32_t)j * 32, tL + da_col(kk), vd, idesc, acc);
          if (split) mma_ts_w(tmem + kAccZ + (uint32_t)j * 32, tL + da_col(kk) + 16, vd, idesc, 1u);
          continue;
        }
        mma_ts_w(tmem + kAccW + (uint32_t)j * 32, tL + da_col(kk), xd, idesc, acc);
        if (split) mma_ts_w(tmem + kAccW + (uint32_t)j * 32, tL + da_col(kk) + 16, xd, idesc, 1u);
        if (MODE == 1) {
          const uint64_t vd = sdesc(st + kVOff + (uint32_t)kk * 1024, 4096, 512, kSw64);
          mma_ts_w(tmem + kAccZ + (uint32_t)j * 32, tD + da_col(kk), vd, idesc, acc);
          if (split) mma_ts_w(tmem + kAccZ + (uint32_t)j * 32, tD + da_col(kk) + 16, vd, idesc, 1u);
        }
      }
      mma_commit_w(&pv_done[bb]);
      mma_commit_w(&st_empty[s]);
      if (kFl) mma_commit_w(&acc_done[j]);
    }
    if (ok) mma_commit_w(acc_full);
    mma_commit_w(&drain[1 + j]);
    mbar_wait_w(&drain[1 + j], 0, ab, nullptr, kWaitNs);
  } else {
    // ------------------------------ softmax warpgroups ------------------------------
    const int wg = (warp - kSoftmaxWarp0) >> 2;
    const int wq = warp & 3;
    const int r = wq * 32 + lane;  // TMEM lane: slot g_base + r
    const uint32_t lane_addr = (uint32_t)(wq * 32) << 16;
    bool ok = true;
    float dt = 0.f, db = 0.f;
    if (kWT && wg == 0) {
      // Slot r's W' row from the block's image in shared memory (64B / 32B swizzled
      // rows) into TMEM columns [kAccZ, kAccZ + 48) of lane r: packed bf16 pairs of W'
      // (16), its residual (16), the extra block (8, then 8 zero columns).
      if ((ok = mbar_wait(w_full, 0, ab, status))) {
        const uint32_t tW = tmem + lane_addr + kAccZ;
        // a slot-block image's row r: bf16 pairs of the main half and of the residual
        auto copy_rows = [&](const uint8_t* img, uint32_t tdst) {
          uint32_t hi[16], lo[16];
#pragma unroll
          for (int c = 0; c < 16; c++) {
            hi[c] = *reinterpret_cast<const uint32_t*>(img + off_sw64(r, 2 * c));
            lo[c] = split ? *reinterpret_cast<const uint32_t*>(img + kGC * 96 + off_sw64(r, 2 * c)) : 0u;
          }
          tmem_st16(tdst, hi);
          tmem_st16(tdst + 16, lo);
        };
        copy_rows(s_w, tW);
        if (kTT) {
          copy_rows(s_t, tW + 32);
        } else {
          uint32_t ex[16];
#pragma unroll
          for (int c = 0; c < 16; c++)
            ex[c] = c < 8 ? *reinterpret_cast<const uint32_t*>(s_w + kGC * 64 + off_sw32(r, 2 * c)) : 0u;
          tmem_st16(tW + 32, ex);
        }
        tmem_wait_st();
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(wt_ready);
    }
    float acc[kD];  // this warpgroup's flushed share of dWx (MODE 0: dZ)
#pragma unroll
    for (int k = 0; k < kD; k++) acc[k] = 0.f;
    auto add_acc = [&]() {
      uint32_t a[32];
      tmem_ld32(tmem + lane_addr + kAccF + (uint32_t)wg * 32, a);
      tmem_wait_ld(a);
#pragma unroll
      for (int k = 0; k < kD; k++) acc[k] += __uint_as_float(a[k]);
    };
    for (int u = wg; ok && u < units; u += 2) {
      const int bb = u % kSBuf;
      if (!(ok = mbar_wait(&s_full[bb], (uint32_t)((u / kSBuf) & 1), ab, status))) break;
      tc_fence_after();
      const uint32_t tL = tmem + lane_addr + (uint32_t)bb * kGC;
      if (MODE == 0) {
        w_unit<split>(tL);
      } else {
        float t = 0.f, sb = 0.f;
        da_unit<split, MODE == 1, true>(tL, tL + 64, t, sb);
        dt += t;
        db += sb;
      }
      tmem_wait_st();
      if (kFl && u >= 2 && slot_flush_at(u)) {
        // This warpgroup's units up to u - 2 have completed their products.
        if (!(ok = mbar_wait(&acc_done[wg], (uint32_t)(((u - 2) >> 1) & 1), ab, status))) break;
        tc_fence_after();
        add_acc();
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_ready[wg * kSBuf + bb]);
    }
    // Epilogue.  Warpgroup 1 hands its sums dt, db to warpgroup 0 through shared
    // memory.  Flushed modes: each warpgroup adds what its accumulator holds since
    // its last flush; warpgroup 1 passes its share through the partial row and
    // warpgroup 0 adds the two in a fixed order (MODE 0: dZ; MODES 2, 3: dWx and the
    // sums).  MODE 1: warpgroup 0 writes dWx (both accumulators) and the sums,
    // warpgroup 1 dZ.
    const int64_t BH = gridDim.z;
    const int PS = MODE == 1 ? 2 * kD + 2 : (MODE == 0 ? kD : kD + 2);
    float* o = part + (((int64_t)blockIdx.y * BH + wk.bh) * G + g_base + r) * PS;
    const bool have = ok && wk.ntiles > 0 && mbar_wait(acc_full, 0, ab, status);
    if (have) tc_fence_after();
    if (kFl) {
      if (have) add_acc();
      if (wg == 1) {
#pragma unroll
        for (int k = 0; k < kD; k++) o[k] = acc[k];
        if (MODE != 0) {
          s_red[r] = dt;
          s_red[kGC + r] = db;
        }
      }
      named_barrier(1, 256);
      if (wg == 0) {
#pragma unroll
        for (int k = 0; k < kD; k++) o[k] = acc[k] + o[k];
        if (MODE != 0) {
          dt += s_red[r];
          db += s_red[kGC + r];
          o[kD] = db;
          o[kD + 1] = 0.f;
          s_red[2 * kGC + r] = dt;
          named_barrier(2, 128);
          if (r == 0) {
            float sum = 0.f;
            for (int k = 0; k < kGC; k++) sum += s_red[2 * kGC + k];
            dt_part[wk.bh * ((int64_t)gridDim.x * gridDim.y) + (int64_t)blockIdx.y * gridDim.x + blockIdx.x] =
                sum * kLn2;
          }
        }
      }
    } else {
      if (wg == 1) {
        s_red[r] = dt;
        s_red[kGC + r] = db;
      }
      named_barrier(1, 256);
      if (wg == 0) {
        dt += s_red[r];
        db += s_red[kGC + r];
        constexpr int off = kD;
        if (have) {
          uint32_t a0[32], a1[32];
          tmem_ld32(tmem + lane_addr + kAccW, a0);
          tmem_ld32(tmem + lane_addr + kAccW + 32, a1);
          tmem_wait_ld2(a0, a1);
#pragma unroll
          for (int k = 0; k < kD; k++) o[off + k] = __uint_as_float(a0[k]) + __uint_as_float(a1[k]);
        } else {
          for (int k = 0; k < kD; k++) o[off + k] = 0.f;
        }
        o[off + kD] = db;
        o[off + kD + 1] = 0.f;
        s_red[2 * kGC + r] = dt;
        named_barrier(2, 128);
        if (r == 0) {
          float sum = 0.f;
          for (int k = 0; k < kGC; k++) sum += s_red[2 * kGC + k];
          dt_part[wk.bh * ((int64_t)gridDim.x * gridDim.y) + (int64_t)blockIdx.y * gridDim.x + blockIdx.x] = sum * kLn2;
        }
      } else {
        if (have) {
          uint32_t z0[32], z1[32];
          tmem_ld32(tmem + lane_addr + kAccZ, z0);
          tmem_ld32(tmem + lane_addr + kAccZ + 32, z1);
          tmem_wait_ld2(z0, z1);
#pragma unroll
          for (int k = 0; k < kD; k++) o[k] = __uint_as_float(z0[k]) + __uint_as_float(z1[k]);
        } else {
          for (int k = 0; k < kD; k++) o[k] = 0.f;
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

// =========================================================================================
// Point pass: dx_n = ln2 * sum_g da_ng W'_g (W' = W log2(e)/tau).  CTA (split, bh)
// walks its point tiles; block q is (tile q / nb, 64-slot chunk q % nb).  Warp 1
// forms L (x tile vs W rows) and dw - delta (v tile vs T rows), M = 128 points,
// N = 64 slots, into set q % 3; softmax warpgroup q % 2 writes da in place (hi, lo
// pairs); warp 2 + j issues K-steps [2 j, 2 j + 2) of the chunk into O_j:
//   O_j += da W'^T (B: the W'^T image, channel rows, slots along K).
// kComb (the whole coupling's backward): da is the sum of the deslice's and the
// slice's, which share the weights, so one pass serves both: dw - delta is two chains
// into the same accumulator, dO against the deslice's T image (c = 0, so no extra
// block) and [fx | 1, 1, -delta] against the slice's (t = dU, c = dS): one extra K
// step adds dS - delta, with delta = delta_D + delta_S in the point rows.  Each stage
// also holds the fx tile.
// smem: [W img G x (96 | 160)][T img G x 96][kComb: T2 img G x 96][W'^T img G x 64]
//       [stages][zero 2K][bars]
// TMEM: sets [0, 384) of (L 64 | dw 64); O_(j, tile parity) at [384 + 32 (2 j + parity)).
// =========================================================================================
template <bool split, bool kComb = false>
__global__ void __launch_bounds__(kThreads, 1)
    k_bwd_dx_tc(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ CUtensorMap vmap,
                const __grid_constant__ CUtensorMap pmap, const __grid_constant__ CUtensorMap dmap,
                const __grid_constant__ CUtensorMap fmap, const uint8_t* __restrict__ wimg,
                const uint8_t* __restrict__ timg, const uint8_t* __restrict__ timg2,
                const uint8_t* __restrict__ wtimg, __nv_bfloat16* __restrict__ dx, int64_t N, int64_t Np, int H,
                int G, int splits, int hilo, int accumulate, uint32_t* status) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  constexpr uint32_t kStg = kBStage + (kComb ? kXBytes : 0u);  // x | v | px | dpx [| fx]
  const uint32_t wbytes = (uint32_t)G * (hilo ? kWRow : 96);
  uint8_t* s_w = smem;
  uint8_t* s_t = s_w + wbytes;
  uint8_t* s_t2 = s_t + (uint32_t)G * 96;
  uint8_t* s_wt = s_t2 + (kComb ? (uint32_t)G * 96 : 0u);
  uint8_t* s_st = s_wt + (uint32_t)G * 64;
  uint8_t* s_zero = s_st + kDxStages * kStg;
  uint64_t* bars = reinterpret_cast<uint64_t*>(s_zero + kPxZero);
  uint64_t* wz_full = bars;
  uint64_t* x_full = bars + 1;
  uint64_t* x_empty = x_full + kDxStages;
  uint64_t* s_full = x_empty + kDxStages;
  uint64_t* p_ready = s_full + kSBuf;
  uint64_t* pv_done = p_ready + kSBuf;
  uint64_t* o_full = pv_done + kSBuf;
  uint64_t* o_free = o_full + 2;
  uint64_t* drain = o_free + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 3);
  Abort* ab = reinterpret_cast<Abort*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const Work wk = work_of(N, splits, blockIdx.x, blockIdx.y);
  const int64_t b = wk.bh / H;
  const int h = (int)(wk.bh % H);
  const int nch = G / 64;
  const int total = wk.ntiles * nch;
  constexpr uint32_t kO = kSBuf * kGC;
  constexpr uint32_t kVOff = kXBytes, kPOff = 2 * kXBytes, kDOff = 2 * kXBytes + kPxBytes;

  if (threadIdx.x == 0) {
    mbar_init(wz_full, 1);
    for (int s = 0; s < kDxStages; s++) {
      mbar_init(&x_full[s], 1);
      mbar_init(&x_empty[s], 1);
    }
    for (int i = 0; i < kSBuf; i++) {
      mbar_init(&s_full[i], 1);
      mbar_init(&p_ready[i], 4);
      mbar_init(&pv_done[i], 2);
    }
    for (int i = 0; i < 2; i++) {
      mbar_init(&o_full[i], 2);
      mbar_init(&o_free[i], 4);
    }
    for (int i = 0; i < 3; i++) mbar_init(&drain[i], 1);
    ab->flag = 0;
    fence_mbar_init();
  }
  zero_smem(s_zero, kPxZero);
  fence_proxy_async_smem();
  if (warp == 1) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0 && wk.ntiles > 0) {
      prefetch_tmap(&xmap);
      prefetch_tmap(&vmap);
      prefetch_tmap(&pmap);
      prefetch_tmap(&dmap);
      if (kComb) prefetch_tmap(&fmap);
      mbar_expect_tx(wz_full, wbytes + (uint32_t)G * 96 * (kComb ? 2u : 1u) + (uint32_t)G * 64);
      load_images(s_w, wimg + (size_t)h * G * kWRow, wbytes, wz_full);
      load_images(s_t, timg + (size_t)wk.bh * G * kWRow, (uint32_t)G * 96, wz_full);
      if (kComb) load_images(s_t2, timg2 + (size_t)wk.bh * G * kWRow, (uint32_t)G * 96, wz_full);
      load_images(s_wt, wtimg + (size_t)h * G * 128, (uint32_t)G * 64, wz_full);
      int i = 0;
      for (; i < wk.ntiles; i++) {
        const int s = i % kDxStages;
        if (i >= kDxStages && !mbar_wait(&x_empty[s], (uint32_t)(((i / kDxStages) - 1) & 1), ab, status)) break;
        uint8_t* st = s_st + s * kStg;
        const int n0 = (int)((wk.tile0 + i) * kTile);
        mbar_expect_tx(&x_full[s], kStg);
        tma_load_3d(st, &xmap, h * kD, n0, (int)b, &x_full[s]);
        tma_load_3d(st + kVOff, &vmap, h * kD, n0, (int)b, &x_full[s]);
        tma_load_2d(st + kPOff, &pmap, 0, (int)(wk.bh * Np + n0), &x_full[s]);
        tma_load_2d(st + kDOff, &dmap, 0, (int)(wk.bh * Np + n0), &x_full[s]);
        if (kComb) tma_load_3d(st + kBStage, &fmap, h * kD, n0, (int)b, &x_full[s]);
      }
      for (int j = (i > kDxStages ? i - kDxStages : 0); j < i; j++)
        mbar_wait(&x_full[j % kDxStages], (uint32_t)((j / kDxStages) & 1), ab, nullptr, kWaitNs);
      mbar_wait(wz_full, 0, ab, nullptr, kWaitNs);
    }
  } else if (warp == 1) {
    if (wk.ntiles > 0) {
      const uint32_t sw = smem_u32(s_w), stt = smem_u32(s_t), stt2 = smem_u32(s_t2), sz = smem_u32(s_zero);
      bool ok = mbar_wait_w(wz_full, 0, ab, status);
      BlockPos pos(0, nch);
      for (int q = 0; ok && q < total; q++, pos.step(1, nch)) {
        const int i = pos.i, c = pos.c;
        const int s = i % kDxStages;
        const int bb = q % kSBuf;
        if (c == 0 && !(ok = mbar_wait_w(&x_full[s], (uint32_t)((i / kDxStages) & 1), ab, status))) break;
        if (q >= kSBuf && !(ok = mbar_wait_w(&pv_done[bb], (uint32_t)(((q / kSBuf) - 1) & 1), ab, status))) break;
        tc_fence_after();
        const uint32_t st = smem_u32(s_st + s * kStg);
        const uint32_t tL = tmem + (uint32_t)bb * kGC;
        const uint32_t rows = (uint32_t)c * 64 * 64, erows = (uint32_t)c * 64 * 32;
        issue_dot64<false>(tL, st, sw + rows, px_desc(st + kPOff, sz),
                           sdesc(sw + (uint32_t)G * 64 + erows, 16, 256, kSw32),
                           hilo ? sw + (uint32_t)G * 96 + rows : 0u);
        if (kComb) {
          // As in the slot pass: the deslice's chain without an extra block, the slice's
          // extra block against delta's rows (dS - delta in one K step).
          issue_dot64<false, false>(tL + 64, st + kVOff, stt + rows, 0ull, 0ull, 0u);
          issue_dot64<false>(tL + 64, st + kBStage, stt2 + rows, px_desc(st + kDOff, sz),
                             sdesc(stt2 + (uint32_t)G * 64 + erows, 16, 256, kSw32), 0u, 1u);
        } else {
          issue_dot64<false>(tL + 64, st + kVOff, stt + rows, px_desc(st + kDOff, sz),
                             sdesc(stt + (uint32_t)G * 64 + erows, 16, 256, kSw32), 0u);
        }
        mma_commit_w(&s_full[bb]);
        if (c == nch - 1) mma_commit_w(&x_empty[s]);
      }
      mma_commit_w(&drain[0]);
      mbar_wait_w(&drain[0], 0, ab, nullptr, kWaitNs);
    }
  } else if (warp == 2 || warp == 3) {
    const int j = warp - 2;
    if (wk.ntiles > 0) {
      constexpr uint32_t idesc = idesc_bf16(128, kD, false, false);
      const uint32_t swt = smem_u32(s_wt);
      bool ok = mbar_wait_w(wz_full, 0, ab, status);
      BlockPos pos(0, nch);
      for (int q = 0; ok && q < total; q++, pos.step(1, nch)) {
        const int i = pos.i, c = pos.c;
        const int ob = i & 1;
        const int bb = q % kSBuf;
        if (c == 0 && i >= 2 && !(ok = mbar_wait_w(&o_free[ob], (uint32_t)(((i >> 1) - 1) & 1), ab, status))) break;
        if (!(ok = mbar_wait_w(&p_ready[bb], (uint32_t)((q / kSBuf) & 1), ab, status))) break;
        tc_fence_after();
        const uint32_t tL = tmem + (uint32_t)bb * kGC;
        const uint32_t tO = tmem + kO + (uint32_t)(j * 2 + ob) * kD;
#pragma unroll
        for (int e = 0; e < 2; e++) {
          const int kk = 2 * j + e;
          const uint64_t bd = sdesc(swt + (uint32_t)c * 4096 + (uint32_t)kk * 32, 16, 1024, kSw128);
          mma_ts_w(tO, tL + da_col(kk), bd, idesc, (c > 0 || e > 0) ? 1u : 0u);
          if (split) mma_ts_w(tO, tL + da_col(kk) + 16, bd, idesc, 1u);
        }
        mma_commit_w(&pv_done[bb]);
        if (c == nch - 1) mma_commit_w(&o_full[ob]);
      }
      mma_commit_w(&drain[1 + j]);
      mbar_wait_w(&drain[1 + j], 0, ab, nullptr, kWaitNs);
    }
  } else {
    const int wg = (warp - kSoftmaxWarp0) >> 2;
    const int wq = warp & 3;
    const int r = wq * 32 + lane;
    const uint32_t lane_addr = (uint32_t)(wq * 32) << 16;
    bool ok = true;
    auto epilogue = [&](int t) -> bool {
      const int ob = t & 1;
      if (!mbar_wait(&o_full[ob], (uint32_t)((t >> 1) & 1), ab, status)) return false;
      tc_fence_after();
      uint32_t o0[32], o1[32];
      tmem_ld32(tmem + lane_addr + kO + (uint32_t)ob * kD, o0);
      tmem_ld32(tmem + lane_addr + kO + (uint32_t)(2 + ob) * kD, o1);
      tmem_wait_ld2(o0, o1);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&o_free[ob]);
      const int64_t n = (wk.tile0 + t) * kTile + r;
      if (n < N) {
        uint4* dst = reinterpret_cast<uint4*>(dx + ((b * N + n) * H + h) * kD);
        float add[kD];
#pragma unroll
        for (int k = 0; k < kD; k++) add[k] = 0.f;
        if (accumulate) {
#pragma unroll
          for (int k = 0; k < 4; k++) {
            const uint4 q4 = dst[k];
            const uint32_t w[4] = {q4.x, q4.y, q4.z, q4.w};
#pragma unroll
            for (int e = 0; e < 4; e++) {
              add[8 * k + 2 * e] = __uint_as_float(w[e] << 16);
              add[8 * k + 2 * e + 1] = __uint_as_float(w[e] & 0xFFFF0000u);
            }
          }
        }
#pragma unroll
        for (int k = 0; k < 4; k++) {
          uint32_t w[4];
#pragma unroll
          for (int e = 0; e < 4; e++) {
            const int c0 = 8 * k + 2 * e;
            w[e] = pack_bf16(fmaf(__uint_as_float(o0[c0]) + __uint_as_float(o1[c0]), kLn2, add[c0]),
                             fmaf(__uint_as_float(o0[c0 + 1]) + __uint_as_float(o1[c0 + 1]), kLn2, add[c0 + 1]));
          }
          dst[k] = make_uint4(w[0], w[1], w[2], w[3]);
        }
      }
      return true;
    };
    BlockPos pos(wg, nch);
    for (int q = wg; ok && q < total; q += 2, pos.step(2, nch)) {
      const int i = pos.i, c = pos.c;
      const int bb = q % kSBuf;
      if (!(ok = mbar_wait(&s_full[bb], (uint32_t)((q / kSBuf) & 1), ab, status))) break;
      tc_fence_after();
      const uint32_t tL = tmem + lane_addr + (uint32_t)bb * kGC;
      float unused0 = 0.f, unused1 = 0.f;
      da_unit<split, false, false>(tL, tL + 64, unused0, unused1);
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_ready[bb]);
      if (c == 0 && i > 0 && !(ok = epilogue(i - 1))) break;
    }
    if (ok && total > 0 && total % 2 == wg) epilogue(wk.ntiles - 1);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

// ---- host side ---------------------------------------------------------------------------------

size_t smem_bwd_slot(int mode = 1) {
  const bool m3 = mode == 3;
  return 1024 + (m3 ? 3 : 2) * (size_t)kWBlockB + (m3 ? kBStages - 1 : kBStages) * (size_t)(kBStage + (m3 ? kXBytes : 0)) +
         kPxZero + 3 * kGC * 4 + 512;
}
size_t smem_bwd_dx(int G, bool hilo, bool comb = false) {
  return 1024 + (size_t)G * ((hilo ? kWRow : 96) + 96 * (comb ? 2 : 1) + 64) +
         kDxStages * (size_t)(kBStage + (comb ? kXBytes : 0)) + kPxZero + 512;
}

int bwd_slot_blocks(const Shape& s) { return s.G / kGC; }
int bwd_slot_splits(const Shape& s) { return point_splits(s, (int)(s.BH() * bwd_slot_blocks(s))); }

// Slot ranges.  The point pass holds three images of its slots in shared memory,
// which fits up to kBwdSlotsMax slots.  A larger G runs every pass over ranges of
// `size` slots (a multiple of 128; the last range may hold fewer real slots), all
// with the full problem's lse, so that the weights of a range are those of the
// softmax over all G.  The sums over slots (delta, dfx, dx) add up over the
// ranges; the slot-owned gradients of a range are its own.  `size` minimises the
// padded slots plus half a block per range (a range re-reads x and v); ties go to
// the larger size.
constexpr int kBwdSlotsMax = 640;
struct SlotRanges {
  int n, size;
};
SlotRanges slot_ranges(int G) {
  if (G <= kBwdSlotsMax) return {1, (G + kGC - 1) / kGC * kGC};
  SlotRanges best{0, 0};
  for (int size = kGC; size <= kBwdSlotsMax; size += kGC) {
    const int n = (G + size - 1) / size;
    if (best.n == 0 || (int64_t)n * (size + kGC / 2) <= (int64_t)best.n * (best.size + kGC / 2)) best = {n, size};
  }
  return best;
}

// The backward forms every weight with split products whatever the forward's
// arithmetic: its lse comes from split products (recomputed when the forward's
// did not), and weights from bf16 logits would not sum to one against it; the
// excess would bias the gradients that are sums of cancelling terms (dbias, dtau).
Shape split_shape(const Shape& s) {
  Shape r = s;
  r.dot = FS_DOT_BF16X2;
  return r;
}

// The shape the passes see: split products, G = the slot range.
Shape pass_shape(const Shape& s0) {
  Shape s = split_shape(s0);
  s.G = slot_ranges(s0.G).size;
  return s;
}

// Workspace layout of one tensor-core backward call (offsets from the tc region).
// With several slot ranges it also holds a range's slice of W, bias and t (wc, bc,
// tc) and its slot-owned gradients (dwc, dbc, dzc) before they go to their places.
struct BwdLayout {
  size_t wimg, wtimg, timg, zimg, px, dpx, delta, wds, ds, dtp, part, wc, bc, tc, dwc, dbc, dzc, total;
};
BwdLayout bwd_layout(const Shape& s0, int mode) {
  BwdLayout L{};
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = align_up(off + bytes, 256);
    return o;
  };
  const Shape s = pass_shape(s0);
  const size_t BHG = (size_t)s.BH() * s.G;
  const size_t pts = (size_t)s.BH() * s.N;
  const int P = bwd_slot_splits(s), R = bwd_slot_blocks(s);
  L.wimg = take(w_image_bytes(s));
  L.wtimg = take((size_t)s.H * s.G * 128);
  L.timg = take(BHG * kWRow);
  L.zimg = take(BHG * 128);
  L.px = take(px_bytes(s));
  L.dpx = take(px_bytes(s));
  L.delta = take(pts * sizeof(float));
  L.wds = take(mode == 2 ? 2 * pts * sizeof(float) : 0);
  L.ds = take(BHG * sizeof(float));
  L.dtp = take((size_t)s.BH() * P * R * sizeof(float));
  L.part = take((size_t)P * BHG * (mode == 1 ? 2 * kD + 2 : kD + 2) * sizeof(float));
  const size_t rs = slot_ranges(s0.G).n > 1 ? (size_t)s.G : 0;
  L.wc = take((size_t)s.H * kD * rs * sizeof(float));
  L.bc = take((size_t)s.H * rs * sizeof(float));
  L.tc = take((size_t)s.BH() * rs * (kD + 1) * sizeof(float));
  L.dwc = take((size_t)s.H * kD * rs * sizeof(float));
  L.dbc = take((size_t)s.H * rs * sizeof(float));
  L.dzc = take(mode == 1 ? (size_t)s.BH() * rs * kD * sizeof(float) : 0);
  L.total = off;
  return L;
}

bool make_maps(const Shape& s, const void* x, const void* v, const void* px, const void* dpx, CUtensorMap* xmap,
               CUtensorMap* vmap, CUtensorMap* pmap, CUtensorMap* dmap) {
  const int64_t Np = padded_n(s);
  return make_point_map(xmap, x, s, kD, CU_TENSOR_MAP_SWIZZLE_64B) &&
         make_point_map(vmap, v, s, kD, CU_TENSOR_MAP_SWIZZLE_64B) && make_px_map(pmap, px, s.BH(), Np) &&
         make_px_map(dmap, dpx, s.BH(), Np);
}

// Slot-side images of t (T image, its c column, Z-layout image) for G slots.
cudaError_t prep_t_images(const Shape& s, int G, const float* t, int tstride, int has_c, uint8_t* ws,
                          const BwdLayout& L, cudaStream_t st) {
  const int64_t BHG = s.BH() * s.G;
  k_prep_t<<<(unsigned)((BHG + 127) / 128), 128, 0, st>>>(t, tstride, has_c, ws + L.timg,
                                                            reinterpret_cast<float*>(ws + L.ds), s.BH(), G, s.G);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_prep_z2<<<(unsigned)((BHG * kD + 255) / 256), 256, 0, st>>>(t, tstride, ws + L.zimg, s.BH(), G, s.G);
  return cudaGetLastError();
}

// One backward call: mode 1 (deslice; t = z', v = dO, writes dzp) or 2 (slice; t =
// dU | dS with tstride 33, v = fx, writes dfx).  t: [BH][G][tstride] fp32.
//   1. lse rows; for each slot range: its images, then the rows pass (delta, dfx
//      and the wds partials add up over the ranges);
//   2. delta's rows; for each slot range: the slot pass, its reduction into the
//      range's dW, dbias, dtau (and dz') partials, and the point pass (dx; skipped
//      when dx is null).
// delta_out: where delta goes (null: the layout's own buffer).
cudaError_t run_backward(const Shape& s0, int mode, const void* x, const void* v, const float* W,
                         const float* bias, const float* tau, const float* t, int tstride, const float* lse,
                         void* dfx, void* dx, float* dzp, float* dW, float* db, float* dtau, int accumulate,
                         uint8_t* ws, uint32_t* status, cudaStream_t st, float* delta_out = nullptr) {
  const SlotRanges sr = slot_ranges(s0.G);
  const Shape s = pass_shape(s0);
  const BwdLayout L = bwd_layout(s0, mode);
  const bool ranged = sr.n > 1;
  const int64_t Np = padded_n(s);
  const int64_t npx = s.BH() * Np;
  const int has_c = mode == 2 ? 1 : 0;
  cudaError_t e;
  auto range_g = [&](int k) { return k < sr.n - 1 ? sr.size : s0.G - (sr.n - 1) * sr.size; };

  // Images of range k: t's, W's (and W'^T's when wt).
  auto prep_range = [&](int k, bool wt) -> cudaError_t {
    const int g0 = k * sr.size, G = range_g(k);
    const float *Wk = W, *bk = bias, *tk = t;
    cudaError_t r;
    if (ranged) {
      float* wc = reinterpret_cast<float*>(ws + L.wc);
      float* bc = reinterpret_cast<float*>(ws + L.bc);
      float* tc = reinterpret_cast<float*>(ws + L.tc);
      if ((r = copy_rows(wc, G, W + g0, s0.G, G, (int64_t)s.H * kD, st)) != cudaSuccess) return r;
      if ((r = copy_rows(bc, G, bias + g0, s0.G, G, s.H, st)) != cudaSuccess) return r;
      if ((r = copy_rows(tc, (int64_t)G * tstride, t + (int64_t)g0 * tstride, (int64_t)s0.G * tstride,
                         (int64_t)G * tstride, s.BH(), st)) != cudaSuccess)
        return r;
      Wk = wc, bk = bc, tk = tc;
    }
    if ((r = prep_t_images(s, G, tk, tstride, has_c, ws, L, st)) != cudaSuccess) return r;
    if ((r = prep_w(s, G, Wk, bk, tau, ws + L.wimg, status, st)) != cudaSuccess) return r;
    if (wt) {
      const int64_t nwt = (int64_t)s.H * kD * s.G;
      k_prep_wt<<<(unsigned)((nwt + 255) / 256), 256, 0, st>>>(Wk, tau, ws + L.wtimg, s.H, G, s.G, status);
      r = cudaGetLastError();
    }
    return r;
  };

  k_prep_px<<<(unsigned)((npx + 255) / 256), 256, 0, st>>>(lse, reinterpret_cast<uint4*>(ws + L.px), s.BH(), s.N,
                                                             Np);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  float* delta = delta_out ? delta_out : reinterpret_cast<float*>(ws + L.delta);
  float* wds = mode == 2 ? reinterpret_cast<float*>(ws + L.wds) : nullptr;
  if (wds && (e = cudaMemsetAsync(wds, 0, 2 * (size_t)s.BH() * s.N * sizeof(float), st)) != cudaSuccess) return e;
  for (int k = 0; k < sr.n; k++) {
    if ((e = prep_range(k, false)) != cudaSuccess) return e;
    if ((e = tc_rows_bwd(s, mode, x, ws + L.wimg, ws + L.zimg, ws + L.px, v, dfx, delta, wds,
                         reinterpret_cast<const float*>(ws + L.ds), k > 0 ? 1 : 0, status, st)) != cudaSuccess)
      return e;
  }
  k_prep_dpx<<<(unsigned)((npx + 255) / 256), 256, 0, st>>>(delta, nullptr, wds,
                                                              reinterpret_cast<uint4*>(ws + L.dpx), s.BH(), s.N, Np);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;

  CUtensorMap xmap, vmap, pmap, dmap;
  if (!make_maps(s, x, v, ws + L.px, ws + L.dpx, &xmap, &vmap, &pmap, &dmap)) return cudaErrorInvalidValue;
  const int R = bwd_slot_blocks(s), P = bwd_slot_splits(s);
  for (int k = 0; k < sr.n; k++) {
    const int g0 = k * sr.size, G = range_g(k);
    // The images of the last range are still in place after the rows passes; W'^T
    // (for the point pass, when dx is wanted) is not.
    if (ranged) {
      if ((e = prep_range(k, dx != nullptr)) != cudaSuccess) return e;
    } else if (dx) {
      const int64_t nwt = (int64_t)s.H * kD * s.G;
      k_prep_wt<<<(unsigned)((nwt + 255) / 256), 256, 0, st>>>(W, tau, ws + L.wtimg, s.H, G, s.G, status);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    {
      const size_t sm = smem_bwd_slot(mode);
      const auto kernel = mode == 1 ? k_bwd_slot_tc<1, true> : k_bwd_slot_tc<2, true>;
      if ((e = set_smem(kernel, sm)) != cudaSuccess) return e;
      kernel<<<dim3((unsigned)R, (unsigned)P, (unsigned)s.BH()), kThreads, sm, st>>>(
          xmap, vmap, pmap, dmap, xmap, ws + L.wimg, ws + L.timg, nullptr, reinterpret_cast<float*>(ws + L.part),
          reinterpret_cast<float*>(ws + L.dtp), s.N, Np, s.H, s.G, P, status);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    // The slot-owned gradients of range k: straight into dW, dbias (and dz') with
    // one range; else into the range's buffers (holding dW, dbias's values when
    // they are added to), then to their places.  dtau sums over the ranges.
    const int acc = accumulate || k > 0;
    Shape sk = s0;
    sk.G = G;
    float *dWk = dW, *dbk = db, *dzk = dzp;
    if (ranged) {
      dWk = reinterpret_cast<float*>(ws + L.dwc);
      dbk = reinterpret_cast<float*>(ws + L.dbc);
      dzk = mode == 1 ? reinterpret_cast<float*>(ws + L.dzc) : nullptr;
      if (accumulate) {
        if ((e = copy_rows(dWk, G, dW + g0, s0.G, G, (int64_t)s.H * kD, st)) != cudaSuccess) return e;
        if ((e = copy_rows(dbk, G, db + g0, s0.G, G, s.H, st)) != cudaSuccess) return e;
      } else if (acc) {
        if ((e = cudaMemsetAsync(dWk, 0, (size_t)s.H * kD * G * sizeof(float), st)) != cudaSuccess) return e;
        if ((e = cudaMemsetAsync(dbk, 0, (size_t)s.H * G * sizeof(float), st)) != cudaSuccess) return e;
      }
    }
    if ((e = simt_reduce_bwd(sk, P, reinterpret_cast<const float*>(ws + L.part), s.G,
                             mode == 1 ? 2 * kD + 2 : kD + 2, mode == 1 ? 1 : 0, tau, dzk, dWk, dbk, dtau,
                             reinterpret_cast<const float*>(ws + L.dtp), (int64_t)P * R, acc, st)) != cudaSuccess)
      return e;
    if (ranged) {
      if ((e = copy_rows(dW + g0, s0.G, dWk, G, G, (int64_t)s.H * kD, st)) != cudaSuccess) return e;
      if ((e = copy_rows(db + g0, s0.G, dbk, G, G, s.H, st)) != cudaSuccess) return e;
      if (mode == 1 && (e = copy_rows(dzp + (int64_t)g0 * kD, (int64_t)s0.G * kD, dzk, (int64_t)G * kD,
                                      (int64_t)G * kD, s.BH(), st)) != cudaSuccess)
        return e;
    }
    if (dx) {
      const bool hilo = smem_bwd_dx(s.G, true) <= kMaxSmem;
      const size_t sm = smem_bwd_dx(s.G, hilo);
      const int Pd = point_splits(s, (int)s.BH());
      const auto kernel = k_bwd_dx_tc<true>;
      if ((e = set_smem(kernel, sm)) != cudaSuccess) return e;
      kernel<<<dim3((unsigned)Pd, (unsigned)s.BH()), kThreads, sm, st>>>(
          xmap, vmap, pmap, dmap, xmap, ws + L.wimg, ws + L.timg, nullptr, ws + L.wtimg,
          static_cast<__nv_bfloat16*>(dx), s.N, Np, s.H, s.G, Pd, hilo ? 1 : 0, acc, status);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
  }
  return cudaSuccess;
}

// The coupling's backward in one call (fs_coupling_bwd).  The deslice's and the
// slice's da share the weights, so their slot-owned and point-owned products can be
// formed once from da_D + da_S; what has to come first is d z' (it feeds the mix
// backward, and so dU, dS and the slice's part).  Per slot range (as in the separate
// calls):
//   1. the deslice part's rows pass: delta_D;
//   2. d z' = sum_n w_ng dO_n: the forward's slice with dO for fx (its unnormalised
//      numerators) where the forward's kernels take the shape, else the slot pass in
//      mode 0 (the weights alone);
//   3. the mix backward and the dU | dS prologue;
//   4. the slice part's rows pass: delta_S, dfx, the sum_g w dS partials;
//   5. delta = delta_S + delta_D + sum_g w dS into the point rows;
//   6. the slot pass in mode 3: dW, dbias, dtau of da_D + da_S;
//   7. one point pass (k_bwd_dx_tc<., true>) for dx, over ranges of at most 256
//      slots (it holds two T images besides W' and W'^T).
constexpr int kCombSlotsMax = 256;
SlotRanges comb_ranges(const Shape& s0) {
  const int cap = std::min(kCombSlotsMax, pass_shape(s0).G);
  const int Gp = (s0.G + kGC - 1) / kGC * kGC;
  if (Gp <= cap) return {1, Gp};
  SlotRanges best{0, 0};
  for (int size = kGC; size <= cap; size += kGC) {
    const int n = (s0.G + size - 1) / size;
    if (best.n == 0 || (int64_t)n * (size + kGC / 2) <= (int64_t)best.n * (best.size + kGC / 2)) best = {n, size};
  }
  return best;
}

// Workspace of the coupling backward: the slice backward's layout, then delta_D, a
// second T image (the slice's, beside the deslice's), the ranges' d z' slices, and a
// range's slices of W, bias, z' and dU | dS (for the passes' ranges and the point
// pass's, whichever are larger).
struct CoupLayout {
  size_t deltaD, timg2, dzc, wc, bc, zc, uc, sl_part, sl_prep, sl_wsum, total;
};
CoupLayout coup_layout(const Shape& s0) {
  CoupLayout C{};
  size_t off = bwd_layout(s0, 2).total;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = align_up(off + bytes, 256);
    return o;
  };
  const Shape s = pass_shape(s0);
  const SlotRanges sr = slot_ranges(s0.G), cr = comb_ranges(s0);
  const size_t rp = sr.n > 1 ? (size_t)sr.size : 0;
  const size_t rs = std::max(rp, cr.n > 1 ? (size_t)cr.size : 0);
  C.deltaD = take((size_t)s.BH() * s.N * sizeof(float));
  C.timg2 = take((size_t)s.BH() * std::max(s.G, cr.size) * kWRow);
  C.dzc = take((size_t)s.BH() * rp * kD * sizeof(float));
  C.wc = take((size_t)s.H * kD * rs * sizeof(float));
  C.bc = take((size_t)s.H * rs * sizeof(float));
  C.zc = take((size_t)s.BH() * rs * kD * sizeof(float));
  C.uc = take((size_t)s.BH() * rs * (kD + 1) * sizeof(float));
  // d z' through the forward's slice (split products, as the backward's weights)
  const Shape ss = split_shape(s0);
  const bool via_slice = tc_forward_supported(ss);
  C.sl_part = take(via_slice ? tc_slice_partials_bytes(ss) : 0);
  C.sl_prep = take(via_slice ? tc_slice_prep_bytes(ss) : 0);
  C.sl_wsum = take(via_slice ? (size_t)s.BH() * s0.G * sizeof(float) : 0);
  C.total = off;
  return C;
}

cudaError_t run_coupling_bwd(const Shape& s0, const void* x, const void* f, const void* dout, const float* W,
                             const float* bias, const float* tau, const float* M, const float* z, const float* wsum,
                             const float* zp, const float* lse, float* dzp, float* dz, float* dM, void* dx, void* dfx,
                             float* dW, float* db, float* dtau, int accumulate, float* dUS, uint8_t* ws,
                             uint32_t* status, cudaStream_t st) {
  const SlotRanges sr = slot_ranges(s0.G);
  const Shape s = pass_shape(s0);
  const BwdLayout L = bwd_layout(s0, 2);
  const CoupLayout C = coup_layout(s0);
  const bool ranged = sr.n > 1;
  const int64_t Np = padded_n(s), npx = s.BH() * Np;
  float* deltaD = reinterpret_cast<float*>(ws + C.deltaD);
  float* deltaS = reinterpret_cast<float*>(ws + L.delta);
  float* wds = reinterpret_cast<float*>(ws + L.wds);
  float* wc = reinterpret_cast<float*>(ws + C.wc);
  float* bc = reinterpret_cast<float*>(ws + C.bc);
  float* zc = reinterpret_cast<float*>(ws + C.zc);
  float* uc = reinterpret_cast<float*>(ws + C.uc);
  cudaError_t e;
  // Slices [g0, g0 + G) of W, bias, z' and dU | dS (the gathered ones when `slice`).
  struct Src {
    const float *W, *b, *z, *u;
  };
  auto gather = [&](int g0, int G, bool slice, bool wz, bool zt, bool ut, Src* o) -> cudaError_t {
    *o = {W, bias, zp, dUS};
    if (!slice) return cudaSuccess;
    cudaError_t r;
    if (wz) {
      if ((r = copy_rows(wc, G, W + g0, s0.G, G, (int64_t)s.H * kD, st)) != cudaSuccess) return r;
      if ((r = copy_rows(bc, G, bias + g0, s0.G, G, s.H, st)) != cudaSuccess) return r;
      o->W = wc, o->b = bc;
    }
    if (zt) {
      if ((r = copy_rows(zc, (int64_t)G * kD, zp + (int64_t)g0 * kD, (int64_t)s0.G * kD, (int64_t)G * kD, s.BH(),
                         st)) != cudaSuccess)
        return r;
      o->z = zc;
    }
    if (ut) {
      if ((r = copy_rows(uc, (int64_t)G * (kD + 1), dUS + (int64_t)g0 * (kD + 1), (int64_t)s0.G * (kD + 1),
                         (int64_t)G * (kD + 1), s.BH(), st)) != cudaSuccess)
        return r;
      o->u = uc;
    }
    return cudaSuccess;
  };
  auto range_g = [&](int k) { return k < sr.n - 1 ? sr.size : s0.G - (sr.n - 1) * sr.size; };

  k_prep_px<<<(unsigned)((npx + 255) / 256), 256, 0, st>>>(lse, reinterpret_cast<uint4*>(ws + L.px), s.BH(), s.N,
                                                             Np);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  // 1. delta_D
  for (int k = 0; k < sr.n; k++) {
    const int g0 = k * sr.size, G = range_g(k);
    Src a;
    if ((e = gather(g0, G, ranged, true, true, false, &a)) != cudaSuccess) return e;
    if ((e = prep_w(s, G, a.W, a.b, tau, ws + L.wimg, status, st)) != cudaSuccess) return e;
    if ((e = prep_t_images(s, G, a.z, kD, 0, ws, L, st)) != cudaSuccess) return e;
    if ((e = tc_rows_bwd(s, 1, x, ws + L.wimg, ws + L.zimg, ws + L.px, dout, nullptr, deltaD, nullptr,
                         reinterpret_cast<const float*>(ws + L.ds), k > 0 ? 1 : 0, status, st)) != cudaSuccess)
      return e;
  }
  const int R = bwd_slot_blocks(s), P = bwd_slot_splits(s);
  CUtensorMap xmap, vmap, pmap, dmap, fmap;
  if (!make_maps(s, x, dout, ws + L.px, ws + L.dpx, &xmap, &vmap, &pmap, &dmap) ||
      !make_point_map(&fmap, f, s, kD, CU_TENSOR_MAP_SWIZZLE_64B))
    return cudaErrorInvalidValue;
  // 2. d z'
  const Shape ssl = split_shape(s0);
  if (tc_forward_supported(ssl)) {
    if ((e = tc_slice_fwd_lse(ssl, x, dout, W, bias, tau, lse, dzp, reinterpret_cast<float*>(ws + C.sl_wsum), 0,
                              reinterpret_cast<float*>(ws + C.sl_part), ws + C.sl_prep, status, st)) != cudaSuccess)
      return e;
  } else {  // the slot pass in mode 0 (the W image of the last range is in place)
    const size_t sm = smem_bwd_slot(0);
    const auto kernel = k_bwd_slot_tc<0, true>;
    if ((e = set_smem(kernel, sm)) != cudaSuccess) return e;
    for (int k = 0; k < sr.n; k++) {
      const int g0 = k * sr.size, G = range_g(k);
      if (ranged) {
        Src a;
        if ((e = gather(g0, G, true, true, false, false, &a)) != cudaSuccess) return e;
        if ((e = prep_w(s, G, a.W, a.b, tau, ws + L.wimg, status, st)) != cudaSuccess) return e;
      }
      kernel<<<dim3((unsigned)R, (unsigned)P, (unsigned)s.BH()), kThreads, sm, st>>>(
          xmap, vmap, pmap, pmap, xmap, ws + L.wimg, ws + L.timg, nullptr, reinterpret_cast<float*>(ws + L.part),
          reinterpret_cast<float*>(ws + L.dtp), s.N, Np, s.H, s.G, P, status);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
      Shape sk = s0;
      sk.G = G;
      float* dzk = ranged ? reinterpret_cast<float*>(ws + C.dzc) : dzp;
      if ((e = simt_reduce_dzp(sk, P, reinterpret_cast<const float*>(ws + L.part), s.G, kD, dzk, st)) != cudaSuccess)
        return e;
      if (ranged && (e = copy_rows(dzp + (int64_t)g0 * kD, (int64_t)s0.G * kD, dzk, (int64_t)G * kD, (int64_t)G * kD,
                                   s.BH(), st)) != cudaSuccess)
        return e;
    }
  }
  // 3. the mix backward and dU | dS
  if ((e = simt_mix_bwd(s0, M, z, dzp, dz, dM, st)) != cudaSuccess) return e;
  if ((e = simt_slice_bwd_prep(s0, z, wsum, dz, dUS, st)) != cudaSuccess) return e;
  // 4. delta_S, dfx, sum_g w dS
  if ((e = cudaMemsetAsync(wds, 0, 2 * (size_t)s.BH() * s.N * sizeof(float), st)) != cudaSuccess) return e;
  for (int k = 0; k < sr.n; k++) {
    const int g0 = k * sr.size, G = range_g(k);
    Src a;
    if ((e = gather(g0, G, ranged, true, false, true, &a)) != cudaSuccess) return e;
    if ((e = prep_w(s, G, a.W, a.b, tau, ws + L.wimg, status, st)) != cudaSuccess) return e;
    if ((e = prep_t_images(s, G, a.u, kD + 1, 1, ws, L, st)) != cudaSuccess) return e;
    if ((e = tc_rows_bwd(s, 2, x, ws + L.wimg, ws + L.zimg, ws + L.px, f, dfx, deltaS, wds,
                         reinterpret_cast<const float*>(ws + L.ds), k > 0 ? 1 : 0, status, st)) != cudaSuccess)
      return e;
  }
  // 5. delta's point rows
  k_prep_dpx<<<(unsigned)((npx + 255) / 256), 256, 0, st>>>(deltaS, deltaD, wds, reinterpret_cast<uint4*>(ws + L.dpx),
                                                              s.BH(), s.N, Np);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  // 6. dW, dbias, dtau of da_D + da_S
  {
    const size_t sm = smem_bwd_slot(3);
    const auto kernel = k_bwd_slot_tc<3, true>;
    if ((e = set_smem(kernel, sm)) != cudaSuccess) return e;
    for (int k = 0; k < sr.n; k++) {
      const int g0 = k * sr.size, G = range_g(k);
      Src a;
      if ((e = gather(g0, G, ranged, true, true, true, &a)) != cudaSuccess) return e;
      if ((e = prep_w(s, G, a.W, a.b, tau, ws + L.wimg, status, st)) != cudaSuccess) return e;
      const int64_t BHG = s.BH() * s.G;
      k_prep_t<<<(unsigned)((BHG + 127) / 128), 128, 0, st>>>(a.z, kD, 0, ws + L.timg, nullptr, s.BH(), G, s.G);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
      k_prep_t<<<(unsigned)((BHG + 127) / 128), 128, 0, st>>>(a.u, kD + 1, 1, ws + C.timg2, nullptr, s.BH(), G, s.G);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
      kernel<<<dim3((unsigned)R, (unsigned)P, (unsigned)s.BH()), kThreads, sm, st>>>(
          xmap, vmap, pmap, dmap, fmap, ws + L.wimg, ws + L.timg, ws + C.timg2, reinterpret_cast<float*>(ws + L.part),
          reinterpret_cast<float*>(ws + L.dtp), s.N, Np, s.H, s.G, P, status);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
      const int acc = accumulate || k > 0;
      Shape sk = s0;
      sk.G = G;
      float *dWk = dW, *dbk = db;
      if (ranged) {
        dWk = reinterpret_cast<float*>(ws + L.dwc);
        dbk = reinterpret_cast<float*>(ws + L.dbc);
        if (accumulate) {
          if ((e = copy_rows(dWk, G, dW + g0, s0.G, G, (int64_t)s.H * kD, st)) != cudaSuccess) return e;
          if ((e = copy_rows(dbk, G, db + g0, s0.G, G, s.H, st)) != cudaSuccess) return e;
        } else if (acc) {
          if ((e = cudaMemsetAsync(dWk, 0, (size_t)s.H * kD * G * sizeof(float), st)) != cudaSuccess) return e;
          if ((e = cudaMemsetAsync(dbk, 0, (size_t)s.H * G * sizeof(float), st)) != cudaSuccess) return e;
        }
      }
      if ((e = simt_reduce_bwd(sk, P, reinterpret_cast<const float*>(ws + L.part), s.G, kD + 2, 0, tau, nullptr, dWk,
                               dbk, dtau, reinterpret_cast<const float*>(ws + L.dtp), (int64_t)P * R, acc, st)) !=
          cudaSuccess)
        return e;
      if (ranged) {
        if ((e = copy_rows(dW + g0, s0.G, dWk, G, G, (int64_t)s.H * kD, st)) != cudaSuccess) return e;
        if ((e = copy_rows(db + g0, s0.G, dbk, G, G, s.H, st)) != cudaSuccess) return e;
      }
    }
  }
  // 7. dx from da_D + da_S
  const SlotRanges cr = comb_ranges(s0);
  Shape sc = s;
  sc.G = cr.size;
  const bool hilo = smem_bwd_dx(sc.G, true, true) <= kMaxSmem;
  const size_t sm = smem_bwd_dx(sc.G, hilo, true);
  if (sm > kMaxSmem) return cudaErrorInvalidValue;
  const auto kernel = k_bwd_dx_tc<true, true>;
  if ((e = set_smem(kernel, sm)) != cudaSuccess) return e;
  const int Pd = point_splits(sc, (int)sc.BH());
  for (int k = 0; k < cr.n; k++) {
    const int g0 = k * cr.size, G = k < cr.n - 1 ? cr.size : s0.G - (cr.n - 1) * cr.size;
    Src a;
    if ((e = gather(g0, G, cr.n > 1, true, true, true, &a)) != cudaSuccess) return e;
    if ((e = prep_w(sc, G, a.W, a.b, tau, ws + L.wimg, status, st)) != cudaSuccess) return e;
    const int64_t nwt = (int64_t)sc.H * kD * sc.G, BHG = sc.BH() * sc.G;
    k_prep_wt<<<(unsigned)((nwt + 255) / 256), 256, 0, st>>>(a.W, tau, ws + L.wtimg, sc.H, G, sc.G, status);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    k_prep_t<<<(unsigned)((BHG + 127) / 128), 128, 0, st>>>(a.z, kD, 0, ws + L.timg, nullptr, sc.BH(), G, sc.G);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    k_prep_t<<<(unsigned)((BHG + 127) / 128), 128, 0, st>>>(a.u, kD + 1, 1, ws + C.timg2, nullptr, sc.BH(), G, sc.G);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    kernel<<<dim3((unsigned)Pd, (unsigned)sc.BH()), kThreads, sm, st>>>(
        xmap, vmap, pmap, dmap, fmap, ws + L.wimg, ws + L.timg, ws + C.timg2, ws + L.wtimg,
        static_cast<__nv_bfloat16*>(dx), sc.N, Np, sc.H, sc.G, Pd, hilo ? 1 : 0, (accumulate || k > 0) ? 1 : 0,
        status);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace

// A single point (N = 1) takes the fp32 SIMT backward: every token is then that
// point's fx times S/(S + eps), so the slice's gradients are O(eps) and come from
// cancelling terms of size |dz||fx|/(S + eps) that split bf16 products resolve only
// to ~2^-17 of that size.
bool tc_backward_supported(const Shape& s0) {
  if (s0.dtype != FS_BF16 || s0.d != kD || s0.N < 2 || s0.G > 4096) return false;
  const Shape s = pass_shape(s0);
  return tc_forward_supported(s) && smem_bwd_dx(s.G, false) <= kMaxSmem &&
         tc_rows_smem(s, 2, false, false) <= kMaxSmem;
}

size_t tc_backward_bytes(const Shape& s, int mode) {
  return tc_backward_supported(s) ? bwd_layout(s, mode).total : 0;
}

int tc_backward_launch_count(const Shape& s, int mode) {
  const SlotRanges sr = slot_ranges(s.G);
  // per range: prep_t, prep_z2, prep_w, rows; then prep_px, prep_dpx; per range: the
  // images again (or prep_wt alone with one range), slot, dx and the reductions of
  // the parameters and dtau (and of dz' in mode 1); mode 2 also the dU/dS prologue.
  const int images = sr.n > 1 ? 4 : 1;
  const int reduce = mode == 1 ? 3 : 2;
  return 4 * sr.n + 2 + sr.n * (images + 2 + reduce) + (mode == 2 ? 1 : 0);
}

cudaError_t tc_deslice_bwd(const Shape& s0, const void* x, const float* W, const float* bias, const float* tau,
                           const float* zp, const float* lse, const void* dout, float* dzp, void* dx, float* dW,
                           float* db, float* dtau, int accumulate, void* ws_tc, uint32_t* status, cudaStream_t st) {
  return run_backward(s0, 1, x, dout, W, bias, tau, zp, kD, lse, nullptr, dx, dzp, dW, db, dtau, accumulate,
                      static_cast<uint8_t*>(ws_tc), status, st);
}

size_t tc_coupling_bwd_bytes(const Shape& s) { return tc_backward_supported(s) ? coup_layout(s).total : 0; }

int tc_coupling_bwd_launch_count(const Shape& s) {
  const SlotRanges sr = slot_ranges(s.G), cr = comb_ranges(s);
  const int n = sr.n, r = n > 1 ? 1 : 0;
  // lse rows; per range: the deslice rows pass with its images (4), the d z' slot
  // pass with its reduction (2, and the W image again with several ranges); the mix
  // backward (2) and the dU | dS prologue; per range the slice rows pass with its
  // images (4); delta's rows; per range the combined slot pass with its images and
  // reductions (6); per point-pass range its images and the pass (5)
  const int dz = tc_forward_supported(split_shape(s)) ? 4 /*prep_w, prep_px, slice, reduce*/ : n * (2 + r);
  return 1 + 4 * n + dz + 3 + 4 * n + 1 + 6 * n + 5 * cr.n;
}

cudaError_t tc_coupling_bwd(const Shape& s0, const void* x, const void* f, const void* dout, const float* W,
                            const float* bias, const float* tau, const float* M, const float* z, const float* wsum,
                            const float* zp, const float* lse, float* dzp, float* dz, float* dM, void* dx, void* dfx,
                            float* dW, float* db, float* dtau, int accumulate, float* dUS, void* ws_tc,
                            uint32_t* status, cudaStream_t st) {
  return run_coupling_bwd(s0, x, f, dout, W, bias, tau, M, z, wsum, zp, lse, dzp, dz, dM, dx, dfx, dW, db, dtau,
                          accumulate, dUS, static_cast<uint8_t*>(ws_tc), status, st);
}

cudaError_t tc_slice_bwd(const Shape& s0, const void* x, const void* f, const float* W, const float* bias,
                         const float* tau, const float* z, const float* wsum, const float* lse, const float* dz,
                         void* dx, void* dfx, float* dW, float* db, float* dtau, int accumulate, float* dUS,
                         void* ws_tc, uint32_t* status, cudaStream_t st) {
  cudaError_t e = simt_slice_bwd_prep(s0, z, wsum, dz, dUS, st);
  if (e != cudaSuccess) return e;
  return run_backward(s0, 2, x, f, W, bias, tau, dUS, kD + 1, lse, dfx, dx, nullptr, dW, db, dtau, accumulate,
                      static_cast<uint8_t*>(ws_tc), status, st);
}

}  // namespace fs
