// Tensor-core forward path on sm_103a (tcgen05 + TMEM + TMA), and the rows pass
// of the backward (the deslice kernel in modes 1 and 2, see k_deslice).
//
// Inputs: bf16 point tensors as they are; fp32 point tensors split beforehand
// into bf16 hi and residual tensors (k_split_bf16), with the residual products
// added in the X3 instantiations.  G is padded to whole 128-slot blocks whose
// padding slots carry weight 0.
//
// The three streaming passes of the paper's G-blocked family (Appendix G.1):
//   k_stats   : per point and head, lse_n = log sum_g exp(a_ng)        (point-owned)
//   k_slice   : per slot, U_g = sum_n w_ng f_n and S_g = sum_n w_ng     (slot-owned,
//               split over points; the partials are summed in a fixed order after)
//   k_deslice : per point, out_n = sum_g w_ng z'_g                      (point-owned)
// w is recomputed tile by tile in every pass and never leaves the SM.
//
// Logits.  A 128-point x 128-slot block of base-2 logits a2 = a * log2(e) is one
// tcgen05.mma chain with K = 48:
//   point side [ x (32 bf16) | 1, 1, -lse2 (three bf16 parts), 0 ... ]  (stats: 1, 1, 0 ...)
//   slot side  [ W*log2e/tau (32) | b'_hi, b'_lo, 1, 1, 1, 0 ... ]  (b' = bias*log2e/tau
//                                                                 in two bf16 halves)
// The point-major passes (stats, deslice) put points on the MMA's M (TMEM lane
// = point); the slice swaps the operands, so its TMEM lane is a slot and its
// column a point.  In the slice and the deslice the point side's extra block is
// [1, 1, -lse2 in three parts, 0 ...], so the accumulator holds a2 - lse2, the
// log2 of the slice weight itself.  The stats pass writes these 16-byte rows per
// point to memory and the later passes load them by TMA with each tile: no
// thread writes a tensor-core operand per tile (that would cost a generic ->
// async proxy fence per tile).
//
// Products.  The bf16 weights are written back into the S buffer they came
// from and feed the second MMA as its TMEM A operand: P x Z' in the deslice
// (M = points, K = slots, N = 32 channels), E x [F | 1] in the slice (M =
// slots, K = points, N = 48: 32 channels and a ones column for the weight sums).
//
// Issue.  Each MMA-issuing role is a whole converged warp in which one elected
// lane issues (a lone lane in a divergent branch issues several times slower).
// Warp 1 issues the logits (stats: warps 1 and 2); warps 2 and 3 issue the
// products into accumulators of their own, which are summed in a fixed order,
// so the result is deterministic.
//
// CTA (384 threads): warp 0 TMA producer, warps 1..3 MMA issuers, warps 4..11
// two softmax warpgroups that take alternate blocks (so they run out of phase);
// a thread owns one TMEM lane (tcgen05.ld/st 32x32b).  Every wait is bounded
// (2 s): a wait that gives up writes FS_ERR_TIMEOUT to the status word, the CTA
// drains its copies and MMAs, frees TMEM and exits.
//
// Shared-memory operand layouts (all bases 1024-byte aligned):
//   x tile          K-major, 64 B rows, 64B swizzle (TMA)        128 points x 32
//   constant extra  K-major, 32 B rows, 32B swizzle              128 rows x 16
//   point extra     K-major, no swizzle: core matrices of 8 rows x 16 B, the
//                   k = 0..7 half from memory (TMA), the k = 8..15 half zero
//   W image         K-major, 64 B rows, 64B swizzle, then its 32 B extra rows
//   Z' image        K-major rows = channels, 128 B rows, 128B swizzle
//   [F | 1]         MN-major, three 16-channel blocks, 32B swizzle (TMA)
#include "fs_tc_common.cuh"

namespace fs {
namespace {

using namespace tc;

// =========================================================================================
// Deslice: out_n = sum_g w_ng z'_g.
// smem: [W img G*96][Z' img G*64][stages: x | point extra (TMA half, zero half)][barriers]
// TMEM: S buffers [0, 384); P x Z' accumulators O_0 [384, 448), O_1 [448, 512),
// each double-buffered by tile parity.  Block q (tile q / nb, slot block q % nb)
// uses S buffer q % 3 and softmax warpgroup q % 2, which writes the bf16 weights
// of its 128 slots, packed in pairs, into columns [0, 64) of the same buffer;
// warp 2 + j turns slots [64 j, 64 j + 64) of every block into products
// (K-steps [4 j, 4 j + 4)) accumulated in O_j.
//
// The same pass serves the backward (Sec. 3.3): with R_n = sum_g w_ng t_g,
//   MODE 1 (deslice backward, t = z', v = dO): delta_n = dO_n . R_n (fp32);
//   MODE 2 (slice backward, t = dU, v = fx): dfx_n = R_n (bf16, into out) and
//     delta_n = fx_n . R_n + sum_g w_ng dS_g.  The second sum is formed by the
//     softmax warpgroups from the fp32 weights; each warpgroup adds its own
//     partial per point to wds[wg][bh][n] (cleared beforehand) and the consumer adds them.
// accumulate (MODES 1, 2, and MODE 0 with X3): the pass covers a later range of the
// slots, whose contributions to delta and dfx (to the fp32 out) are added to those of
// the earlier ranges.
// PS (split products): the weights and t as bf16 hi + lo halves, P t = Phi thi +
// Plo thi + Phi tlo; the image then holds t's residual half after its bf16 half.
// The split weights of slot half j (slots [64 j, 64 j + 64) of the block) go to
// columns [64 j, 64 j + 64) of the S buffer: the hi pairs, then the lo pairs.
// =========================================================================================
constexpr uint32_t kDStage = kXBytes + 2 * kPxBytes;  // x tile, point extra (both halves)

// X3 (fp32 inputs, MODE 0 with PS): each stage also holds x's residual tile
// (xrmap), the logits add x_r W'_hi, and out is fp32.
// The forward with single-level products (MODE 0, !PS) runs four softmax
// warpgroups (640 threads): warpgroups 2p and 2p + 1 take the blocks q with
// q % 2 == p, each one 64-slot half of every row, and half j's packed weights go to
// columns [64 j, 64 j + 32) of the S buffer, where product issuer j reads them as
// soon as half j is ready.  The other modes keep two warpgroups on whole rows.
template <int MODE, bool PS>
constexpr bool desl_wg4() { return MODE == 0 && !PS; }
constexpr int kDesl4Threads = 640;
template <int MODE, bool PS, bool X3 = false>
__global__ void __launch_bounds__(desl_wg4<MODE, PS>() ? kDesl4Threads : kThreads, 1)
    k_deslice(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ CUtensorMap pmap,
              const __grid_constant__ CUtensorMap xrmap,
              const uint8_t* __restrict__ wimg, const uint8_t* __restrict__ zimg, __nv_bfloat16* __restrict__ out,
              const __nv_bfloat16* __restrict__ v, float* __restrict__ delta, float* __restrict__ wds,
              const float* __restrict__ dS, int64_t N, int64_t Np, int H, int G, int splits, int hilo,
              uint32_t zstride, int accumulate, uint32_t* status) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  // hilo: the residual half of W' fits in shared memory too (K = 80 logits, as in
  // the statistics pass); else bf16 W' only (K = 48).
  const uint32_t wbytes = (uint32_t)G * (hilo ? kWRow : 96), zbytes = (uint32_t)G * (PS ? 128 : 64);
  uint8_t* s_w = smem;
  uint8_t* s_z = s_w + wbytes;
  float* s_ds = reinterpret_cast<float*>(s_z + zbytes);  // MODE 2: dS of the G slots
  // (the stages stay 1024-byte aligned for their swizzled tiles)
  uint8_t* s_x = s_z + zbytes + (MODE == 2 ? (((uint32_t)G * 4 + 1023u) & ~1023u) : 0u);  // stage s at s_x + s * kDSt
  constexpr uint32_t kDSt = kDStage + (X3 ? kXBytes : 0u);  // stage: x | px (2 halves) [| x residual]
  uint64_t* bars = reinterpret_cast<uint64_t*>(s_x + kStages * kDSt);
  uint64_t* wz_full = bars;
  uint64_t* x_full = bars + 1;
  uint64_t* x_empty = x_full + kStages;
  uint64_t* s_full = x_empty + kStages;
  constexpr bool kWG4 = desl_wg4<MODE, PS>();
  uint64_t* p_ready = s_full + kSBuf;  // [kSBuf][2 halves] with four warpgroups, else [kSBuf]
  uint64_t* pv_done = p_ready + 2 * kSBuf;
  uint64_t* o_full = pv_done + kSBuf;
  uint64_t* o_free = o_full + 2;
  uint64_t* drain = o_free + 2;  // one per issuing warp
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 3);
  Abort* ab = reinterpret_cast<Abort*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const Work wk = work_of(N, splits, blockIdx.x, blockIdx.y);
  const int64_t b = wk.bh / H;
  const int h = (int)(wk.bh % H);
  const int nch = G / kGC;
  constexpr uint32_t kO = kSBuf * kGC;  // TMEM column base of the O accumulators
  const int total = wk.ntiles * nch;

  if (threadIdx.x == 0) {
    mbar_init(wz_full, 1);
    for (int s = 0; s < kStages; s++) {
      mbar_init(&x_full[s], 1);
      mbar_init(&x_empty[s], 1);
    }
    for (int i = 0; i < kSBuf; i++) {
      mbar_init(&s_full[i], 1);
      mbar_init(&p_ready[2 * i], 4);  // the four warps of the warpgroup that owns the block (half)
      mbar_init(&p_ready[2 * i + 1], 4);
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
  for (int s = 0; s < kStages; s++) zero_smem(s_x + s * kDSt + kXBytes + kPxBytes, kPxBytes);
  if (MODE == 2)
    for (int g = threadIdx.x; g < G; g += kThreads) s_ds[g] = dS[wk.bh * G + g];
  fence_proxy_async_smem();
  if (warp == 1) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ------------------------------ producer ------------------------------
    if (lane == 0 && wk.ntiles > 0) {
      prefetch_tmap(&xmap);
      prefetch_tmap(&pmap);
      if (X3) prefetch_tmap(&xrmap);
      mbar_expect_tx(wz_full, wbytes + zbytes);
      load_images(s_w, wimg + (size_t)h * G * kWRow, wbytes, wz_full);
      load_images(s_z, zimg + (size_t)wk.bh * zstride, zbytes, wz_full);
      int i = 0;
      for (; i < wk.ntiles; i++) {
        const int s = i % kStages;
        if (i >= kStages && !mbar_wait(&x_empty[s], (uint32_t)(((i / kStages) - 1) & 1), ab, status)) break;
        const int n0 = (int)((wk.tile0 + i) * kTile);
        mbar_expect_tx(&x_full[s], kXBytes + kPxBytes + (X3 ? kXBytes : 0u));
        tma_load_3d(s_x + s * kDSt, &xmap, h * kD, n0, (int)b, &x_full[s]);
        tma_load_2d(s_x + s * kDSt + kXBytes, &pmap, 0, (int)(wk.bh * Np + n0), &x_full[s]);
        if (X3) tma_load_3d(s_x + s * kDSt + kDStage, &xrmap, h * kD, n0, (int)b, &x_full[s]);
      }
      // Drain: the newest load of each stage has landed before the CTA exits.
      for (int j = (i > kStages ? i - kStages : 0); j < i; j++)
        mbar_wait(&x_full[j % kStages], (uint32_t)((j / kStages) & 1), ab, nullptr, kWaitNs);
      mbar_wait(wz_full, 0, ab, nullptr, kWaitNs);
    }
  } else if (warp == 1) {
    // ------------------------------ logits issuer ------------------------------
    // Block q uses S buffer q % 3; it is rewritten only after the products of
    // block q - 3 (issued by the other warps) have completed.
    if (wk.ntiles > 0) {
      const uint32_t sw = smem_u32(s_w), swe = sw + (uint32_t)G * 64;
      bool ok = mbar_wait_w(wz_full, 0, ab, status);
      BlockPos pos(0, nch);
      for (int q = 0; ok && q < total; q++, pos.step(1, nch)) {
        const int i = pos.i, c = pos.c;
        const int s = i % kStages;
        const int bb = q % kSBuf;
        if (c == 0 && !(ok = mbar_wait_w(&x_full[s], (uint32_t)((i / kStages) & 1), ab, status))) break;
        if (q >= kSBuf && !(ok = mbar_wait_w(&pv_done[bb], (uint32_t)(((q / kSBuf) - 1) & 1), ab, status))) break;
        tc_fence_after();
        const uint32_t xs = smem_u32(s_x + s * kDSt);
        issue_logits(tmem + (uint32_t)bb * kGC, xs, point_extra_desc(xs + kXBytes), sw, swe,
                     hilo ? sw + (uint32_t)G * 96 : 0u, c, true, X3 ? xs + kDStage : 0u);
        mma_commit_w(&s_full[bb]);
        if (c == nch - 1) mma_commit_w(&x_empty[s]);
      }
      mma_commit_w(&drain[0]);
      mbar_wait_w(&drain[0], 0, ab, nullptr, kWaitNs);
    }
  } else if (warp == 2 || warp == 3) {
    // ------------------------------ P x Z' issuers ------------------------------
    const int j = warp - 2;  // K-steps [4j, 4j + 4) of every block, accumulator O_j
    if (wk.ntiles > 0) {
      constexpr uint32_t idesc_pv = idesc_bf16(128, kD, false, false);
      const uint32_t sz = smem_u32(s_z);
      bool ok = mbar_wait_w(wz_full, 0, ab, status);
      BlockPos pos(0, nch);
      for (int q = 0; ok && q < total; q++, pos.step(1, nch)) {
        const int i = pos.i, c = pos.c;
        const int ob = i & 1;
        const int bb = q % kSBuf;
        if (c == 0 && i >= 2 && !(ok = mbar_wait_w(&o_free[ob], (uint32_t)(((i >> 1) - 1) & 1), ab, status))) break;
        if (!(ok = mbar_wait_w(&p_ready[kWG4 ? 2 * bb + j : 2 * bb], (uint32_t)((q / kSBuf) & 1), ab, status))) break;
        tc_fence_after();
        // weights of slots 64j.. (packed pairs; PS: hi pairs, then lo pairs 32 on)
        const uint32_t tP = tmem + (uint32_t)bb * kGC + (uint32_t)j * ((kWG4 || PS) ? 64 : 32);
        const uint32_t tO = tmem + kO + (uint32_t)(j * 2 + ob) * kD;
#pragma unroll
        for (int kk = 0; kk < 4; kk++) {
          const int g0 = c * kGC + (4 * j + kk) * 16;
          const uint32_t zaddr = sz + (uint32_t)((g0 >> 6) * 4096 + (g0 & 63) * 2);
          mma_ts_w(tO, tP + (uint32_t)kk * 8, sdesc(zaddr, 16, 1024, kSw128), idesc_pv, (c > 0 || kk > 0) ? 1u : 0u);
          if (PS) {
            mma_ts_w(tO, tP + 32 + (uint32_t)kk * 8, sdesc(zaddr, 16, 1024, kSw128), idesc_pv, 1u);
            mma_ts_w(tO, tP + (uint32_t)kk * 8, sdesc(zaddr + (uint32_t)G * 64, 16, 1024, kSw128), idesc_pv, 1u);
          }
        }
        mma_commit_w(&pv_done[bb]);
        if (c == nch - 1) mma_commit_w(&o_full[ob]);
      }
      mma_commit_w(&drain[1 + j]);
      mbar_wait_w(&drain[1 + j], 0, ab, nullptr, kWaitNs);
    }
  } else if (warp >= kSoftmaxWarp0) {
    // ------------------------------ softmax warpgroups ------------------------------
    const int wg4 = (warp - kSoftmaxWarp0) >> 2;
    const int wg = kWG4 ? wg4 >> 1 : wg4;  // the block parity this warpgroup takes
    const int hf = kWG4 ? wg4 & 1 : 0;     // four warpgroups: the half of each row
    const int wq = warp & 3;  // TMEM sub-partition of this warp
    const int r = wq * 32 + lane;
    const uint32_t lane_addr = (uint32_t)(wq * 32) << 16;
    bool ok = true;
    // Output of tile t: O_0 + O_1 (fixed order) -> bf16 -> global, 64 B per point.
    auto epilogue = [&](int t) -> bool {
      const int ob = (int)(t & 1);
      if (!mbar_wait(&o_full[ob], (uint32_t)((t >> 1) & 1), ab, status)) return false;
      tc_fence_after();
      float R[kD];  // O_0 + O_1, in that order
      {
        uint32_t o0[32], o1[32];
        tmem_ld32(tmem + lane_addr + kO + (uint32_t)ob * kD, o0);
        tmem_ld32(tmem + lane_addr + kO + (uint32_t)(2 + ob) * kD, o1);
        tmem_wait_ld2(o0, o1);
#pragma unroll
        for (int k = 0; k < kD; k++) R[k] = __uint_as_float(o0[k]) + __uint_as_float(o1[k]);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&o_free[ob]);
      const int64_t n = (wk.tile0 + t) * kTile + r;
      if (n < N) {
        const int64_t row = ((b * N + n) * H + h) * kD;
        if (X3) {
          // accumulate: a later slot range, added to the earlier ranges' output
          float4* dst = reinterpret_cast<float4*>(reinterpret_cast<float*>(out) + row);
#pragma unroll
          for (int k = 0; k < 8; k++) {
            const float4 p = accumulate ? dst[k] : make_float4(0.f, 0.f, 0.f, 0.f);
            dst[k] = make_float4(p.x + R[4 * k], p.y + R[4 * k + 1], p.z + R[4 * k + 2], p.w + R[4 * k + 3]);
          }
        } else if (MODE != 1) {
          uint4* dst = reinterpret_cast<uint4*>(out + row);
#pragma unroll
          for (int k = 0; k < 4; k++) {
            // MODE 2 over a later slot range: add the dfx of the earlier ranges
            uint4 p4 = make_uint4(0u, 0u, 0u, 0u);
            if (MODE == 2 && accumulate) p4 = dst[k];
            const uint32_t pw[4] = {p4.x, p4.y, p4.z, p4.w};
            uint32_t w[4];
#pragma unroll
            for (int e = 0; e < 4; e++)
              w[e] = pack_bf16(R[8 * k + 2 * e] + __uint_as_float(pw[e] << 16),
                               R[8 * k + 2 * e + 1] + __uint_as_float(pw[e] & 0xFFFF0000u));
            dst[k] = make_uint4(w[0], w[1], w[2], w[3]);
          }
        }
        if (MODE != 0) {
          // delta_n = v_n . R_n from the fp32 accumulators.
          const uint4* src = reinterpret_cast<const uint4*>(v + row);
          float acc = 0.f;
#pragma unroll
          for (int k = 0; k < 4; k++) {
            const uint4 q4 = src[k];
            const uint32_t w[4] = {q4.x, q4.y, q4.z, q4.w};
#pragma unroll
            for (int e = 0; e < 4; e++) {
              const int c0 = 8 * k + 2 * e;
              acc = fmaf(__uint_as_float(w[e] << 16), R[c0], acc);
              acc = fmaf(__uint_as_float(w[e] & 0xFFFF0000u), R[c0 + 1], acc);
            }
          }
          delta[wk.bh * N + n] = accumulate ? delta[wk.bh * N + n] + acc : acc;
        }
      }
      return true;
    };
    // MODE 2: this warpgroup's sum_g w dS_g for point r of its current tile.
    float wds_acc = 0.f;
    int wds_tile = -1;
    auto flush_wds = [&]() {
      if (MODE == 2 && wds_tile >= 0) {
        const int64_t n = (wk.tile0 + wds_tile) * kTile + r;
        if (n < N) wds[((int64_t)wg * gridDim.y + wk.bh) * N + n] += wds_acc;
      }
      wds_acc = 0.f;
    };
    // Warpgroup wg takes the whole blocks q with q % 2 == wg, so the two warpgroups
    // run half a block out of phase: one exponentiates while the other waits.
    BlockPos pos(wg, nch);
    for (int q = wg; ok && q < total; q += 2, pos.step(2, nch)) {
      const int i = pos.i, c = pos.c;
      const int bb = q % kSBuf;
      if (!(ok = mbar_wait(&s_full[bb], (uint32_t)((q / kSBuf) & 1), ab, status))) break;
      tc_fence_after();
      if (MODE == 2) {
        if (i != wds_tile) {
          flush_wds();
          wds_tile = i;
        }
        if (PS) {
          weights_hilo_half_ds(tmem + lane_addr + (uint32_t)bb * kGC, s_ds + c * kGC, wds_acc);
          weights_hilo_half_ds(tmem + lane_addr + (uint32_t)bb * kGC + 64, s_ds + c * kGC + 64, wds_acc);
        } else
          weights_in_halves_ds(tmem + lane_addr + (uint32_t)bb * kGC, s_ds + c * kGC, wds_acc);
      } else if (PS) {
        weights_hilo_half(tmem + lane_addr + (uint32_t)bb * kGC);
        weights_hilo_half(tmem + lane_addr + (uint32_t)bb * kGC + 64);
      } else if (kWG4) {
        weights_half(tmem + lane_addr + (uint32_t)bb * kGC + (uint32_t)hf * 64);
      } else {
        weights_in_halves(tmem + lane_addr + (uint32_t)bb * kGC);
      }
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_ready[2 * bb + hf]);
      // The output of the previous tile is drained by the warpgroup (half 0 of the
      // pair) that took the first block of this tile, when the last products of that
      // tile have long finished.
      if (c == 0 && i > 0 && hf == 0 && !(ok = epilogue(i - 1))) break;
    }
    if (ok && total > 0 && total % 2 == wg && hf == 0) epilogue(wk.ntiles - 1);
    if (ok) flush_wds();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

// =========================================================================================
// Statistics: lse_n = log sum_g exp(a_ng) (natural log) to lse[bh*N + n], and
// the point-extra row [1, 1, -lse2 in three bf16 parts, 0 x 3] (lse2 = lse*log2(e)) to
// px[bh*Np + n] (Np = N rounded up to a whole tile; padded points get -1e30 so
// that their weights vanish).
// Two logits issuers and four softmax warpgroups (640 threads): block q (tile
// q / nb, slot block q % nb) goes through S buffer p = q % 2, issuer 1 + p and
// warpgroups 2p and 2p + 1, each of which takes one half (64 slots) of every row,
// so that each SM sub-partition holds four softmax warps whose exponentials and
// reductions interleave.  Each warpgroup keeps a running (max, sum) over the slots
// it took and hands it over through shared memory after its last block of the tile.
// With two or more blocks per tile all four warpgroups take blocks of every tile and
// warp 3 combines their shares and writes lse and the px rows, so no softmax warp
// waits for the others.  With one block per tile (G <= 128) the pair that takes it
// combines in place: half 1 hands its share to half 0, which writes (at two tiles or
// so per CTA an extra hop to warp 3 would lengthen each CTA's tail).
// smem: [W img G*96][x stages][constant extra][ml exchange][barriers]
// TMEM: two S buffers [0, 256).
// =========================================================================================
// X3 (fp32 inputs): x arrives as bf16 hi and residual tiles (xmap, xrmap), one stage
// holding both, and the logits add x_r W'_hi.
constexpr int kStatsThreads = 640;
template <bool split, bool X3>
__global__ void __launch_bounds__(kStatsThreads, 1)
    k_stats(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ CUtensorMap xrmap,
            const uint8_t* __restrict__ wimg, float* __restrict__ lse, uint4* __restrict__ px, int64_t N,
            int64_t Np, int H, int G, int splits, uint32_t* status) {
  constexpr uint32_t kXSt = X3 ? 2 * kXBytes : kXBytes;  // x stage
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  // split (FS_DOT_BF16X2): the residual half of W' too (K = 80 logits).
  const uint32_t wbytes = (uint32_t)G * (split ? kWRow : 96);
  uint8_t* s_w = smem;
  uint8_t* s_x = s_w + wbytes;
  uint8_t* s_ex = s_x + kStages * kXSt;
  float2* s_ml = reinterpret_cast<float2*>(s_ex + kExBytes);  // [2 tile parities][4 warpgroups][128 rows]
  uint64_t* bars = reinterpret_cast<uint64_t*>(s_ml + 8 * kTile);
  uint64_t* w_full = bars;
  uint64_t* x_full = bars + 1;
  uint64_t* x_empty = x_full + kStages;
  uint64_t* s_full = x_empty + kStages;
  uint64_t* s_free = s_full + 2;
  uint64_t* ml_full = s_free + 2;   // the warpgroups' shares of a tile written (per tile parity)
  uint64_t* ml_empty = ml_full + 2; // warp 3 has read them
  uint64_t* drain = ml_empty + 2;   // one per issuing warp
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 2);
  Abort* ab = reinterpret_cast<Abort*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const Work wk = work_of(N, splits, blockIdx.x, blockIdx.y);
  const int64_t b = wk.bh / H;
  const int h = (int)(wk.bh % H);
  const int nch = G / kGC;

  if (threadIdx.x == 0) {
    mbar_init(w_full, 1);
    for (int s = 0; s < kStages; s++) {
      mbar_init(&x_full[s], 1);
      mbar_init(&x_empty[s], (uint32_t)(nch < 2 ? nch : 2));
    }
    for (int i = 0; i < 2; i++) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_free[i], 8);
      mbar_init(&ml_full[i], nch >= 2 ? 16 : 4);
      mbar_init(&ml_empty[i], nch >= 2 ? 1 : 4);
    }
    mbar_init(&drain[0], 1);
    mbar_init(&drain[1], 1);
    ab->flag = 0;
    fence_mbar_init();
  }
  write_const_extra(s_ex);
  fence_proxy_async_smem();
  if (warp == 1) tmem_alloc(tmem_slot, 256);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0 && wk.ntiles > 0) {
      prefetch_tmap(&xmap);
      if (X3) prefetch_tmap(&xrmap);
      mbar_expect_tx(w_full, wbytes);
      load_images(s_w, wimg + (size_t)h * G * kWRow, wbytes, w_full);
      int i = 0;
      for (; i < wk.ntiles; i++) {
        const int s = i % kStages;
        if (i >= kStages && !mbar_wait(&x_empty[s], (uint32_t)(((i / kStages) - 1) & 1), ab, status)) break;
        mbar_expect_tx(&x_full[s], kXSt);
        tma_load_3d(s_x + s * kXSt, &xmap, h * kD, (int)((wk.tile0 + i) * kTile), (int)b, &x_full[s]);
        if (X3) tma_load_3d(s_x + s * kXSt + kXBytes, &xrmap, h * kD, (int)((wk.tile0 + i) * kTile), (int)b, &x_full[s]);
      }
      for (int j = (i > kStages ? i - kStages : 0); j < i; j++)
        mbar_wait(&x_full[j % kStages], (uint32_t)((j / kStages) & 1), ab, nullptr, kWaitNs);
      mbar_wait(w_full, 0, ab, nullptr, kWaitNs);
    }
  } else if (warp == 1 || warp == 2) {
    // With two or more blocks per tile, issuer j takes the blocks q with q % 2 == j
    // (always S buffer j, so each buffer has one producer and one consumer and
    // both issuers touch every tile); with one block per tile issuer 0 takes all.
    const int j = warp - 1;
    const int nis = nch >= 2 ? 2 : 1;
    if (wk.ntiles > 0 && j < nis) {
      const uint32_t sw = smem_u32(s_w), swe = sw + (uint32_t)G * 64;
      bool ok = mbar_wait_w(w_full, 0, ab, status);
      const int total = wk.ntiles * nch;
      BlockPos pos(j, nch);
      for (int q = j; ok && q < total; q += nis, pos.step(nis, nch)) {
        const int i = pos.i, c = pos.c;
        const int s = i % kStages;
        const int bb = q & 1;
        if (c < nis && !(ok = mbar_wait_w(&x_full[s], (uint32_t)((i / kStages) & 1), ab, status))) break;
        if (q >= 2 && !(ok = mbar_wait_w(&s_free[bb], (uint32_t)(((q >> 1) - 1) & 1), ab, status))) break;
        tc_fence_after();
        const uint32_t xs = smem_u32(s_x + s * kXSt);
        issue_logits(tmem + (uint32_t)bb * kGC, xs, const_extra_desc(smem_u32(s_ex)), sw, swe,
                     split ? sw + (uint32_t)G * 96 : 0u, c, true, X3 ? xs + kXBytes : 0u);
        mma_commit_w(&s_full[bb]);
        if (c >= nch - nis) mma_commit_w(&x_empty[s]);
      }
      mma_commit_w(&drain[j]);
      mbar_wait_w(&drain[j], 0, ab, nullptr, kWaitNs);
    }
  } else if (warp == 3) {
    // ------------------------------ combiner ------------------------------
    // Tile i: the four warpgroups' shares -> lse and px rows (two or more blocks per
    // tile).  Lane l takes the points l, l + 32, l + 64, l + 96 of the tile.
    bool ok = nch >= 2;
    for (int i = 0; ok && i < wk.ntiles; i++) {
      const int pb = i & 1;
      if (!(ok = mbar_wait(&ml_full[pb], (uint32_t)((i >> 1) & 1), ab, status))) break;
      float2 sh[4][4];
#pragma unroll
      for (int k = 0; k < 4; k++)
#pragma unroll
        for (int w = 0; w < 4; w++) sh[k][w] = s_ml[(pb * 4 + w) * kTile + lane + 32 * k];
      __syncwarp();
      if (lane == 0) mbar_arrive(&ml_empty[pb]);
#pragma unroll
      for (int k = 0; k < 4; k++) {
        const float M = fmaxf(fmaxf(sh[k][0].x, sh[k][1].x), fmaxf(sh[k][2].x, sh[k][3].x));
        float L = 0.f;
#pragma unroll
        for (int w = 0; w < 4; w++) L += sh[k][w].y * ex2(sh[k][w].x - M);
        const int64_t n = (wk.tile0 + i) * kTile + lane + 32 * k;
        const float lse2 = M + log2f(L);
        if (n < Np) {
          px[wk.bh * Np + n] = extra_row3(n < N ? -lse2 : -1e30f);
          if (n < N) lse[wk.bh * N + n] = lse2 * kLn2;
        }
      }
    }
  } else if (warp >= kSoftmaxWarp0) {
    const int wg = (warp - kSoftmaxWarp0) >> 2;
    const int pr = wg >> 1, hf = wg & 1;  // S buffer (block parity) and the half of each row
    const int wq = warp & 3;
    const int r = wq * 32 + lane;
    const uint32_t lane_addr = (uint32_t)(wq * 32) << 16;
    const int total = wk.ntiles * nch;
    bool ok = true;
    float m = -INFINITY, l = 0.f;
    // The pair of warpgroups of S buffer pr takes the whole blocks q with q % 2 == pr,
    // warpgroup hf the slots [64 hf, 64 hf + 64) of each.  A pair's last block of a
    // tile is one of its last two (c >= nch - 2); after it the warpgroup hands its
    // (max, sum) over the slots it took to warp 3.
    BlockPos pos(pr, nch);
    for (int q = pr; ok && q < total; q += 2, pos.step(2, nch)) {
      const int i = pos.i, c = pos.c;
      if (!(ok = mbar_wait(&s_full[pr], (uint32_t)((q >> 1) & 1), ab, status))) break;
      tc_fence_after();
      const uint32_t tS = tmem + lane_addr + (uint32_t)pr * kGC + (uint32_t)hf * 64;
      uint32_t v[2][32];
      tmem_ld32(tS, v[0]);
      tmem_ld32(tS + 32, v[1]);
      tmem_wait_ld2(v[0], v[1]);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_free[pr]);
      float t[22];
#pragma unroll
      for (int k = 0; k < 21; k++)
        t[k] = max3(__uint_as_float(v[(3 * k) >> 5][(3 * k) & 31]), __uint_as_float(v[(3 * k + 1) >> 5][(3 * k + 1) & 31]),
                    __uint_as_float(v[(3 * k + 2) >> 5][(3 * k + 2) & 31]));
      t[21] = fmaxf(__uint_as_float(v[1][31]), m);
#pragma unroll
      for (int k = 0; k < 7; k++) t[k] = max3(t[3 * k], t[3 * k + 1], t[3 * k + 2]);
      const float mn = max3(max3(t[0], t[1], t[2]), max3(t[3], t[4], t[5]), fmaxf(t[6], t[21]));
      const uint32_t nmb = __float_as_uint(-mn);
      const uint64_t nm2 = pack2(nmb, nmb);
#pragma unroll
      for (int j = 0; j < 2; j++)
#pragma unroll
        for (int k = 0; k < 16; k++) {
          const uint64_t a = add2(pack2(v[j][2 * k], v[j][2 * k + 1]), nm2);
          v[j][2 * k] = __float_as_uint(ex2(lo_f(a)));
          v[j][2 * k + 1] = __float_as_uint(ex2(hi_f(a)));
        }
      uint64_t acc[16];
#pragma unroll
      for (int k = 0; k < 16; k++)
        acc[k] = add2(pack2(v[0][2 * k], v[0][2 * k + 1]), pack2(v[1][2 * k], v[1][2 * k + 1]));
#pragma unroll
      for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
        for (int k = 0; k < w; k++) acc[k] = add2(acc[k], acc[k + w]);
      const float sum = lo_f(acc[0]) + hi_f(acc[0]);
      l = l * ex2(m - mn) + sum;
      m = mn;
      const int pb = i & 1;
      if (nch == 1 && hf == 0) {
        // One block per tile: combine with half 1's share and write.
        if (!(ok = mbar_wait(&ml_full[pb], (uint32_t)((i >> 1) & 1), ab, status))) break;
        const float2 o = s_ml[(pb * 4 + wg + 1) * kTile + r];
        __syncwarp();
        if (lane == 0) mbar_arrive(&ml_empty[pb]);
        const float M = fmaxf(m, o.x);
        const float L = l * ex2(m - M) + o.y * ex2(o.x - M);
        const int64_t n = (wk.tile0 + i) * kTile + r;
        const float lse2 = M + log2f(L);
        if (n < Np) {
          px[wk.bh * Np + n] = extra_row3(n < N ? -lse2 : -1e30f);
          if (n < N) lse[wk.bh * N + n] = lse2 * kLn2;
        }
        m = -INFINITY;
        l = 0.f;
      } else if (c >= nch - 2) {
        // This warpgroup's last block of the tile: hand the share over (to warp 3, or
        // with one block per tile to half 0 of the pair).
        if (i >= 2 && !(ok = mbar_wait(&ml_empty[pb], (uint32_t)(((i >> 1) - 1) & 1), ab, status))) break;
        s_ml[(pb * 4 + wg) * kTile + r] = make_float2(m, l);
        __syncwarp();
        if (lane == 0) mbar_arrive(&ml_full[pb]);
        m = -INFINITY;
        l = 0.f;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 256);
}

// =========================================================================================
// Slice (slot-owned, split over points), slot-major: CTA (p, bh, j) owns the
// 128-slot block j of head h and point split p and computes for its slots
//   U_g = sum_n w_ng f_n,  S_g = sum_n w_ng,  w_ng = 2^(a2_ng - lse2_n).
// The logits are formed transposed (M = 128 slots, N = 128 points), so TMEM
// lane = slot and column = point; the point-extra rows of the tile arrive by
// TMA with it, so the accumulator holds log2 of the weights.  The bf16 weights
// written back in place serve directly as the TMEM A operand of
// U|S += E [F | 1] (K = points), so the weight tile never passes through
// shared memory.
// Writes part[p][bh][g][0..32] = (U_g, S_g).
// smem: [W img block 128*96][stages: x | F_lo F_hi ones | point extra (2 halves)][barriers]
// TMEM: S buffers [0, 384); U|S accumulators A_0 [384, 432), A_1 [432, 480).
// Warp 1 issues the logits of every tile; softmax warpgroup wg takes the whole
// tiles i with i % 2 == wg, and warp 2 + wg issues their products into its own
// accumulator A_wg (the two are summed in a fixed order).
// =========================================================================================
constexpr uint32_t kStageBytes = kXBytes + 3 * kFBlock + 2 * kPxBytes;  // x, [F | 1], point extra
constexpr uint32_t kWBlock = 128 * kWRow;                               // one 128-slot block of the W image

// Flushes.  The tensor cores' fp32 accumulation over a CTA's long point range (a
// thousand and more K steps into one accumulator) loses ~2^-25 of the running sum per
// step, always towards zero: at 27,600 points 4e-5 relative, and the temperature
// gradient magnifies errors of the token gradients many times over (its sum over
// (n, g) cancels to ~1e-5 of its terms' magnitude).  So each accumulator's chain is
// restarted every kSliceFlush of its issuer's tiles, after its warpgroup has added
// what it holds into fp32 registers (round to nearest).  Only with split products
// and fp32 inputs: with single bf16 products the weights' own rounding (~3e-3
// relative in the tokens) dwarfs the drift (~1e-4 at 55,000 points per CTA), and
// the waits on each flushed chain cost the plain slice 4%.
constexpr int kSliceFlush = 4;
template <bool kOn>
__device__ __forceinline__ bool slice_flush_at(int i) { return kOn && ((i >> 1) % kSliceFlush) == 0; }

// X3 (fp32 inputs): each stage also holds the residual tiles of x and fx (xrmap,
// frmap); the logits add x_r W'_hi and the products add P_hi F_r (N = 32: U only).
// Its stages are larger, so there are half as many.
template <bool split, bool X3>
__global__ void __launch_bounds__(kThreads, 1)
    k_slice(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ CUtensorMap fmap,
            const __grid_constant__ CUtensorMap pmap, const __grid_constant__ CUtensorMap xrmap,
            const __grid_constant__ CUtensorMap frmap, const uint8_t* __restrict__ wimg, float* __restrict__ part,
            int64_t N, int64_t Np, int H, int G, int splits, uint32_t* status) {
  constexpr int kNSt = X3 ? kSliceStages / 2 : kSliceStages;
  constexpr uint32_t kStB = kStageBytes + (X3 ? kXBytes + 2 * kFBlock : 0u);
  constexpr uint32_t kXROff = kStageBytes, kFROff = kStageBytes + kXBytes;
  // split (FS_DOT_BF16X2): logits with both halves of W' (K = 80), and the
  // weights as hi + lo bf16 halves in the products (twice the product MMAs).
  // Grid (slot block, point split, bh): the CTAs of all slot blocks of one point
  // range are adjacent in launch order, run together and share each x / F tile
  // through L2 instead of re-reading it from DRAM once per slot block.
  const int g_base = blockIdx.x * kGC;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* s_w = smem;
  uint8_t* s_st = s_w + kWBlock;
  uint64_t* bars = reinterpret_cast<uint64_t*>(s_st + kNSt * kStB);
  uint64_t* w_full = bars;
  uint64_t* x_full = bars + 1;
  uint64_t* st_empty = x_full + kNSt;
  uint64_t* s_full = st_empty + kNSt;
  uint64_t* p_ready = s_full + kSBuf;   // [issuer][S buffer]
  uint64_t* pv_done = p_ready + 2 * kSBuf;
  uint64_t* acc_full = pv_done + kSBuf;
  uint64_t* acc_done = acc_full + 1;  // [issuer]: products of each of its tiles complete
  uint64_t* wt_ready = acc_done + 2;  // single-level products: the W' image is in TMEM
  uint64_t* drain = wt_ready + 1;  // one per issuing warp
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 3);
  Abort* ab = reinterpret_cast<Abort*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const Work wk = work_of(N, splits, blockIdx.y, blockIdx.z);
  const int64_t b = wk.bh / H;
  const int h = (int)(wk.bh % H);
  constexpr uint32_t kA = kSBuf * kGC;  // TMEM column base of the accumulators
  constexpr uint32_t kFOff = kXBytes, kPOff = kXBytes + 3 * kFBlock;
  // With single-level products the slot block's W' image (W' and its extra block: 24
  // columns) fits in the 32 TMEM columns after the accumulators, and the logits read
  // only their point side from shared memory.
  constexpr bool kWT = !split && !X3;
  constexpr uint32_t kTW = kA + 96;

  if (threadIdx.x == 0) {
    mbar_init(w_full, 1);
    for (int s = 0; s < kNSt; s++) {
      mbar_init(&x_full[s], 1);
      mbar_init(&st_empty[s], 2);  // the logits issuer and the tile's product issuer
    }
    for (int i = 0; i < kSBuf; i++) {
      mbar_init(&s_full[i], 1);
      mbar_init(&p_ready[i], 4);  // the four warps of the warpgroup that took the tile
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
  for (int s = 0; s < kNSt; s++) zero_smem(s_st + s * kStB + kPOff + kPxBytes, kPxBytes);
  // Constant "ones" block of every stage: row n = [1, 0 x 15] (32B swizzle).
  for (int idx = threadIdx.x; idx < kNSt * kTile; idx += kThreads) {
    const int s = idx / kTile, r = idx % kTile;
    const uint32_t base = smem_u32(s_st + s * kStB + kFOff + 2 * kFBlock) +
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
      prefetch_tmap(&pmap);
      if (X3) {
        prefetch_tmap(&xrmap);
        prefetch_tmap(&frmap);
      }
      // The slot block's rows of the W image: 128 rows of W' (64 B) then 128 rows of
      // the extra block (32 B); the global image holds G rows of each.
      mbar_expect_tx(w_full, split ? kWBlock : kGC * 96);
      const uint8_t* src = wimg + (size_t)h * G * kWRow;
      load_images(s_w, src + (size_t)g_base * 64, kGC * 64, w_full);
      load_images(s_w + kGC * 64, src + (size_t)G * 64 + (size_t)g_base * 32, kGC * 32, w_full);
      if (split) load_images(s_w + kGC * 96, src + (size_t)G * 96 + (size_t)g_base * 64, kGC * 64, w_full);
      int i = 0;
      for (; i < wk.ntiles; i++) {
        const int s = i % kNSt;
        if (i >= kNSt &&
            !mbar_wait(&st_empty[s], (uint32_t)(((i / kNSt) - 1) & 1), ab, status))
          break;
        uint8_t* st = s_st + s * kStB;
        const int n0 = (int)((wk.tile0 + i) * kTile);
        mbar_expect_tx(&x_full[s], kXBytes + 2 * kFBlock + kPxBytes + (X3 ? kXBytes + 2 * kFBlock : 0u));
        tma_load_3d(st, &xmap, h * kD, n0, (int)b, &x_full[s]);
        tma_load_3d(st + kFOff, &fmap, h * kD, n0, (int)b, &x_full[s]);
        tma_load_3d(st + kFOff + kFBlock, &fmap, h * kD + 16, n0, (int)b, &x_full[s]);
        tma_load_2d(st + kPOff, &pmap, 0, (int)(wk.bh * Np + n0), &x_full[s]);
        if (X3) {
          tma_load_3d(st + kXROff, &xrmap, h * kD, n0, (int)b, &x_full[s]);
          tma_load_3d(st + kFROff, &frmap, h * kD, n0, (int)b, &x_full[s]);
          tma_load_3d(st + kFROff + kFBlock, &frmap, h * kD + 16, n0, (int)b, &x_full[s]);
        }
      }
      for (int j = (i > kNSt ? i - kNSt : 0); j < i; j++)
        mbar_wait(&x_full[j % kNSt], (uint32_t)((j / kNSt) & 1), ab, nullptr, kWaitNs);
      mbar_wait(w_full, 0, ab, nullptr, kWaitNs);
    }
  } else if (warp == 1) {
    // ------------------------------ logits issuer (transposed) ------------------------------
    {
      const uint32_t sw = smem_u32(s_w), swe = sw + kGC * 64;
      bool ok = mbar_wait_w(w_full, 0, ab, status);
      if (kWT && ok) {
        ok = mbar_wait_w(wt_ready, 0, ab, status);
        tc_fence_after();
      }
      for (int i = 0; ok && i < wk.ntiles; i++) {
        const int s = i % kNSt;
        const int bb = i % kSBuf;
        if (!(ok = mbar_wait_w(&x_full[s], (uint32_t)((i / kNSt) & 1), ab, status))) break;
        if (i >= kSBuf && !(ok = mbar_wait_w(&pv_done[bb], (uint32_t)(((i / kSBuf) - 1) & 1), ab, status))) break;
        tc_fence_after();
        const uint32_t xs = smem_u32(s_st + s * kStB);
        if (kWT) {
          constexpr uint32_t idesc = idesc_bf16(128, kGC, false, false);
          const uint32_t tD = tmem + (uint32_t)bb * kGC;
          mma_ts_w(tD, tmem + kTW, sdesc(xs, 16, 512, kSw64), idesc, 0u);
          mma_ts_w(tD, tmem + kTW + 8, sdesc(xs + 32, 16, 512, kSw64), idesc, 1u);
          mma_ts_w(tD, tmem + kTW + 16, point_extra_desc(xs + kPOff), idesc, 1u);
        } else {
          issue_logits(tmem + (uint32_t)bb * kGC, xs, point_extra_desc(xs + kPOff), sw, swe,
                       split ? sw + kGC * 96 : 0u, 0, false, X3 ? xs + kXROff : 0u);
        }
        mma_commit_w(&s_full[bb]);
        mma_commit_w(&st_empty[s]);
      }
      mma_commit_w(&drain[0]);
      mbar_wait_w(&drain[0], 0, ab, nullptr, kWaitNs);
    }
  } else if (warp == 2 || warp == 3) {
    // ------------------------------ product issuers ------------------------------
    const int j = warp - 2;  // tiles i with i % 2 == j, accumulator A_j
    {
      constexpr uint32_t idesc_sl = idesc_bf16(128, 48, false, true);
      bool ok = true;
      for (int i = j; ok && i < wk.ntiles; i += 2) {
        const int s = i % kNSt;
        const int bb = i % kSBuf;
        // This issuer's tiles on buffer bb are 2 kSBuf apart.
        if (!(ok = mbar_wait_w(&p_ready[j * kSBuf + bb], (uint32_t)((i / (2 * kSBuf)) & 1), ab, status))) break;
        tc_fence_after();
        const uint32_t tE = tmem + (uint32_t)bb * kGC;  // packed weights of the 128 points
        const uint32_t fs = smem_u32(s_st + s * kStB) + kFOff;
        const uint32_t tacc = tmem + kA + (uint32_t)j * 48;
        // A chain restarts at this issuer's first tile and at every flush tile (its
        // warpgroup has moved the earlier tiles' sums to registers by then).
        const bool fresh = i < 2 || slice_flush_at<split || X3>(i);
#pragma unroll
        for (int kk = 0; kk < 8; kk++) {
          const uint64_t fdesc = sdesc(fs + (uint32_t)kk * 512, kFBlock, 256, kSw32);
          // 16 points' packed weights: columns kk * 8, or with split products the hi
          // pairs of half kk / 4 at (kk / 4) * 64 + (kk % 4) * 8, their residuals 32 on
          const uint32_t tw = tE + (split ? (uint32_t)(kk >> 2) * 64 + (uint32_t)(kk & 3) * 8 : (uint32_t)kk * 8);
          mma_ts_w(tacc, tw, fdesc, idesc_sl, (!fresh || kk > 0) ? 1u : 0u);
          // The residual halves of the weights: U and S to ~2^-16.
          if (split) mma_ts_w(tacc, tw + 32, fdesc, idesc_sl, 1u);
          if (X3)  // the weights against fx's residual half (U only)
            mma_ts_w(tacc, tw, sdesc(fs - kFOff + kFROff + (uint32_t)kk * 512, kFBlock, 256, kSw32),
                     idesc_bf16(128, 32, false, true), 1u);
        }
        mma_commit_w(&pv_done[bb]);
        mma_commit_w(&st_empty[s]);
        if (split || X3) mma_commit_w(&acc_done[j]);
      }
      if (ok) mma_commit_w(acc_full);
      mma_commit_w(&drain[1 + j]);
      mbar_wait_w(&drain[1 + j], 0, ab, nullptr, kWaitNs);
    }
  } else if (warp >= kSoftmaxWarp0) {
    const int wg = (warp - kSoftmaxWarp0) >> 2;
    const int wq = warp & 3;
    const int r = wq * 32 + lane;  // TMEM lane: slot g_base + r
    const uint32_t lane_addr = (uint32_t)(wq * 32) << 16;
    bool ok = true;
    if (kWT && wg == 0) {
      // Slot r's W' row (64B-swizzled) and extra row (32B-swizzled) from the block's image
      // in shared memory into TMEM columns [kTW, kTW + 24) of lane r (packed bf16 pairs).
      if ((ok = mbar_wait(w_full, 0, ab, status))) {
        uint32_t hi[16], ex[16];
#pragma unroll
        for (int c = 0; c < 16; c++) {
          hi[c] = *reinterpret_cast<const uint32_t*>(s_w + off_sw64(r, 2 * c));
          ex[c] = c < 8 ? *reinterpret_cast<const uint32_t*>(s_w + kGC * 64 + off_sw32(r, 2 * c)) : 0u;
        }
        tmem_st16(tmem + lane_addr + kTW, hi);
        tmem_st16(tmem + lane_addr + kTW + 16, ex);
        tmem_wait_st();
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(wt_ready);
    }
    // This warpgroup's share of (U, S) for slot r, moved out of A_wg at every flush.
    float acc[kD + 1];
#pragma unroll
    for (int k = 0; k <= kD; k++) acc[k] = 0.f;
    const uint32_t tA = tmem + lane_addr + kA + (uint32_t)wg * 48;
    auto add_acc = [&]() {
      uint32_t u[32], sv[16];
      tmem_ld32(tA, u);
      tmem_ld16(tA + 32, sv);
      tmem_wait_ld(u, sv);
#pragma unroll
      for (int k = 0; k < kD; k++) acc[k] += __uint_as_float(u[k]);
      acc[kD] += __uint_as_float(sv[0]);
    };
    // Warpgroup wg takes the whole tiles i with i % 2 == wg (out of phase with the other).
    for (int i = wg; ok && i < wk.ntiles; i += 2) {
      const int bb = i % kSBuf;
      if (!(ok = mbar_wait(&s_full[bb], (uint32_t)((i / kSBuf) & 1), ab, status))) break;
      tc_fence_after();
      if (split) {
        weights_hilo_half(tmem + lane_addr + (uint32_t)bb * kGC);
        weights_hilo_half(tmem + lane_addr + (uint32_t)bb * kGC + 64);
      } else {
        weights_in_halves(tmem + lane_addr + (uint32_t)bb * kGC);
      }
      tmem_wait_st();
      if (i >= 2 && slice_flush_at<split || X3>(i)) {
        // The products of this warpgroup's tiles up to i - 2 are complete (acc_done
        // cannot move past that phase before this warpgroup hands over tile i).
        if (!(ok = mbar_wait(&acc_done[wg], (uint32_t)(((i - 2) >> 1) & 1), ab, status))) break;
        tc_fence_after();
        add_acc();
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_ready[wg * kSBuf + bb]);
    }
    const int64_t BH = gridDim.z;
    float* o = part + (((int64_t)blockIdx.y * BH + wk.bh) * G + g_base + r) * (kD + 1);
    const bool have = ok && wk.ntiles > 0 && mbar_wait(acc_full, 0, ab, status);
    if (split || X3) {
      // Epilogue with flushes: what A_wg holds since the last flush, then the two
      // warpgroups' shares added in a fixed order (warpgroup 1 passes its share
      // through the partial row).
      if (have && wg < wk.ntiles) {
        tc_fence_after();
        add_acc();
      }
      if (wg == 1)
        for (int k = 0; k <= kD; k++) o[k] = acc[k];
      named_barrier(1, 256);
      if (wg == 0)
        for (int k = 0; k <= kD; k++) o[k] = acc[k] + o[k];
    } else if (have) {
      // Without flushes: warpgroup 0 writes the numerators U (A_0 + A_1), warpgroup 1
      // the weight sums S.
      tc_fence_after();
      const bool two = wk.ntiles >= 2;  // A_1 holds tiles only when there are two (else unwritten)
      if (wg == 0) {
        uint32_t u0[32], u1[32];
        tmem_ld32(tmem + lane_addr + kA, u0);
        tmem_ld32(tmem + lane_addr + kA + 48, u1);
        tmem_wait_ld2(u0, u1);
#pragma unroll
        for (int k = 0; k < kD; k++) o[k] = two ? __uint_as_float(u0[k]) + __uint_as_float(u1[k]) : __uint_as_float(u0[k]);
      } else {
        uint32_t s0[16], s1[16];
        tmem_ld16(tmem + lane_addr + kA + 32, s0);
        tmem_ld16(tmem + lane_addr + kA + 48 + 32, s1);
        tmem_wait_ld(s0);
        tmem_wait_ld(s1);
        o[kD] = two ? __uint_as_float(s0[0]) + __uint_as_float(s1[0]) : __uint_as_float(s0[0]);
      }
    } else if (ok && wk.ntiles == 0) {
      if (wg == 0)
        for (int k = 0; k < kD; k++) o[k] = 0.f;
      else
        o[kD] = 0.f;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

// One slice CTA per (point split, batch-head, 128-slot block).
int slice_blocks(const Shape& s) { return s.G / kGC < 1 ? 1 : s.G / kGC; }
int slice_splits(const Shape& s) { return point_splits(s, (int)(s.BH() * slice_blocks(s))); }

// fp32 point tensors take the tensor-core path with every operand as two bf16 halves
// (x, fx and W', the weights, z'): the X3 kernels.  Their inputs are first split
// into bf16 hi and residual tensors in the workspace (k_split_bf16).
bool x3_shape(const Shape& s) { return s.dtype == FS_F32; }

// The X3 deslice holds both halves of W' and of z' in shared memory, which fits up to
// 512 slots; past that it runs over ranges of `size` slots (a multiple of 128), each
// with the full lse, adding its output to the earlier ranges'.  `size` minimises the
// padded slots plus half a block per range (a range re-reads x); ties go to the
// larger size.
constexpr int kX3SlotsMax = 512;
struct X3Ranges {
  int n, size;
};
X3Ranges x3_ranges(const Shape& s0) {
  const int Gp = (s0.G + kGC - 1) / kGC * kGC;
  if (s0.dtype != FS_F32 || s0.G <= kX3SlotsMax) return {1, Gp};
  X3Ranges best{0, 0};
  for (int size = kGC; size <= kX3SlotsMax; size += kGC) {
    const int n = (s0.G + size - 1) / size;
    if (best.n == 0 || (int64_t)n * (size + kGC / 2) <= (int64_t)best.n * (best.size + kGC / 2)) best = {n, size};
  }
  return best;
}
size_t half_bytes(const Shape& s) { return align_up((size_t)s.B * s.N * s.H * s.d * 2, 256); }

size_t smem_deslice(int G, bool hilo, int mode = 0, bool ps = false, bool x3 = false) {
  return 1024 + (size_t)G * ((hilo ? kWRow : 96) + (ps ? 128 : 64)) + (mode == 2 ? align_up((size_t)G * 4, 1024) : 0) +
         kStages * (kDStage + (x3 ? kXBytes : 0)) + 512;
}
size_t smem_stats(int G, bool split, bool x3 = false) {
  return 1024 + (size_t)G * (split ? kWRow : 96) + kStages * kXBytes * (x3 ? 2 : 1) + kExBytes + 8 * kTile * 8 + 512;
}
size_t smem_slice(bool x3 = false) {
  return 1024 + (size_t)kWBlock +
         (x3 ? (size_t)(kSliceStages / 2) * (kStageBytes + kXBytes + 2 * kFBlock) : (size_t)kSliceStages * kStageBytes) +
         512;
}

// v (fp32 [B,N,H,d]) -> bf16 hi at dst, bf16 residual at dst + half_bytes(s).
cudaError_t split_points(const Shape& s, const void* v, uint8_t* dst, cudaStream_t st) {
  const int64_t n = s.B * s.N * s.H * s.d;
  k_split_bf16<<<(unsigned)((n / 4 + 255) / 256), 256, 0, st>>>(
      static_cast<const float*>(v), reinterpret_cast<__nv_bfloat16*>(dst),
      reinterpret_cast<__nv_bfloat16*>(dst + half_bytes(s)), n);
  return cudaGetLastError();
}

// Statistics into lse [B,H,N] and the point-extra rows at px.  xr: x's residual
// half (X3), else null.
cudaError_t run_stats(const Shape& s, const void* x, const void* xr, const uint8_t* wimg, float* lse, void* px,
                      uint32_t* status, cudaStream_t st) {
  CUtensorMap xmap, xrmap;
  if (!make_point_map(&xmap, x, s, kD, CU_TENSOR_MAP_SWIZZLE_64B)) return cudaErrorInvalidValue;
  if (!make_point_map(&xrmap, xr ? xr : x, s, kD, CU_TENSOR_MAP_SWIZZLE_64B)) return cudaErrorInvalidValue;
  const int P = point_splits(s, (int)s.BH());
  const bool x3 = xr != nullptr;
  const bool split = s.dot == FS_DOT_BF16X2 || x3;
  const size_t sm = smem_stats(s.G, split, x3);
  const auto kernel = x3 ? k_stats<true, true> : (split ? k_stats<true, false> : k_stats<false, false>);
  cudaError_t e = set_smem(kernel, sm);
  if (e != cudaSuccess) return e;
  kernel<<<dim3((unsigned)P, (unsigned)s.BH()), kStatsThreads, sm, st>>>(xmap, xrmap, wimg, lse, static_cast<uint4*>(px),
                                                                    s.N, padded_n(s), s.H, s.G, P, status);
  return cudaGetLastError();
}

}  // namespace

// The slice on prepared operands (defined below, after the C-ABI-facing helpers).
cudaError_t run_slice(const Shape& s, int G, const void* x, const void* f, const void* xr, const void* fr,
                      const uint8_t* wimg, void* px, float* tokens, float* wsum, int finalize, float* part,
                      uint32_t* status, cudaStream_t st);

bool tc_forward_supported(const Shape& s) {
  // TMA coordinates and the kernels' block counters are 32-bit.
  const int64_t np = (s.N + kTile - 1) / kTile * kTile;
  // fp32 inputs take the tensor cores only when there is enough work to pay for
  // splitting their inputs: B*N*H*G >= 2^24 (smaller problems keep the exact fp32
  // SIMT kernels).  Their deslice runs over slot ranges past 512 slots (X3 ranges).
  const bool fp32_ok = s.dtype == FS_F32 && (double)s.BH() * s.N * s.G >= 16777216.0;
  return (s.dtype == FS_BF16 || fp32_ok) && s.d == kD && s.G <= 1024 && s.N >= 1 &&
         s.BH() * np < (int64_t(1) << 31) && encode_fn() != nullptr;
}

int tc_stats_launch_count(const Shape& s) { return 2 /*prep_w, stats*/ + (x3_shape(s) ? 1 : 0); }

int tc_forward_launch_count(const Shape& s) {
  return 4 /*prep_w, stats, slice, reduce*/ + 1 /*prep_px*/ + 3 * x3_ranges(s).n /*prep_w, prep_z, deslice*/ +
         (x3_shape(s) ? 3 /*splits of x, fx; of x*/ : 0);
}

size_t tc_slice_partials_bytes(const Shape& s0) {
  if (!tc_forward_supported(s0)) return 0;
  const Shape s = tc_padded(s0);
  return (size_t)slice_splits(s) * s.BH() * s.G * (kD + 1) * sizeof(float);
}
// Layouts of the prepared operands: slice [W img | px | (X3) x hi, x r, fx hi, fx r];
// deslice and statistics [W img | Z' img | px | (X3) x hi, x r].
size_t tc_slice_prep_bytes(const Shape& s0) {
  const Shape s = tc_padded(s0);
  return tc_forward_supported(s0)
             ? align_up(w_image_bytes(s), 256) + align_up(px_bytes(s), 256) + (x3_shape(s) ? 4 * half_bytes(s) : 0)
             : 0;
}
size_t tc_deslice_prep_bytes(const Shape& s0) {
  const Shape s = tc_padded(s0);
  const X3Ranges xr = x3_ranges(s0);
  // with several X3 ranges, a range's slices of W, bias and z' too
  const size_t gather = xr.n > 1 ? align_up((size_t)s.H * (kD + 1) * xr.size * sizeof(float), 256) +
                                       align_up((size_t)s.BH() * xr.size * kD * sizeof(float), 256)
                                 : 0;
  return tc_forward_supported(s0) ? align_up(w_image_bytes(s), 256) + align_up(z_image_bytes(s), 256) +
                                        align_up(px_bytes(s), 256) + (x3_shape(s) ? 2 * half_bytes(s) : 0) + gather
                                  : 0;
}

cudaError_t tc_stats(const Shape& s0, const void* x, const float* W, const float* bias, const float* tau, float* lse,
                     void* prep, uint32_t* status, cudaStream_t st) {
  const Shape s = tc_padded(s0);
  uint8_t* wimg = static_cast<uint8_t*>(prep);
  uint8_t* px = wimg + align_up(w_image_bytes(s), 256) + align_up(z_image_bytes(s), 256);
  uint8_t* xh = px + align_up(px_bytes(s), 256);
  cudaError_t e = prep_w(s, s0.G, W, bias, tau, wimg, status, st);
  if (e != cudaSuccess) return e;
  if (!x3_shape(s)) return run_stats(s, x, nullptr, wimg, lse, px, status, st);
  if ((e = split_points(s, x, xh, st)) != cudaSuccess) return e;
  return run_stats(s, xh, xh + half_bytes(s), wimg, lse, px, status, st);
}

cudaError_t tc_slice_fwd(const Shape& s0, const void* x, const void* f, const float* W, const float* bias,
                         const float* tau, float* tokens, float* wsum, float* lse, int finalize, float* part,
                         void* prep, uint32_t* status, cudaStream_t st) {
  const Shape s = tc_padded(s0);
  uint8_t* wimg = static_cast<uint8_t*>(prep);
  uint8_t* px = wimg + align_up(w_image_bytes(s), 256);
  uint8_t* xh = px + align_up(px_bytes(s), 256);
  uint8_t* fh = xh + 2 * half_bytes(s);
  cudaError_t e = prep_w(s, s0.G, W, bias, tau, wimg, status, st);
  if (e != cudaSuccess) return e;
  const void *xr = nullptr, *fr = nullptr;
  if (x3_shape(s)) {
    if ((e = split_points(s, x, xh, st)) != cudaSuccess) return e;
    if ((e = split_points(s, f, fh, st)) != cudaSuccess) return e;
    x = xh;
    xr = xh + half_bytes(s);
    f = fh;
    fr = fh + half_bytes(s);
  }
  if ((e = run_stats(s, x, xr, wimg, lse, px, status, st)) != cudaSuccess) return e;
  return run_slice(s, s0.G, x, f, xr, fr, wimg, px, tokens, wsum, finalize, part, status, st);
}

// The slice on prepared operands: the W image and the point-extra rows at px; xr and
// fr the residual halves of x and fx (X3), else null.
cudaError_t run_slice(const Shape& s, int G, const void* x, const void* f, const void* xr, const void* fr,
                      const uint8_t* wimg, void* px, float* tokens, float* wsum, int finalize, float* part,
                      uint32_t* status, cudaStream_t st) {
  cudaError_t e;
  const bool x3 = xr != nullptr;
  CUtensorMap xmap, fmap, pmap, xrmap, frmap;
  if (!make_point_map(&xmap, x, s, kD, CU_TENSOR_MAP_SWIZZLE_64B)) return cudaErrorInvalidValue;
  if (!make_point_map(&fmap, f, s, 16, CU_TENSOR_MAP_SWIZZLE_32B)) return cudaErrorInvalidValue;
  if (!make_px_map(&pmap, px, s.BH(), padded_n(s))) return cudaErrorInvalidValue;
  if (!make_point_map(&xrmap, x3 ? xr : x, s, kD, CU_TENSOR_MAP_SWIZZLE_64B)) return cudaErrorInvalidValue;
  if (!make_point_map(&frmap, x3 ? fr : f, s, 16, CU_TENSOR_MAP_SWIZZLE_32B)) return cudaErrorInvalidValue;
  const int R = slice_blocks(s), P = slice_splits(s);
  dim3 grid((unsigned)R, (unsigned)P, (unsigned)s.BH());
  const size_t sm = smem_slice(x3);
  const auto kernel = x3 ? k_slice<true, true> : (s.dot == FS_DOT_BF16X2 ? k_slice<true, false> : k_slice<false, false>);
  if ((e = set_smem(kernel, sm)) != cudaSuccess) return e;
  kernel<<<grid, kThreads, sm, st>>>(xmap, fmap, pmap, xrmap, frmap, wimg, part, s.N, padded_n(s), s.H, s.G, P,
                                     status);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  Shape so = s;
  so.G = G;
  return simt_reduce_tokens(so, P, part, s.G, tokens, wsum, finalize, st);
}

cudaError_t tc_slice_fwd_lse(const Shape& s0, const void* x, const void* f, const float* W, const float* bias,
                             const float* tau, const float* lse, float* tokens, float* wsum, int finalize,
                             float* part, void* prep, uint32_t* status, cudaStream_t st) {
  const Shape s = tc_padded(s0);
  uint8_t* wimg = static_cast<uint8_t*>(prep);
  uint8_t* px = wimg + align_up(w_image_bytes(s), 256);
  uint8_t* xh = px + align_up(px_bytes(s), 256);
  uint8_t* fh = xh + 2 * half_bytes(s);
  cudaError_t e = prep_w(s, s0.G, W, bias, tau, wimg, status, st);
  if (e != cudaSuccess) return e;
  const int64_t Np = padded_n(s), npx = s.BH() * Np;
  k_prep_px<<<(unsigned)((npx + 255) / 256), 256, 0, st>>>(lse, reinterpret_cast<uint4*>(px), s.BH(), s.N, Np);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const void *xr = nullptr, *fr = nullptr;
  if (x3_shape(s)) {
    if ((e = split_points(s, x, xh, st)) != cudaSuccess) return e;
    if ((e = split_points(s, f, fh, st)) != cudaSuccess) return e;
    x = xh;
    xr = xh + half_bytes(s);
    f = fh;
    fr = fh + half_bytes(s);
  }
  return run_slice(s, s0.G, x, f, xr, fr, wimg, px, tokens, wsum, finalize, part, status, st);
}

cudaError_t tc_deslice_fwd(const Shape& s0, const void* x, const float* W, const float* bias, const float* tau,
                           const float* zp, const float* lse, void* out, void* prep, uint32_t* status,
                           cudaStream_t st) {
  const Shape sf = tc_padded(s0);  // the whole problem (layout of the workspace)
  const bool x3 = x3_shape(sf);
  const X3Ranges xr = x3_ranges(s0);
  const bool ranged = xr.n > 1;
  Shape s = sf;  // the shape the kernel sees: G = the range's slots
  s.G = xr.size;
  uint8_t* wimg = static_cast<uint8_t*>(prep);
  uint8_t* zimg = wimg + align_up(w_image_bytes(sf), 256);
  uint8_t* px = zimg + align_up(z_image_bytes(sf), 256);
  uint8_t* xh = px + align_up(px_bytes(sf), 256);
  float* wc = reinterpret_cast<float*>(xh + (x3 ? 2 * half_bytes(sf) : 0));  // range slices (ranged only)
  float* bc = wc + (size_t)s.H * kD * xr.size;
  float* zc = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(wc) +
                                       align_up((size_t)s.H * (kD + 1) * xr.size * sizeof(float), 256));
  cudaError_t e;
  const int64_t Np = padded_n(s), npx = s.BH() * Np;
  k_prep_px<<<(unsigned)((npx + 255) / 256), 256, 0, st>>>(lse, reinterpret_cast<uint4*>(px), s.BH(), s.N, Np);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if (x3 && (e = split_points(s, x, xh, st)) != cudaSuccess) return e;
  CUtensorMap xmap, pmap, xrmap;
  if (!make_point_map(&xmap, x3 ? xh : x, s, kD, CU_TENSOR_MAP_SWIZZLE_64B)) return cudaErrorInvalidValue;
  if (!make_point_map(&xrmap, x3 ? xh + half_bytes(s) : x, s, kD, CU_TENSOR_MAP_SWIZZLE_64B))
    return cudaErrorInvalidValue;
  if (!make_px_map(&pmap, px, s.BH(), Np)) return cudaErrorInvalidValue;
  const int P = point_splits(s, (int)s.BH());
  const bool split = s.dot == FS_DOT_BF16X2 || x3;
  // With split products the image holds z' hi then its residual (G*128 bytes per (b,h)).
  const bool ps = x3;
  const bool hilo = split && smem_deslice(s.G, true, 0, ps, x3) <= kMaxSmem;  // up to G = 768 (bf16)
  const size_t sm = smem_deslice(s.G, hilo, 0, ps, x3);
  if (sm > kMaxSmem) return cudaErrorInvalidValue;
  const auto kernel = x3 ? k_deslice<0, true, true> : k_deslice<0, false>;
  if ((e = set_smem(kernel, sm)) != cudaSuccess) return e;
  for (int k = 0; k < xr.n; k++) {
    const int g0 = k * xr.size, G = ranged ? std::min(xr.size, s0.G - g0) : s0.G;
    const float *Wk = W, *bk = bias, *zk = zp;
    if (ranged) {
      if ((e = copy_rows(wc, G, W + g0, s0.G, G, (int64_t)s.H * kD, st)) != cudaSuccess) return e;
      if ((e = copy_rows(bc, G, bias + g0, s0.G, G, s.H, st)) != cudaSuccess) return e;
      if ((e = copy_rows(zc, (int64_t)G * kD, zp + (int64_t)g0 * kD, (int64_t)s0.G * kD, (int64_t)G * kD, s.BH(),
                         st)) != cudaSuccess)
        return e;
      Wk = wc, bk = bc, zk = zc;
    }
    if ((e = prep_w(s, G, Wk, bk, tau, wimg, status, st)) != cudaSuccess) return e;
    const int64_t nz = s.BH() * s.G * kD;
    if (ps)
      k_prep_z2<<<(unsigned)((nz + 255) / 256), 256, 0, st>>>(zk, kD, zimg, s.BH(), G, s.G);
    else
      k_prep_z<<<(unsigned)((nz + 255) / 256), 256, 0, st>>>(zk, zimg, s.BH(), G, s.G);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    kernel<<<dim3((unsigned)P, (unsigned)s.BH()), x3 ? kThreads : kDesl4Threads, sm, st>>>(
        xmap, pmap, xrmap, wimg, zimg, static_cast<__nv_bfloat16*>(out), nullptr, nullptr, nullptr, nullptr, s.N, Np,
        s.H, s.G, P, hilo ? 1 : 0, (uint32_t)s.G * (ps ? 128 : 64), k > 0 ? 1 : 0, status);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  return cudaSuccess;
}

size_t tc_rows_smem(const Shape& s, int mode, bool ps, bool hilo) { return smem_deslice(s.G, hilo, mode, ps); }

cudaError_t tc_rows_bwd(const Shape& s, int mode, const void* x, const uint8_t* wimg, const uint8_t* zimg,
                        const void* px, const void* v, void* dfx, float* delta, float* wds, const float* dS,
                        int accumulate, uint32_t* status, cudaStream_t st) {
  const bool split = s.dot == FS_DOT_BF16X2;
  const bool ps = split && smem_deslice(s.G, false, mode, true) <= kMaxSmem;
  const bool hilo = split && smem_deslice(s.G, true, mode, ps) <= kMaxSmem;
  const size_t sm = smem_deslice(s.G, hilo, mode, ps);
  if (sm > kMaxSmem) return cudaErrorInvalidValue;
  const int64_t Np = padded_n(s);
  CUtensorMap xmap, pmap;
  if (!make_point_map(&xmap, x, s, kD, CU_TENSOR_MAP_SWIZZLE_64B)) return cudaErrorInvalidValue;
  if (!make_px_map(&pmap, px, s.BH(), Np)) return cudaErrorInvalidValue;
  const int P = point_splits(s, (int)s.BH());
  dim3 grid((unsigned)P, (unsigned)s.BH());
  const auto kernel = mode == 1 ? (ps ? k_deslice<1, true> : k_deslice<1, false>)
                                : (ps ? k_deslice<2, true> : k_deslice<2, false>);
  cudaError_t e = set_smem(kernel, sm);
  if (e != cudaSuccess) return e;
  kernel<<<grid, kThreads, sm, st>>>(xmap, pmap, xmap, wimg, zimg, static_cast<__nv_bfloat16*>(dfx),
                                     static_cast<const __nv_bfloat16*>(v), delta, wds, dS, s.N, Np, s.H, s.G, P,
                                     hilo ? 1 : 0, (uint32_t)s.G * 128, accumulate, status);
  return cudaGetLastError();
}

}  // namespace fs
