// bf16 attention forward on the fifth-generation tensor cores (tcgen05 + TMEM + TMA), sm_103a.
//
// What it computes: O = softmax(scale * Q K^T) V per (b, h) slice (paper Section 4.1,
// Eq. attention; the slices are the independent 2-D problems of the Remark in Section 4.2).
// How it keeps the DNF's memory pattern (Section 4, Fig. pipeline): no score matrix, no
// exponential buffer, no transposed K and no denominator vector exists in global memory.
//
//   * Scores S = Q K^T (Eq. mm_psi) are tensor-core products of a Q tile and a K tile, both
//     read from shared memory in their stored row-major layout (K is the "K-major" B operand,
//     so no transpose copy exists).  S lands in tensor memory (TMEM) as fp32.
//   * Step I (row maximum, Section 4.3), Step II (exponentials, Section 4.4) and Step III
//     (denominator, Section 4.5) run online per row in the registers of one softmax thread:
//     running maximum m and running sum l over the key tiles.  When the maximum of a new tile
//     exceeds m by more than kRescaleLog2 (in log2 units), m is raised and O and l are
//     rescaled by exp2(m_old - m_new); otherwise the stale m is kept.  Both are exact: O and l
//     always share the same reference maximum, and exponentials stay <= 2^kRescaleLog2.
//   * The unnormalised probabilities P are rounded to bf16 and stored where the second
//     tensor-core product O += P V (Eq. output_dnf) reads them: TMEM columns of their own, the
//     A operand of that product.  V is the "MN-major" B operand, again as stored.
//   * Step IV (division, Section 4.5) is applied once per row in the epilogue: O / l.
//
// CTA organisation, two-tile kernel (one CTA per SM: 512 TMEM columns, up to ~225 KB shared
// memory):
//   work item = (b*H + h, block of 256 query rows) = two 128-row Q tiles;
//   warps 0-3: softmax + epilogue of Q tile 0; warps 4-7: same for Q tile 1
//              (thread t of such a warpgroup owns query row t of its tile);
//   warp 8:    TMEM allocation; issues the tcgen05.mma products of Q tile 0;
//   warp 9:    the single thread that issues all TMA loads;
//   warp 10:   issues the tcgen05.mma products of Q tile 1;
//   warp 11:   idle (it completes warps 8-11 as one warpgroup for the register split).
// One-tile kernel (d_k = d_v = 64 without a split key axis; two CTAs per SM, 256 TMEM columns
// and ~98 KB of shared memory each): work item = (b*H + h, block of 128 query rows); warps 0-3
// softmax + epilogue, warp 4 TMEM allocation and tcgen05.mma, warp 5 TMA loads.
// K and V tiles of 128 keys stream through an NS-stage shared-memory ring, in the order the
// products use them: K0 K1 V0 K2 V1 ...  TMEM columns: S0 S1 P0 P1 O0 O1 at d_v = 64; one S
// buffer shared by the two tiles, S P0 P1 O0 O1, at d_v = 128 (the two O take 256 columns);
// one tile: S0 P0 O0.  As soon as the S buffer's last reader holds S_j(n) in registers, tile
// j's issuing thread computes S_j(n+1); it runs O_j += P_j(n) V(n) once P_j(n) is written.  The
// softmax writes P_j(n) once O_j += P_j(n-1) V(n-1) is done (it computes the first chunks of
// exponentials before waiting for that).  TMEM lane = row of the Q tile.

// Every mbarrier wait is bounded (globaltimer); on expiry the kernel records
// MOA_ERR_DEVICE_TIMEOUT in g_moa_bf16_status, makes every role leave its loop, and still
// frees its TMEM before returning.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <cstdio>
#include <mutex>

#include "internal.h"
#include "ptx.cuh"
#include "tc_common.cuh"

namespace moa {

__device__ unsigned int g_moa_bf16_status = 0;

namespace {

using namespace ptx;
using namespace tc;

constexpr int kBM = 128;          // query rows per Q tile (= TMEM lanes)
constexpr int kBN = 128;          // keys per K/V tile
constexpr int kQTiles = 2;        // Q tiles per CTA of the two-tile kernel
constexpr float kRescaleLog2 = 8.0f;  // lazy-rescale threshold: exponentials stay <= 2^8
// Every wait polls.  A suspension hint on the MMA issuers' and TMA producer's waits (20 us) gave
// +3.6 % with an earlier d_v = 64 schedule; with the current schedules it is neutral there and
// costs 4 % at d_v = 128 (1712 -> 1638 TFLOP/s on 2x32x8192^2), where the MMA issuers' waits are
// on the critical path; the one-tile kernel ran at 709 instead of 740 with it.

template <int DK, int DV, int QT = 2>
struct Cfg {
  static_assert(DK == 64 || DK == 128, "d_k must be 64 or 128");
  static_assert(QT == 1 || QT == 2, "one or two Q tiles per CTA");
  static_assert(QT == 2 || DV == 64, "one-tile CTAs hold S, P and O of d_v = 64");
  // Warps: 4 softmax warps per Q tile, then the MMA warp of tile 0 (it also allocates and frees
  // TMEM), the TMA warp and, with two tiles, the MMA warp of tile 1.  One-tile CTAs run two per
  // SM (half the registers, TMEM and shared memory each).
  static constexpr int kThreads = QT == 2 ? 384 : 192;
  static constexpr int kMinBlocks = QT == 2 ? 1 : 2;
  static constexpr int kMmaWarp0 = 4 * QT;
  static constexpr int kLoadWarp = 4 * QT + 1;
  static constexpr int kMmaWarp1 = QT == 2 ? 10 : -1;
  // Two tiles: warps 8-11 (MMA issuer of tile 0, TMA, MMA issuer of tile 1, one idle warp) form
  // one warpgroup whose registers move to the two softmax warpgroups with setmaxnreg.  Launched
  // with kRegsLaunch per thread; 256 * kRegsSoftmax + 128 * kRegsCtrl equals the launch
  // allocation, so the softmax warps never wait for registers the CTA does not hold (the host
  // checks the compiled count), and each scheduler's two softmax warps and one control warp fit
  // its 16K registers.  Measured +1.1 to +2 % on 2x32x8192^2, 1x16x32768^2 and
  // 8x8x1024x4096 against 11 warps at 168 registers each (216/56 the same; 4 early chunks no
  // better).
  static constexpr bool kRegSplit = QT == 2;
  static constexpr int kRegsLaunch = 168, kRegsSoftmax = 208, kRegsCtrl = 88;
  static_assert(!kRegSplit || 256 * kRegsSoftmax + 128 * kRegsCtrl <= kThreads * kRegsLaunch,
                "register split");
  static constexpr int kTmemCols = 256 * QT;
  static_assert(DV == 64 || DV == 128, "d_v must be 64 or 128");
  // One 128-byte swizzle panel holds 64 bf16 columns of 128 rows: 16 KB.
  static constexpr int kPanelBytes = 128 * 128;
  static constexpr int kQTileBytes = kBM * DK * 2;
  static constexpr int kKTileBytes = kBN * DK * 2;
  static constexpr int kVTileBytes = kBN * DV * 2;
  static constexpr int kStageBytes = kKTileBytes > kVTileBytes ? kKTileBytes : kVTileBytes;
  // P has TMEM columns of its own, so the next block's scores can be computed as soon as the
  // softmax has read this block's S into registers.  Two tiles with d_v = 64: S0 S1 P0 P1 O0 O1
  // fill the 512 columns.  Two tiles with d_v = 128: O0 O1 take 256 columns, so the two tiles
  // share one S buffer (S P0 P1 O0 O1), and their score products alternate: tile 1's S(n) is
  // computed once tile 0's softmax holds S(n) in registers, tile 0's S(n+1) once tile 1's
  // softmax holds its S(n).  (P in shared memory instead, with an S buffer per tile, measured
  // the same; it moves 128 KB more per key block through shared memory.)  One tile: S0 P0 O0.
  static constexpr bool kSharedS = QT == 2 && DV == 128;
  static constexpr int kStages = QT == 1 ? (DK == 64 ? 5 : 2)
                                 : (DK == 64 && DV == 64) ? 8
                                 : kSharedS ? (DK == 128 ? 5 : 6) : 4;
  static constexpr int kOffQ = 0;
  static constexpr int kOffKV = kOffQ + QT * kQTileBytes;
  static constexpr int kOffBar = kOffKV + kStages * kStageBytes;
  // Each Q tile gets its own issuing thread (its chain of products never waits behind the
  // other tile's).
  static constexpr int kIssuers = QT;
  // Chunks of 32 exponentials computed before the wait for P's buffer (the rest after it), so
  // that the wait for the previous block's P V overlaps them (measured on 4x16x2048^2, d=64:
  // 0 -> 2 chunks 740 -> 812 TFLOP/s; 1x16x32768^2, d=128: 0 -> 3 chunks +2 %; with the
  // two-tile register split, 8x8x1024x4096 (d_k=128, d_v=64): 0 -> 2 chunks 1064 -> 1087, 3 no
  // better; more chunks than these spill or gain nothing).
  static constexpr int kEarlyChunks = QT == 1 ? 2 : DV == 64 ? 2 : 3;
  // barriers: full[NS], empty[NS], q_full, s_full[2], p_ready[2], o_done[2], s_free[2], p_free[2]
  static constexpr int kNumBars = 2 * kStages + 11;
  static constexpr int kOffMisc = kOffBar + kNumBars * 8;  // tmem base, abort flag
  static constexpr int kSmemBytes = kOffMisc + 16 + 1024;  // + slack for 1024-B alignment
  static constexpr uint32_t kTmemS0 = 0, kTmemS1 = kSharedS ? 0 : 128;
  static constexpr uint32_t kTmemP0 = kSharedS ? 128 : 128 * QT;
  static constexpr uint32_t kTmemP1 = kSharedS ? 192 : 320;
  static constexpr uint32_t kTmemO0 = kSharedS ? 256 : 192 * QT;
  static constexpr uint32_t kTmemO1 = kTmemO0 + DV;
  static_assert((QT == 2 ? kTmemO1 : kTmemO0) + DV <= kTmemCols, "TMEM budget");
  // Per SM: 228 KB, 1 KB of it reserved per CTA.
  static_assert(kSmemBytes <= (QT == 2 ? 232448 : 233472 / 2 - 1024), "shared memory budget");
};

// Maximum of 128 values (of their negations if NEG) with four independent 3-input chains.
template <bool NEG>
__device__ __forceinline__ float row_max128(const float* s) {
  auto v = [&](int i) { return NEG ? -s[i] : s[i]; };
  float a0 = v(0), a1 = v(1), a2 = v(2), a3 = v(3);
#pragma unroll
  for (int i = 4; i < 124; i += 8) {
    a0 = max3f(a0, v(i), v(i + 1));
    a1 = max3f(a1, v(i + 2), v(i + 3));
    a2 = max3f(a2, v(i + 4), v(i + 5));
    a3 = max3f(a3, v(i + 6), v(i + 7));
  }
  a0 = max3f(a0, v(124), v(125));
  a1 = max3f(a1, v(126), v(127));
  return max3f(a0, a1, fmaxf(a2, a3));
}

// Multiplies DV fp32 TMEM columns of this thread's lane by alpha (warp-collective).
template <int DV>
__device__ __forceinline__ void tmem_scale_row(uint32_t taddr, float alpha) {
#pragma unroll
  for (int c = 0; c < DV; c += 32) {
    uint32_t o[32];
    tmem_ld_32x32b_x32(taddr + c, o);
    tmem_wait_ld();
    reg_anchor_x32(o);
#pragma unroll
    for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
    tmem_st_32x32b_x32(taddr + c, o);
  }
  tmem_wait_st();
}

// SPLIT: this CTA covers one range of the key axis and writes fp32 partials for the merge kernel
// (separate instantiation, so the unsplit kernel carries none of it).
template <int DK, int DV, bool SPLIT, int QT>
__global__ void __launch_bounds__(Cfg<DK, DV, QT>::kThreads, Cfg<DK, DV, QT>::kMinBlocks)
attn_fwd_bf16_tc_kernel(const __grid_constant__ CUtensorMap tmQ,
                        const __grid_constant__ CUtensorMap tmK,
                        const __grid_constant__ CUtensorMap tmV, __nv_bfloat16* __restrict__ O,
                        int Nq, int Nk, int n_qblocks, float c_log2, uint64_t wait_limit_ns,
                        int n_splits, int kv_per_split, float* __restrict__ ws_o,
                        float2* __restrict__ ws_ml, float* __restrict__ lse) {
  using C = Cfg<DK, DV, QT>;
  static_assert(!SPLIT || QT == 2, "split key axes use two-tile CTAs");
  constexpr int kQTiles = QT;
  constexpr int kMmaWarp0 = C::kMmaWarp0, kLoadWarp = C::kLoadWarp, kMmaWarp1 = C::kMmaWarp1;
  constexpr int kTmemCols = C::kTmemCols;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const uint32_t sQ = smem_u32(smem + C::kOffQ);
  const uint32_t sKV = smem_u32(smem + C::kOffKV);
  const uint32_t bar0 = smem_u32(smem + C::kOffBar);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (C::kStages + s); };
  const uint32_t q_full = bar0 + 8u * (2 * C::kStages);
  auto s_full = [&](int j) { return bar0 + 8u * (2 * C::kStages + 1 + j); };
  auto p_ready = [&](int j) { return bar0 + 8u * (2 * C::kStages + 3 + j); };
  auto o_done = [&](int j) { return bar0 + 8u * (2 * C::kStages + 5 + j); };
  auto s_free = [&](int j) { return bar0 + 8u * (2 * C::kStages + 7 + j); };
  auto p_free = [&](int j) { return bar0 + 8u * (2 * C::kStages + 9 + j); };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::kOffMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::kOffMisc + 4);
  // Split instance only: keys from this CTA's first key block to the end of the key axis, and
  // its key range.  Read from shared memory where needed, so that no register holds them
  // across the key loop (held in registers they made the split instance spill).
  volatile int* keys_from = reinterpret_cast<volatile int*>(smem + C::kOffMisc + 8);
  volatile int* split_s = reinterpret_cast<volatile int*>(smem + C::kOffMisc + 12);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // CTA -> (b*H + h, 128·QT-row query block, key split); splits of one block are adjacent, and
  // blocks of one head are adjacent (head-major), so concurrently running CTAs share K/V in L2.
  const int split = SPLIT ? int(blockIdx.x % n_splits) : 0;
  const int item = SPLIT ? int(blockIdx.x / n_splits) : int(blockIdx.x);
  const int bh = item / n_qblocks;
  const int q0 = (item % n_qblocks) * (kQTiles * kBM);
  // This CTA's key blocks: [kb0, kb0 + n_kt) (all of them unless the key axis is split).
  const int kb0 = SPLIT ? split * kv_per_split : 0;
  const int n_kt = SPLIT ? min((Nk + kBN - 1) / kBN - kb0, kv_per_split) : (Nk + kBN - 1) / kBN;
  const WaitCtl wc{abort_flag, wait_limit_ns, 0u, &g_moa_bf16_status};

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), C::kIssuers);  // one commit from each MMA issuer
    }
    mbar_init(q_full, 1);
    for (int j = 0; j < kQTiles; ++j) {
      mbar_init(s_full(j), 1);
      mbar_init(p_ready(j), 4 * 32);
      mbar_init(o_done(j), 1);
      mbar_init(s_free(j), 4 * 32);
      mbar_init(p_free(j), 1);
    }
    *abort_flag = 0;
    if constexpr (SPLIT) {
      *keys_from = Nk - kb0 * kBN;
      *split_s = split;
    }
    fence_barrier_init();
  }
  if (warp == kMmaWarp0) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  if (warp >= 4 * QT) {
    // Control warps (MMA issuers, TMA producer, and with two tiles an idle warp).
    if constexpr (C::kRegSplit)
      asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(C::kRegsCtrl));
  if (warp == kLoadWarp) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      mbar_arrive_expect_tx(q_full, kQTiles * C::kQTileBytes);
      for (int j = 0; j < kQTiles; ++j)
#pragma unroll
        for (int p = 0; p < DK / 64; ++p)
          tma_load_3d(sQ + j * C::kQTileBytes + p * C::kPanelBytes, &tmQ, q_full, p * 64,
                      q0 + j * kBM, bh);
      int slot = 0;
      uint32_t phase = 0;
      uint32_t issued = 0, issued_phase = 0;  // per slot: a load was issued / its phase bit
      bool aborted = false;
      // Ring order = the MMA issuers' consumption order: K0 K1 V0 K2 V1 ... (block n+1's scores
      // come before block n's P V).
      for (int t = 0; t < 2 * n_kt; ++t) {
        bool is_k;
        int n;
        if (t == 0) {
          is_k = true;
          n = 0;
        } else {
          const int u = t - 1, nn = u >> 1;
          is_k = (u & 1) == 0 && nn + 1 < n_kt;
          n = is_k ? nn + 1 : nn;
        }
        if (!wait_bounded(empty_bar(slot), phase ^ 1u, wc)) {
          aborted = true;
          break;
        }
        issued |= 1u << slot;
        issued_phase = (issued_phase & ~(1u << slot)) | (phase << slot);
        const uint32_t dst = sKV + slot * C::kStageBytes;
        if (is_k) {
          mbar_arrive_expect_tx(full_bar(slot), C::kKTileBytes);
#pragma unroll
          for (int p = 0; p < DK / 64; ++p)
            tma_load_3d(dst + p * C::kPanelBytes, &tmK, full_bar(slot), p * 64, (kb0 + n) * kBN,
                        bh);
        } else {
          mbar_arrive_expect_tx(full_bar(slot), C::kVTileBytes);
#pragma unroll
          for (int p = 0; p < DV / 64; ++p)
            tma_load_3d(dst + p * C::kPanelBytes, &tmV, full_bar(slot), p * 64, (kb0 + n) * kBN,
                        bh);
        }
        if (++slot == C::kStages) {
          slot = 0;
          phase ^= 1u;
        }
      }
      if (aborted || *abort_flag) {
        // Let every copy already issued land before the CTA can exit.
        wait_quiesce(q_full, 0, wait_limit_ns, &g_moa_bf16_status);
        for (int sl = 0; sl < C::kStages; ++sl)
          if (issued & (1u << sl))
            wait_quiesce(full_bar(sl), (issued_phase >> sl) & 1u, wait_limit_ns, &g_moa_bf16_status);
      }
    }
  } else if (warp == kMmaWarp0 || warp == kMmaWarp1) {
    // ---------------------------------------------------------------- MMA issuers
    // One issuing thread per Q tile, so that neither tile's products wait behind the other's.
    // Straight-line issue code: every operand of every tcgen05.mma is a loop invariant or an
    // unrolled constant offset, so each thread issues at the tensor pipe's rate.
    if (lane == 0) {
      const int j = warp == kMmaWarp0 ? 0 : 1;
      constexpr uint32_t kIdescQK = make_idesc(kBM, kBN, false);
      constexpr uint32_t kIdescPV = make_idesc(kBM, DV, true);
      const uint32_t tS = tmem + (j ? C::kTmemS1 : C::kTmemS0);
      const uint32_t tP = tmem + (j ? C::kTmemP1 : C::kTmemP0);
      const uint32_t tO = tmem + (j ? C::kTmemO1 : C::kTmemO0);
      const uint32_t sQj = sQ + j * C::kQTileBytes;
      const uint32_t bar_s_full = s_full(j), bar_p_ready = p_ready(j), bar_s_free = s_free(j);
      const uint32_t bar_p_free = p_free(j);
      int slot = 0;
      uint32_t phase = 0;
      auto next = [&]() {
        if (++slot == C::kStages) {
          slot = 0;
          phase ^= 1u;
        }
      };
      // S = Q K^T: DK/16 MMAs (M=128, N=128, K=16), both operands K-major; the k-th step is
      // panel k/4 of the 128-byte-swizzled tile, 32 bytes further for each step inside it.
      auto issue_qk = [&](uint32_t kb) {
#pragma unroll
        for (int kk = 0; kk < DK / 16; ++kk) {
          const uint32_t off = (kk >> 2) * C::kPanelBytes + (kk & 3) * 32;
          mma_f16_ss(tS, make_sdesc_sw128(sQj + off, 16, 1024),
                     make_sdesc_sw128(kb + off, 16, 1024), kIdescQK, kk > 0 ? 1u : 0u);
        }
      };
      // O (+)= P V: 8 MMAs (M=128, N=DV, K=16).  A = P from TMEM (bf16 pairs: 8 columns per
      // 16 keys).  B = V tile, MN-major: groups of 8 keys 1024 B apart (stride byte offset),
      // 64-column panels kPanelBytes apart (leading byte offset).
      auto issue_pv = [&](uint32_t vb, uint32_t acc_first) {
#pragma unroll
        for (int kk = 0; kk < kBN / 16; ++kk)
          mma_f16_ts(tO, tP + kk * 8, make_sdesc_sw128(vb + kk * 2048, C::kPanelBytes, 1024),
                     kIdescPV, kk > 0 ? 1u : acc_first);
      };
      bool ok = wait_bounded(q_full, 0, wc) && wait_bounded(full_bar(slot), phase, wc);
      // Tile 1's first scores wait until tile 0 holds its own in registers: required with one
      // S buffer for both tiles (d_v = 128); with an S buffer per tile and d_k = 128 it keeps
      // the tiles' reads of S from tensor memory from coinciding (measured +2 % on
      // 8x8x1024x4096, d_k = 128, d_v = 64; -2 % with d_k = 64, which therefore starts both).
      if ((DK == 128 || C::kSharedS) && j == 1) ok = ok && wait_bounded(s_free(0), 0, wc);
      if (ok) {
        tc_fence_after_sync();
        const int ks = slot;
        next();
        issue_qk(sKV + ks * C::kStageBytes);
        mma_commit(bar_s_full);
        mma_commit(empty_bar(ks));
      }
      {
        // P_j has TMEM columns of its own: S_j(n+1) is issued as soon as the S buffer's last
        // reader has its scores in registers, and O_j += P_j(n) V(n) once P_j(n) is written.
        for (int n = 0; ok && n < n_kt; ++n) {
          const uint32_t par = uint32_t(n) & 1u;
          if (n + 1 < n_kt) {
            const int ks = slot;
            // The S buffer may take block n+1's scores once its last reader has them in
            // registers: this tile's softmax (own S buffer), or with one S buffer shared by the
            // two tiles, the other tile's softmax (block n for tile 0, block n+1 for tile 1).
            ok = wait_bounded(full_bar(slot), phase, wc) &&
                 (C::kSharedS ? wait_bounded(s_free(j ^ 1), j ? (par ^ 1u) : par, wc)
                              : wait_bounded(bar_s_free, par, wc));
            next();
            if (!ok) break;
            tc_fence_after_sync();
            issue_qk(sKV + ks * C::kStageBytes);
            mma_commit(bar_s_full);
            mma_commit(empty_bar(ks));
          }
          const int vs = slot;
          ok = wait_bounded(full_bar(slot), phase, wc) && wait_bounded(bar_p_ready, par, wc);
          next();
          if (!ok) break;
          tc_fence_after_sync();
          issue_pv(sKV + vs * C::kStageBytes, n > 0 ? 1u : 0u);
          mma_commit(bar_p_free);
          mma_commit(empty_bar(vs));
        }
      }
      // Always signal the epilogue barrier once everything issued has completed, so that the
      // TMEM is quiescent before it is freed even on the abort path.
      mma_commit(o_done(j));
    }
  }
  } else {
    if constexpr (C::kRegSplit)
      asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(C::kRegsSoftmax));
    // ---------------------------------------------------------------- softmax warpgroups
    const int j = warp >> 2;                // Q tile of this warpgroup
    const int lane_base = (warp & 3) * 32;  // TMEM lanes of this warp
    const int row = lane_base + lane;       // query row inside the tile
    const uint32_t tS = tmem + (uint32_t(lane_base) << 16) + (j ? C::kTmemS1 : C::kTmemS0);
    const uint32_t tO = tmem + (uint32_t(lane_base) << 16) + (j ? C::kTmemO1 : C::kTmemO0);
    const uint32_t tP = tmem + (uint32_t(lane_base) << 16) + (j ? C::kTmemP1 : C::kTmemP0);
    const bool neg = c_log2 < 0.f;
    float m = -INFINITY;  // running maximum of c_log2 * s (log2 units)
    float l = 0.f;        // running sum of exp2(c_log2 * s - m)
    bool ok = true;
    for (int n = 0; n < n_kt; ++n) {
      if (!wait_bounded(s_full(j), uint32_t(n) & 1u, wc)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
      uint32_t sr[128];
      tmem_load_row128(tS, sr);
      // S_j(n) is in registers: the MMA issuer may overwrite it with S_j(n+1).
      tc_fence_before_sync();
      mbar_arrive(s_free(j));
      float* s = reinterpret_cast<float*>(sr);
      // Keys of this tile that exist.
      const int valid = SPLIT ? min(kBN, *keys_from - n * kBN) : min(kBN, Nk - (kb0 + n) * kBN);
      // Step I: maximum of the scaled scores of this tile (max of s if c >= 0, else of -s).
      float tmax;
      if (valid == kBN) {
        tmax = neg ? -row_max128<true>(s) : row_max128<false>(s);
      } else {
        float mx = -INFINITY;
#pragma unroll
        for (int i = 0; i < kBN; ++i)
          if (i < valid) mx = fmaxf(mx, neg ? -s[i] : s[i]);
        tmax = neg ? -mx : mx;
      }
      const float m_tile = c_log2 * tmax;  // max over the tile's keys of c_log2 * s
      bool rescale = false;  // warp-uniform
      float alpha = 1.f;
      if (n == 0) {
        m = m_tile;
      } else {
        const bool need = m_tile > m + kRescaleLog2;
        if (__any_sync(0xffffffffu, need)) {
          const float m_new = fmaxf(m, m_tile);
          alpha = ex2_approx(m - m_new);
          l *= alpha;
          m = m_new;
          rescale = true;
        }
      }
      // Step II + III: p = exp2(c*s - m), row sum, P -> bf16 pairs into P_j's TMEM columns
      // (chunk c of 32 scores becomes 16 packed columns at column 16c of P_j).
      const uint64_t cc = pack_f32x2(c_log2, c_log2);
      const uint64_t mm = pack_f32x2(-m, -m);
      float l0 = 0.f, l1 = 0.f, l2 = 0.f, l3 = 0.f;
      const bool full = valid == kBN;
      // Chunk c of 32 scores -> p = exp2(c*s - m), row sums, bf16 pairs in pk.
      auto exp_chunk = [&](int c, uint32_t* pk) {
#pragma unroll
        for (int i = 0; i < 32; i += 4) {
          const int k = 32 * c + i;
          float x0, x1, x2, x3;
          ffma2(x0, x1, s[k], s[k + 1], cc, mm);
          ffma2(x2, x3, s[k + 2], s[k + 3], cc, mm);
          if (!full) {
            x0 = k < valid ? x0 : -INFINITY;
            x1 = k + 1 < valid ? x1 : -INFINITY;
            x2 = k + 2 < valid ? x2 : -INFINITY;
            x3 = k + 3 < valid ? x3 : -INFINITY;
          }
          const float p0 = ex2_approx(x0), p1 = ex2_approx(x1);
          const float p2 = ex2_approx(x2), p3 = ex2_approx(x3);
          fadd2(l0, l1, p0, p1);
          fadd2(l2, l3, p2, p3);
          pk[i >> 1] = pack_bf16x2(p0, p1);
          pk[(i >> 1) + 1] = pack_bf16x2(p2, p3);
        }
      };
      // Chunk c of P to where O += P V reads it: 16 packed TMEM columns at column 16c.
      auto store_chunk = [&](int c, const uint32_t* pk) { tmem_st_32x32b_x16(tP + 16 * c, pk); };
      // The first kEarlyChunks chunks are computed before waiting for P_j's buffer, so that
      // the wait overlaps their exponentials.
      constexpr int kEarly = C::kEarlyChunks;
      uint32_t pe[kEarly > 0 ? 16 * kEarly : 1];
#pragma unroll
      for (int c = 0; c < kEarly; ++c) exp_chunk(c, pe + 16 * c);
      // P_j's buffer is free, and O_j may be rescaled, once O_j += P_j(n-1) V(n-1) is done.
      if (n > 0 && !wait_bounded(p_free(j), uint32_t(n - 1) & 1u, wc)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
#pragma unroll
      for (int c = 0; c < kEarly; ++c) store_chunk(c, pe + 16 * c);
#pragma unroll
      for (int c = kEarly; c < 4; ++c) {
        uint32_t pk[16];
        exp_chunk(c, pk);
        store_chunk(c, pk);
      }
      l += (l0 + l1) + (l2 + l3);
      // O_j holds P V of tiles < n, complete because S_j(n) was committed after that product;
      // rescaled here, after the scores are dead, and before P_j(n) is released to the MMA.
      if (rescale) tmem_scale_row<DV>(tO, alpha);
      tmem_wait_st();
      tc_fence_before_sync();
      mbar_arrive(p_ready(j));
    }
    // Natural-log LSE of the scaled scores, final once the loop is done: m and l are in log2
    // units of c_log2 * s, and l is relative to m whether or not the last maximum update was
    // taken (lazy rescale).
    if (!SPLIT && lse != nullptr && ok && q0 + j * kBM + row < Nq)
      lse[size_t(bh) * Nq + q0 + j * kBM + row] = (m + lg2_approx(l)) * 0.69314718055994531f;
    // Epilogue, Step IV: O / l -> bf16 -> global.  With a split key axis this CTA instead
    // writes its unnormalised fp32 O rows and (m, l) for the merge kernel.
    if (SPLIT && ok && wait_bounded(o_done(j), 0, wc)) {
      tc_fence_after_sync();
      const int grow = q0 + j * kBM + row;
      const size_t prow = (size_t(*split_s) * (gridDim.x / n_splits / n_qblocks) + bh) * Nq + grow;
      float* orow = ws_o + prow * DV;
#pragma unroll
      for (int c = 0; c < DV; c += 16) {
        uint32_t o[16];
        tmem_ld_32x32b_x16(tO + c, o);
        tmem_wait_ld();
        reg_anchor_x16(o);
        if (grow < Nq) {
          float4* dst = reinterpret_cast<float4*>(orow + c);
#pragma unroll
          for (int i = 0; i < 4; ++i)
            dst[i] = make_float4(__uint_as_float(o[4 * i]), __uint_as_float(o[4 * i + 1]),
                                 __uint_as_float(o[4 * i + 2]), __uint_as_float(o[4 * i + 3]));
        }
      }
      if (grow < Nq) ws_ml[prow] = make_float2(m, l);
    } else if (!SPLIT && ok && wait_bounded(o_done(j), 0, wc)) {
      tc_fence_after_sync();
      const float inv_l = 1.0f / l;
      const int grow = q0 + j * kBM + row;
      __nv_bfloat16* orow = O + (size_t(bh) * Nq + grow) * DV;
#pragma unroll
      for (int c = 0; c < DV; c += 32) {
        uint32_t o[32];
        tmem_ld_32x32b_x32(tO + c, o);
        tmem_wait_ld();
        reg_anchor_x32(o);
        if (grow < Nq) {
          uint4 pkt[4];
          uint32_t* w = reinterpret_cast<uint32_t*>(pkt);
#pragma unroll
          for (int i = 0; i < 16; ++i)
            w[i] = pack_bf16x2(__uint_as_float(o[2 * i]) * inv_l,
                               __uint_as_float(o[2 * i + 1]) * inv_l);
          uint4* dst = reinterpret_cast<uint4*>(orow + c);
#pragma unroll
          for (int i = 0; i < 4; ++i) dst[i] = pkt[i];
        }
      }
    }
  }

  // Teardown: wait for the tensor core to go quiet before freeing TMEM.
  if (warp == kMmaWarp0) {
    wait_quiesce(o_done(0), 0, wait_limit_ns, &g_moa_bf16_status);
    if (QT == 2) wait_quiesce(o_done(1), 0, wait_limit_ns, &g_moa_bf16_status);
  }
  tc_fence_before_sync();
  __syncthreads();
  if (warp == kMmaWarp0) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// Merge of a split key axis (the identity behind Eq. stable_softmax applied across key ranges):
// with per-split reference maxima m_s (log2 units), unnormalised rows O_s and sums l_s,
//   M = max_s m_s,  O = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s.
// One warp per output row; lane c handles columns c, c+32, ...
template <int DV>
__global__ void __launch_bounds__(256)
splitkv_merge_kernel(const float* __restrict__ ws_o, const float2* __restrict__ ws_ml,
                     __nv_bfloat16* __restrict__ O, long long rows, int n_splits) {
  const long long r = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= rows) return;
  float M = -INFINITY;
  for (int s = 0; s < n_splits; ++s) M = fmaxf(M, ws_ml[s * rows + r].x);
  float L = 0.f;
  float acc[DV / 32];
#pragma unroll
  for (int i = 0; i < DV / 32; ++i) acc[i] = 0.f;
  for (int s = 0; s < n_splits; ++s) {
    const float2 ml = ws_ml[s * rows + r];
    const float w = ex2_approx(ml.x - M);
    L = fmaf(w, ml.y, L);
    const float* src = ws_o + (s * rows + r) * DV;
#pragma unroll
    for (int i = 0; i < DV / 32; ++i) acc[i] = fmaf(w, src[lane + 32 * i], acc[i]);
  }
  const float inv = 1.0f / L;
#pragma unroll
  for (int i = 0; i < DV / 32; ++i) O[r * DV + lane + 32 * i] = __float2bfloat16_rn(acc[i] * inv);
}

// Failure-path self test: one thread waits, with the kernel's bounded wait, on an mbarrier
// phase that nothing completes.  The wait must give up after limit_ns, record
// MOA_ERR_DEVICE_TIMEOUT in the status word and return, leaving the context usable.
__global__ void __launch_bounds__(32, 1) wait_timeout_selftest_kernel(uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);
    abort_flag = 0;
    fence_barrier_init();
  }
  __syncwarp();
  if (threadIdx.x == 0) {
    const WaitCtl wc{&abort_flag, limit_ns, 0u, &g_moa_bf16_status};
    if (wait_bounded(smem_u32(&bar), 0, wc)) atomicExch(&g_moa_bf16_status, 0xBADu);
  }
}

// ------------------------------------------------------------------------------------------
// Host side
// ------------------------------------------------------------------------------------------
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode_fn(char* msg, size_t msglen) {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  static char err[256] = {0};
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                                     cudaEnableDefault, &q);
    if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || p == nullptr) {
      snprintf(err, sizeof(err), "cuTensorMapEncodeTiled unavailable: %s",
               cudaGetErrorString(e));
      return;
    }
    fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  if (!fn) snprintf(msg, msglen, "%s", err);
  return fn;
}

}  // namespace

// 3-D map over a contiguous [BH, N, d] bf16 tensor; box = 64 columns x 128 rows x 1 slice,
// 128-byte swizzle.  Rows past N inside a slice read as zero (never the next slice).
bool encode_bf16_map(CUtensorMap* map, const void* base, int64_t BH, int64_t N, int64_t d,
                     char* msg, size_t msglen) {
  return encode_bf16_map_box(map, base, BH, N, d, 128, msg, msglen);
}

bool encode_bf16_map_box(CUtensorMap* map, const void* base, int64_t BH, int64_t N, int64_t d,
                         int box_rows, char* msg, size_t msglen) {
  EncodeTiledFn enc = get_encode_fn(msg, msglen);
  if (!enc) return false;
  const cuuint64_t dims[3] = {cuuint64_t(d), cuuint64_t(N), cuuint64_t(BH)};
  const cuuint64_t strides[2] = {cuuint64_t(d * 2), cuuint64_t(N * d * 2)};
  const cuuint32_t box[3] = {64, cuuint32_t(box_rows), 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims,
                   strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    snprintf(msg, msglen, "cuTensorMapEncodeTiled failed (%d) for [%lld,%lld,%lld]", int(r),
             (long long)BH, (long long)N, (long long)d);
    return false;
  }
  return true;
}

// 3-D map over a contiguous fp32 [BH, N, d] tensor; box = box_cols columns (32: one 128-byte
// swizzle row) x box_rows rows x 1 slice, 128-byte swizzle.
bool encode_f32_map_sw128(CUtensorMap* map, const void* base, int64_t BH, int64_t N, int64_t d,
                          int box_cols, int box_rows, char* msg, size_t msglen) {
  EncodeTiledFn enc = get_encode_fn(msg, msglen);
  if (!enc) return false;
  const cuuint64_t dims[3] = {cuuint64_t(d), cuuint64_t(N), cuuint64_t(BH)};
  const cuuint64_t strides[2] = {cuuint64_t(d * 4), cuuint64_t(N * d * 4)};
  const cuuint32_t box[3] = {cuuint32_t(box_cols), cuuint32_t(box_rows), 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<void*>(base), dims, strides,
                   box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    snprintf(msg, msglen, "cuTensorMapEncodeTiled failed (%d) for fp32 [%lld,%lld,%lld]", int(r),
             (long long)BH, (long long)N, (long long)d);
    return false;
  }
  return true;
}

namespace {

// One-tile CTAs, two per SM, for d_k = d_v = 64 when the key axis is not split: the two CTAs
// on an SM can overlap each other's start-up and epilogue (measured 680 -> 740 TFLOP/s on
// 4x16x2048^2; SM active cycles 81 % -> 91 %).  With d_k = 128 only two
// 32 KB ring stages fit beside the Q tile, and the two-tile kernel stays faster (1063 vs 981).
template <int DK, int DV>
constexpr bool kUseOneTile = DV == 64 && DK == 64;

template <int DK, int DV>
int launch_tc(const AttnArgs& a, const CUtensorMap& mq, const CUtensorMap& mk,
              const CUtensorMap& mv, const SplitPlan& sp, void* ws, char* msg, size_t msglen) {
  using C = Cfg<DK, DV>;
  constexpr int QT1 = kUseOneTile<DK, DV> ? 1 : 2;
  using C1 = Cfg<DK, DV, QT1>;
  if (sp.n_splits > 1 && a.lse != nullptr) {
    snprintf(msg, msglen, "the log-sum-exp output is not available with a split key axis");
    return 1;
  }
  const bool split = sp.n_splits > 1;
  auto kern = split ? attn_fwd_bf16_tc_kernel<DK, DV, true, 2>
                    : attn_fwd_bf16_tc_kernel<DK, DV, false, QT1>;
  const int threads = split ? C::kThreads : C1::kThreads;
  const int smem_bytes = split ? C::kSmemBytes : C1::kSmemBytes;
  const int tile_rows = split ? kQTiles * kBM : QT1 * kBM;
  const cudaError_t attr_err = ensure_smem_limit(reinterpret_cast<const void*>(kern), smem_bytes);
  if (attr_err != cudaSuccess) {
    snprintf(msg, msglen, "cudaFuncSetAttribute (bf16 kernel): %s", cudaGetErrorString(attr_err));
    return 5;
  }
  if (split || QT1 == 2) {
    // The register split of the two-tile kernel moves registers inside the CTA's launch
    // allocation: refuse a build whose allocation is short of the split's sum.
    static std::atomic<int> regs_of[2] = {-1, -1};  // unsplit and split instance
    std::atomic<int>& regs = regs_of[split ? 1 : 0];
    if (regs.load(std::memory_order_relaxed) < 0) {
      cudaFuncAttributes fa;
      const cudaError_t e = cudaFuncGetAttributes(&fa, reinterpret_cast<const void*>(kern));
      if (e != cudaSuccess) {
        snprintf(msg, msglen, "cudaFuncGetAttributes (bf16 kernel): %s", cudaGetErrorString(e));
        return 5;
      }
      regs.store(fa.numRegs, std::memory_order_relaxed);
    }
    const int r = regs.load(std::memory_order_relaxed);
    if (r * C::kThreads < 256 * C::kRegsSoftmax + 128 * C::kRegsCtrl) {
      snprintf(msg, msglen, "bf16 kernel compiled to %d registers per thread, short of the "
               "register split", r);
      return 5;
    }
  }
  const int64_t n_qblocks = (a.Nq + tile_rows - 1) / tile_rows;
  const int64_t grid = a.B * a.H * n_qblocks * sp.n_splits;
  if (grid > 0x7fffffffLL) {
    snprintf(msg, msglen, "bf16 path: %lld CTAs exceeds the grid limit", (long long)grid);
    return 3;
  }
  const float c_log2 = a.scale * 1.4426950408889634f;
  const int64_t rows = a.B * a.H * a.Nq;
  float* ws_o = sp.n_splits > 1 ? static_cast<float*>(ws) : nullptr;
  float2* ws_ml = sp.n_splits > 1
                      ? reinterpret_cast<float2*>(static_cast<float*>(ws) + sp.n_splits * rows * DV)
                      : nullptr;
  kern<<<dim3(unsigned(grid)), dim3(threads), smem_bytes, a.stream>>>(
      mq, mk, mv, static_cast<__nv_bfloat16*>(a.O), int(a.Nq), int(a.Nk), int(n_qblocks), c_log2,
      wait_limit_ns(), sp.n_splits, sp.kv_per_split, ws_o, ws_ml, a.lse);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    snprintf(msg, msglen, "bf16 kernel launch: %s", cudaGetErrorString(e));
    return 5;
  }
  if (sp.n_splits > 1) {
    const long long blocks = (rows + 7) / 8;
    splitkv_merge_kernel<DV><<<dim3(unsigned(blocks)), dim3(256), 0, a.stream>>>(
        ws_o, ws_ml, static_cast<__nv_bfloat16*>(a.O), rows, sp.n_splits);
    e = cudaGetLastError();
    if (e != cudaSuccess) {
      snprintf(msg, msglen, "split merge launch: %s", cudaGetErrorString(e));
      return 5;
    }
  }
  return 0;
}

}  // namespace

SplitPlan plan_splits(int64_t Nk, int requested) {
  const int64_t n_kt = (Nk + kBN - 1) / kBN;
  int64_t want = requested < 1 ? 1 : requested;
  if (want > n_kt) want = n_kt;
  const int64_t per = (n_kt + want - 1) / want;
  SplitPlan sp;
  sp.kv_per_split = int(per);
  sp.n_splits = int((n_kt + per - 1) / per);  // every split gets at least one key block
  return sp;
}

static_assert(kQTiles * kBM == kQBlockRows, "query block size");

// Model: a whole query block takes time 1; a split of `per` of its n_kt key blocks takes
// per/n_kt + kSplitFixed (the Q load, the pipeline fill and drain, and the fp32 partial rows,
// measured at about 0.08 of a 16-block CTA).  The split CTAs of t blocks run as
// ceil(t * splits / sms) rounds.  Splitting only pays when the blocks leave SMs idle: with a
// full wave or more, every split CTA adds its fixed cost and the merge to work that already
// fills the GPU (measured slower on every such shape tried).  Splits keep >= 2 key blocks.
SplitPlan plan_splits_auto(int64_t units, int64_t Nk, int sms) {
  constexpr double kSplitFixed = 0.08;
  constexpr int kMaxSplits = 32;
  SplitPlan none;
  if (units <= 0 || Nk <= 0 || sms <= 0 || units >= sms) return none;
  const int64_t n_kt = (Nk + kBN - 1) / kBN;
  double best = 1.0;  // one round of whole blocks
  SplitPlan pick = none;
  for (int64_t s = 2; s <= kMaxSplits && s <= n_kt / 2; ++s) {
    const int64_t per = (n_kt + s - 1) / s;
    const int64_t used = (n_kt + per - 1) / per;
    const double rounds = double((units * used + sms - 1) / sms);
    const double est = rounds * (double(per) / double(n_kt) + kSplitFixed);
    if (est < best - 0.02) {
      best = est;
      pick.n_splits = int(used);
      pick.kv_per_split = int(per);
    }
  }
  return best <= 0.85 ? pick : none;
}

size_t splitkv_workspace_bytes(int64_t rows, int64_t dv, const SplitPlan& sp) {
  if (sp.n_splits <= 1) return 0;
  return size_t(sp.n_splits) * size_t(rows) * (size_t(dv) * 4 + 8);
}

int launch_attn_fwd_bf16(const AttnArgs& a, char* msg, size_t msglen) {
  return launch_attn_fwd_bf16_split(a, plan_splits(a.Nk, 1), nullptr, msg, msglen);
}

int launch_attn_fwd_bf16_split(const AttnArgs& a, const SplitPlan& sp, void* ws, char* msg,
                               size_t msglen) {
  const int64_t BH = a.B * a.H;
  CUtensorMap mq, mk, mv;
  if (!encode_bf16_map(&mq, a.Q, BH, a.Nq, a.dk, msg, msglen)) return 5;
  if (!encode_bf16_map(&mk, a.K, BH, a.Nk, a.dk, msg, msglen)) return 5;
  if (!encode_bf16_map(&mv, a.V, BH, a.Nk, a.dv, msg, msglen)) return 5;
  if (a.dk == 64 && a.dv == 64) return launch_tc<64, 64>(a, mq, mk, mv, sp, ws, msg, msglen);
  if (a.dk == 128 && a.dv == 128) return launch_tc<128, 128>(a, mq, mk, mv, sp, ws, msg, msglen);
  if (a.dk == 128 && a.dv == 64) return launch_tc<128, 64>(a, mq, mk, mv, sp, ws, msg, msglen);
  if (a.dk == 64 && a.dv == 128) return launch_tc<64, 128>(a, mq, mk, mv, sp, ws, msg, msglen);
  snprintf(msg, msglen, "bf16 path supports d_k, d_v in {64, 128}; got d_k=%lld d_v=%lld",
           (long long)a.dk, (long long)a.dv);
  return 3;
}

// ------------------------------------------------------------------------------------------
// Split key axis without any allocation: the partial rows live in a fixed device array
// ------------------------------------------------------------------------------------------
// One array per device that loads this library, held until the process exits.  Every call of
// the allocation-free entry point on a device uses the same array, so calls that overlap on the
// GPU (different streams, no ordering between them) race on it.  Nothing in it needs to start
// at zero: the split kernel writes every partial row and (m, l) pair the merge kernel reads.
static __device__ __align__(256) unsigned char g_splitkv_scratch[kNoallocScratchBytes];

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of g_splitkv_scratch on the current device.  In host code the array's name
// only stands for the device symbol; its address on a device comes from cudaGetSymbolAddress,
// asked once per device, with that device current.
void* scratch_address(char* msg, size_t msglen) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    snprintf(msg, msglen, "no usable current device for the static scratch (%s)",
             cudaGetErrorString(e));
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_splitkv_scratch);
    if (e != cudaSuccess || p == nullptr) {
      snprintf(msg, msglen, "cudaGetSymbolAddress(static scratch) on device %d: %s", dev,
               cudaGetErrorString(e));
      return nullptr;
    }
    g_scratch_addr[dev] = p;
  }
  return g_scratch_addr[dev];
}
}  // namespace

int launch_attn_fwd_bf16_split_noalloc(const AttnArgs& a, const SplitPlan& sp, char* msg,
                                       size_t msglen) {
  const size_t need = splitkv_workspace_bytes(a.B * a.H * a.Nq, a.dv, sp);
  if (need > kNoallocScratchBytes) {
    snprintf(msg, msglen,
             "split needs %zu bytes of scratch but the static scratch holds %zu; use fewer "
             "splits or moa_attn_fwd_splitkv with a workspace of your own",
             need, size_t(kNoallocScratchBytes));
    return 3;
  }
  void* ws = nullptr;
  if (need > 0) {
    ws = scratch_address(msg, msglen);
    if (ws == nullptr) return 5;
  }
  return launch_attn_fwd_bf16_split(a, sp, ws, msg, msglen);
}

cudaError_t launch_wait_timeout_selftest(uint64_t limit_ns, cudaStream_t stream) {
  wait_timeout_selftest_kernel<<<1, 32, 0, stream>>>(limit_ns);
  return cudaGetLastError();
}

cudaError_t bf16_read_and_clear_status(unsigned* value) {
  cudaError_t e = cudaMemcpyFromSymbol(value, g_moa_bf16_status, sizeof(unsigned));
  if (e != cudaSuccess) return e;
  const unsigned zero = 0;
  return cudaMemcpyToSymbol(g_moa_bf16_status, &zero, sizeof(unsigned));
}

}  // namespace moa
