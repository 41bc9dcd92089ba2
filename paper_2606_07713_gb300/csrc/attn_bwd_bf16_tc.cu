// bf16 attention backward on the fifth-generation tensor cores (tcgen05 + TMEM + TMA), sm_103a.
//
// What it computes (paper Stage 5, Section 9): for O = softmax(scale * Q K^T) V and a given
// dO = dL/dO, the gradients
//     dV = W^T dO,   dS = W * (dO V^T - D),   dQ = scale * dS K,   dK = scale * dS^T Q,
// with W the attention weights and D_i = sum_c dO_ic O_ic = sum_k W_ik (dO V^T)_ik, which is
// the softmax Jacobian (diag(w) - w w^T) applied row by row without ever forming it.  As in the
// forward pass, no N_q x N_k array (scores, weights, dP, dS) exists in global memory: the
// weights are rebuilt tile by tile from the scores and the forward pass's per-row log-sum-exp,
// W_ik = exp2(c * s_ik - LSE_i * log2 e), c = scale * log2 e.
//
// Three kernels:
//   attn_bwd_pre_kernel   per query row: D_i and -LSE_i * log2 e into a padded fp32 workspace
//                         (rows past N_q get D = 0 and -inf, so padded queries weigh nothing);
//   attn_bwd_dkdv_kernel  one CTA per (b, h, block of 128 keys); streams every 128-row query
//                         block through a shared-memory ring and accumulates dV and dK in TMEM:
//                           S^T = K Q^T, dP^T = V dO^T            (TMEM, fp32)
//                           P^T = exp2(c S^T - L), dS^T = P^T (dP^T - D)   (registers, per key row)
//                           dV += P^T dO,  dK += dS^T Q           (A operand from TMEM, bf16)
//   attn_bwd_dq_kernel    one CTA per (b, h, block of 128 query rows); streams the key blocks:
//                           S = Q K^T, dP = dO V^T, dS = P (dP - D), dQ += dS K.
// Splitting dQ from dK/dV keeps every accumulation inside one CTA (no atomics, deterministic
// results) at the price of computing S and dP twice: 7 tile products per (query, key) block
// pair instead of 5.
//
// CTA organisation of both tile kernels (one CTA per SM: 512 TMEM columns):
//   warps 0..4P-1: 128 rows x P column parts (P = 4 for d_k + d_v = 128, else 2).  Warp w owns
//              TMEM lanes 32*(w%4).. (its rows) and columns [(128/P)*(w/4), +128/P) of the
//              128-wide score tiles; it writes its bf16 P or dS back into the first half of those
//              columns, so the parts never overwrite each other's unread values (part_col gives
//              the products' operand columns).
//   warp 4P:   TMEM allocation and the single thread that issues every tcgen05.mma;
//   warp 4P+1: the single thread that issues every TMA copy.
// Every mbarrier wait is bounded; on expiry the kernel records MOA_ERR_DEVICE_TIMEOUT in
// g_moa_bwd_status, every role leaves its loop, and TMEM is still freed.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdio>

#include "internal.h"
#include "ptx.cuh"
#include "tc_common.cuh"

namespace moa {

__device__ unsigned int g_moa_bwd_status = 0;

namespace {

using namespace ptx;
using namespace tc;

constexpr int kBlk = 128;          // rows of every tile (= TMEM lanes) and keys per key block

// Shared-memory loads by 32-bit shared address.  The kernels realign their dynamic shared memory
// with integer arithmetic, after which a pointer no longer tells the compiler that the data live
// in shared memory, and it may emit generic loads, which take the global-memory path.  Explicit
// shared loads of the per-row vectors made the dK/dV kernel up to 4 % faster (8x8x1024x4096,
// d_k = 128, d_v = 64); in the fused kernel they were 1 % slower, so it keeps its pointers.
__device__ __forceinline__ float4 lds_f32x4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}

// Compute-warp layout: P parts of the 128-wide tiles per TMEM lane quarter, 4P compute warps,
// then the MMA warp and the TMA warp.  P = 4 (four warps per scheduler) where the tile products
// are short (d_k + d_v = 128) and the exponentials dominate; P = 2 otherwise.
template <int P>
struct Warps {
  static constexpr int kParts = P;
  static constexpr int kCols = kBlk / P;             // fp32 columns per compute thread
  static constexpr int kComputeWarps = 4 * P;
  static constexpr int kComputeThreads = 32 * kComputeWarps;
  static constexpr int kThreads = kComputeThreads + 64;
  static constexpr int kMmaWarp = kComputeWarps;     // also allocates and frees TMEM
  static constexpr int kLoadWarp = kComputeWarps + 1;
};
__host__ __device__ constexpr int bwd_parts(int dk, int dv) { return dk + dv <= 128 ? 4 : 2; }
constexpr int kTmemCols = 512;
constexpr int kPanelBytes = 128 * 128;  // one 128-byte-swizzle panel: 64 bf16 columns x 128 rows
constexpr int kVecBytes = kBlk * 4;     // 128 fp32 per-row values
constexpr float kLog2e = 1.4426950408889634f;

__host__ __device__ constexpr int ring_stages(int dk, int dv) {
  return dk + dv <= 128 ? 4 : (dk + dv <= 192 ? 3 : 2);
}

// TMEM column of K-step kk (16 rows of the reduction axis) of a bf16 operand written by the
// column parts: part p packs its COLS values into the first COLS/2 columns of its own range
// [p*COLS, +COLS), so the 16 rows of step kk sit at column (16kk/COLS)*COLS + (16kk%COLS)/2.
template <int COLS>
__device__ __forceinline__ uint32_t part_col(int kk) {
  return uint32_t((kk * 16 / COLS) * COLS + (kk * 16 % COLS) / 2);
}

// Loads COLS fp32 TMEM columns of this thread's lane and waits.
template <int COLS>
__device__ __forceinline__ void tmem_load_part(uint32_t taddr, uint32_t* r) {
#pragma unroll
  for (int c = 0; c < COLS; c += 32) tmem_ld_32x32b_x32(taddr + c, r + c);
  tmem_wait_ld();
#pragma unroll
  for (int c = 0; c < COLS; c += 32) reg_anchor_x32(r + c);
}

// Stores COLS/2 packed bf16 pairs to this thread's lane.
template <int COLS>
__device__ __forceinline__ void tmem_store_part(uint32_t taddr, const uint32_t* pk) {
  if constexpr (COLS == 64)
    tmem_st_32x32b_x32(taddr, pk);
  else
    tmem_st_32x32b_x16(taddr, pk);
}

// Writes ncols fp32 TMEM columns of this thread's lane, times mul, as bf16 to dst (16-B aligned).
template <int NCOLS>
__device__ __forceinline__ void store_row_bf16(uint32_t taddr, float mul, __nv_bfloat16* dst,
                                               bool valid) {
#pragma unroll
  for (int c = 0; c < NCOLS; c += 32) {
    uint32_t o[32];
    tmem_ld_32x32b_x32(taddr + c, o);
    tmem_wait_ld();
    reg_anchor_x32(o);
    if (valid) {
      uint4 pkt[4];
      uint32_t* w = reinterpret_cast<uint32_t*>(pkt);
#pragma unroll
      for (int i = 0; i < 16; ++i)
        w[i] = pack_bf16x2(__uint_as_float(o[2 * i]) * mul, __uint_as_float(o[2 * i + 1]) * mul);
      uint4* d4 = reinterpret_cast<uint4*>(dst + c);
#pragma unroll
      for (int i = 0; i < 4; ++i) d4[i] = pkt[i];
    }
  }
}

// ------------------------------------------------------------------------------------------
// Per-row preprocessing
// ------------------------------------------------------------------------------------------
// One group of G = DV/8 lanes per padded query row r = bh * Nq_pad + i (one 16-byte load of O
// and of dO per lane, 32/G rows per warp):
//   Dd[r] = sum_c dO[bh,i,c] * O[bh,i,c] (fp32 products of the bf16 values),
//   nL[r] = -LSE[bh,i] * log2 e;  rows i >= N_q: Dd = 0, nL = -inf;
// and, for the fused kernel (ZERO_COLS > 0), zeros the row's ZERO_COLS fp32 dQ accumulators.
template <int DV, int ZERO_COLS = 0>
__global__ void __launch_bounds__(256)
attn_bwd_pre_kernel(const __nv_bfloat16* __restrict__ O, const __nv_bfloat16* __restrict__ dO,
                    const float* __restrict__ lse, float* __restrict__ nL, float* __restrict__ Dd,
                    int Nq, int Nq_pad, long long rows_pad, float* __restrict__ dq_acc = nullptr) {
  constexpr int G = DV / 8;      // lanes per row: 8 bf16 (16 bytes) per lane
  constexpr int kRows = 32 / G;  // rows per warp
  const int lane = threadIdx.x & 31;
  const long long r = ((long long)blockIdx.x * 8 + (threadIdx.x >> 5)) * kRows + lane / G;
  const int gl = lane % G;
  const bool in_range = r < rows_pad;
  const long long bh = in_range ? r / Nq_pad : 0;
  const int i = in_range ? int(r % Nq_pad) : 0;
  const bool real = in_range && i < Nq;
  const long long src = bh * Nq + i;
  float acc = 0.f;
  if (real) {
    const uint4 ov = *reinterpret_cast<const uint4*>(O + src * DV + gl * 8);
    const uint4 gv = *reinterpret_cast<const uint4*>(dO + src * DV + gl * 8);
    const __nv_bfloat162* o2 = reinterpret_cast<const __nv_bfloat162*>(&ov);
    const __nv_bfloat162* g2 = reinterpret_cast<const __nv_bfloat162*>(&gv);
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const float2 of = __bfloat1622float2(o2[t]), gf = __bfloat1622float2(g2[t]);
      acc = fmaf(of.x, gf.x, acc);
      acc = fmaf(of.y, gf.y, acc);
    }
  }
  // sum over the G lanes of the row (all 32 lanes take part in every shuffle)
#pragma unroll
  for (int off = G / 2; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
  if (in_range && gl == 0) {
    nL[r] = real ? -lse[src] * kLog2e : -INFINITY;
    Dd[r] = real ? acc : 0.f;
  }
  if constexpr (ZERO_COLS > 0) {
    static_assert(ZERO_COLS % (4 * G) == 0, "accumulator row split");
    if (in_range) {
      float4* z = reinterpret_cast<float4*>(dq_acc + r * ZERO_COLS + gl * (ZERO_COLS / G));
#pragma unroll
      for (int t = 0; t < ZERO_COLS / G / 4; ++t) z[t] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
}

// ------------------------------------------------------------------------------------------
// dK and dV: one CTA per (b, h, 128-key block)
// ------------------------------------------------------------------------------------------
template <int DK, int DV>
struct DkDvCfg : Warps<bwd_parts(DK, DV)> {
  static_assert((DK == 64 || DK == 128) && (DV == 64 || DV == 128), "d_k, d_v in {64, 128}");
  static constexpr int kKBytes = kBlk * DK * 2;
  static constexpr int kVBytes = kBlk * DV * 2;
  static constexpr int kQBytes = kBlk * DK * 2;
  static constexpr int kDOBytes = kBlk * DV * 2;
  // stage: Q tile, dO tile, -L (log2 units) and D of its 128 rows; a multiple of 1024 bytes
  static constexpr int kStageBytes = kQBytes + kDOBytes + 2 * kVecBytes;
  static constexpr int kStages = ring_stages(DK, DV);
  static constexpr int kOffK = 0;
  static constexpr int kOffV = kKBytes;
  static constexpr int kOffStage = kKBytes + kVBytes;
  // barriers: full[NS], empty[NS], kv_full, s_full, dp_full, p_ready, ds_ready, acc_done
  static constexpr int kNumBars = 2 * kStages + 6;
  static constexpr int kOffBar = kOffStage + kStages * kStageBytes;
  static constexpr int kOffMisc = kOffBar + kNumBars * 8;
  static constexpr int kSmemBytes = kOffMisc + 16 + 1024;
  static constexpr uint32_t kTmemS = 0, kTmemDP = 128, kTmemDV = 256, kTmemDK = 256 + DV;
  static_assert(kStageBytes % 1024 == 0, "stage alignment");
  static_assert(kTmemDK + DK <= kTmemCols, "TMEM budget");
  static_assert(kSmemBytes <= 232448, "shared memory budget");
};

template <int DK, int DV>
__global__ void __launch_bounds__(DkDvCfg<DK, DV>::kThreads, 1)
attn_bwd_dkdv_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                     const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmDO,
                     const float* __restrict__ nL, const float* __restrict__ Dd,
                     __nv_bfloat16* __restrict__ dK, __nv_bfloat16* __restrict__ dV, int Nk,
                     int Nq_pad, int n_kblocks, float c_log2, float scale, uint64_t wait_limit_ns) {
  using C = DkDvCfg<DK, DV>;
  constexpr int kParts = C::kParts, kCols = C::kCols, kComputeThreads = C::kComputeThreads;
  constexpr int kMmaWarp = C::kMmaWarp, kLoadWarp = C::kLoadWarp;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const uint32_t sK = smem_u32(smem + C::kOffK);
  const uint32_t sV = smem_u32(smem + C::kOffV);
  const uint32_t sStage = smem_u32(smem + C::kOffStage);
  const uint32_t bar0 = smem_u32(smem + C::kOffBar);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (C::kStages + s); };
  const uint32_t kv_full = bar0 + 8u * (2 * C::kStages);
  const uint32_t s_full = kv_full + 8, dp_full = kv_full + 16, p_ready = kv_full + 24;
  const uint32_t ds_ready = kv_full + 32, acc_done = kv_full + 40;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::kOffMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::kOffMisc + 4);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int bh = blockIdx.x / n_kblocks;
  const int k0 = (blockIdx.x % n_kblocks) * kBlk;
  const int n_qb = Nq_pad / kBlk;
  const WaitCtl wc{abort_flag, wait_limit_ns, 0u, &g_moa_bwd_status};

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(kv_full, 1);
    mbar_init(s_full, 1);
    mbar_init(dp_full, 1);
    mbar_init(p_ready, kComputeThreads);
    mbar_init(ds_ready, kComputeThreads);
    mbar_init(acc_done, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  if (warp == kLoadWarp) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      tma_prefetch_desc(&tmDO);
      mbar_arrive_expect_tx(kv_full, C::kKBytes + C::kVBytes);
#pragma unroll
      for (int p = 0; p < DK / 64; ++p)
        tma_load_3d(sK + p * kPanelBytes, &tmK, kv_full, p * 64, k0, bh);
#pragma unroll
      for (int p = 0; p < DV / 64; ++p)
        tma_load_3d(sV + p * kPanelBytes, &tmV, kv_full, p * 64, k0, bh);
      int slot = 0;
      uint32_t phase = 0, issued = 0, issued_phase = 0;
      bool aborted = false;
      for (int i = 0; i < n_qb; ++i) {
        if (!wait_bounded(empty_bar(slot), phase ^ 1u, wc)) {
          aborted = true;
          break;
        }
        issued |= 1u << slot;
        issued_phase = (issued_phase & ~(1u << slot)) | (phase << slot);
        const uint32_t st = sStage + slot * C::kStageBytes;
        mbar_arrive_expect_tx(full_bar(slot), C::kStageBytes);
#pragma unroll
        for (int p = 0; p < DK / 64; ++p)
          tma_load_3d(st + p * kPanelBytes, &tmQ, full_bar(slot), p * 64, i * kBlk, bh);
#pragma unroll
        for (int p = 0; p < DV / 64; ++p)
          tma_load_3d(st + C::kQBytes + p * kPanelBytes, &tmDO, full_bar(slot), p * 64, i * kBlk,
                      bh);
        const size_t vrow = size_t(bh) * Nq_pad + size_t(i) * kBlk;
        bulk_load(st + C::kQBytes + C::kDOBytes, nL + vrow, kVecBytes, full_bar(slot));
        bulk_load(st + C::kQBytes + C::kDOBytes + kVecBytes, Dd + vrow, kVecBytes, full_bar(slot));
        if (++slot == C::kStages) {
          slot = 0;
          phase ^= 1u;
        }
      }
      if (aborted || *abort_flag) {
        wait_quiesce(kv_full, 0, wait_limit_ns, &g_moa_bwd_status);
        for (int sl = 0; sl < C::kStages; ++sl)
          if (issued & (1u << sl))
            wait_quiesce(full_bar(sl), (issued_phase >> sl) & 1u, wait_limit_ns, &g_moa_bwd_status);
      }
    }
  } else if (warp == kMmaWarp) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t kIdescS = make_idesc(kBlk, kBlk, false);
      constexpr uint32_t kIdescDV = make_idesc(kBlk, DV, true);
      constexpr uint32_t kIdescDK = make_idesc(kBlk, DK, true);
      const uint32_t tS = tmem + C::kTmemS, tDP = tmem + C::kTmemDP;
      const uint32_t tDV = tmem + C::kTmemDV, tDK = tmem + C::kTmemDK;
      int slot = 0;
      uint32_t phase = 0;
      // S^T = K Q^T: M = 128 keys, N = 128 queries, both operands K-major (d_k contiguous);
      // reduction step kk is panel kk/4, 32 bytes further per step inside it.
      auto issue_s = [&](uint32_t sQ) {
#pragma unroll
        for (int kk = 0; kk < DK / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kPanelBytes + (kk & 3) * 32;
          mma_f16_ss(tS, make_sdesc_sw128(sK + off, 16, 1024), make_sdesc_sw128(sQ + off, 16, 1024),
                     kIdescS, kk > 0 ? 1u : 0u);
        }
        mma_commit(s_full);
      };
      // dP^T = V dO^T: M = 128 keys, N = 128 queries, reduction over d_v.
      auto issue_dp = [&](uint32_t sDO) {
#pragma unroll
        for (int kk = 0; kk < DV / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kPanelBytes + (kk & 3) * 32;
          mma_f16_ss(tDP, make_sdesc_sw128(sV + off, 16, 1024), make_sdesc_sw128(sDO + off, 16, 1024),
                     kIdescS, kk > 0 ? 1u : 0u);
        }
        mma_commit(dp_full);
      };
      auto stage = [&](int st) { return sStage + st * C::kStageBytes; };
      // Issue order S(0) dP(0) | dV(0) S(1) dK(0) dP(1) | dV(1) S(2) dK(1) dP(2) | ...: the scores
      // of block i+1 are ready when the compute warps finish dS of block i, and the tensor pipe
      // works on dK(i) and dP(i+1) while they form P(i+1).  S(i+1) overwrites the columns of
      // P^T(i) only after dV(i), and dP(i+1) those of dS^T(i) only after dK(i), both issued
      // earlier (tensor-core operations of one CTA complete in issue order).
      bool ok = wait_bounded(kv_full, 0, wc) && wait_bounded(full_bar(0), 0, wc);
      if (ok) {
        tc_fence_after_sync();
        issue_s(stage(0));
        issue_dp(stage(0) + C::kQBytes);
      }
      for (int i = 0; ok && i < n_qb; ++i) {
        const int st = slot;
        if (++slot == C::kStages) {
          slot = 0;
          phase ^= 1u;
        }
        const uint32_t sQ = stage(st), sDO = sQ + C::kQBytes;
        const uint32_t par = uint32_t(i) & 1u;
        // dV += P^T dO: A = P^T (bf16, TMEM), B = dO tile MN-major (d_v contiguous): groups of 8
        // query rows 1024 B apart, 64-column panels kPanelBytes apart.
        ok = wait_bounded(p_ready, par, wc);
        if (!ok) break;
        tc_fence_after_sync();
#pragma unroll
        for (int kk = 0; kk < kBlk / 16; ++kk)
          mma_f16_ts(tDV, tS + part_col<kCols>(kk),
                     make_sdesc_sw128(sDO + kk * 2048, kPanelBytes, 1024), kIdescDV,
                     (kk > 0 || i > 0) ? 1u : 0u);
        const bool more = i + 1 < n_qb;
        if (more) {
          ok = wait_bounded(full_bar(slot), phase, wc);
          if (!ok) break;
          tc_fence_after_sync();
          issue_s(stage(slot));
        }
        // dK += dS^T Q (scale applied in the epilogue): B = Q tile MN-major.
        ok = wait_bounded(ds_ready, par, wc);
        if (!ok) break;
        tc_fence_after_sync();
#pragma unroll
        for (int kk = 0; kk < kBlk / 16; ++kk)
          mma_f16_ts(tDK, tDP + part_col<kCols>(kk),
                     make_sdesc_sw128(sQ + kk * 2048, kPanelBytes, 1024), kIdescDK,
                     (kk > 0 || i > 0) ? 1u : 0u);
        mma_commit(empty_bar(st));
        if (more) issue_dp(stage(slot) + C::kQBytes);
      }
      // Always signal once everything issued has completed, so that TMEM is quiescent before
      // it is freed even on the abort path.
      mma_commit(acc_done);
    }
  } else {
    // ---------------------------------------------------------------- compute warps
    const int part = warp >> 2;              // column part of the 128-query tiles
    const int lane_base = (warp & 3) * 32;   // TMEM lanes (key rows) of this warp
    const int row = lane_base + lane;        // key row inside the block
    const uint32_t lanes = uint32_t(lane_base) << 16;
    const uint32_t tS = tmem + lanes + C::kTmemS + part * kCols;
    const uint32_t tDP = tmem + lanes + C::kTmemDP + part * kCols;
    const uint64_t cc = pack_f32x2(c_log2, c_log2);
    int slot = 0;
    uint32_t phase = 0;
    bool ok = true;
    for (int i = 0; i < n_qb; ++i) {
      const int st = slot;
      const uint32_t par = uint32_t(i) & 1u;
      // The stage's -L and D came with the tiles (TMA); waiting on its full barrier makes
      // them visible to this thread.
      ok = wait_bounded(full_bar(st), phase, wc) && wait_bounded(s_full, par, wc);
      if (++slot == C::kStages) {
        slot = 0;
        phase ^= 1u;
      }
      if (!ok) break;
      tc_fence_after_sync();
      // this stage's -L and D of the 128 queries: this part's kCols of each
      const uint32_t nl4 = sStage + st * C::kStageBytes + C::kQBytes + C::kDOBytes + part * kCols * 4;
      const uint32_t d4 = nl4 + kBlk * 4;
      uint32_t r[kCols];
      tmem_load_part<kCols>(tS, r);
      float p[kCols];
#pragma unroll
      for (int q = 0; q < kCols; q += 4) {
        const float4 l = lds_f32x4(nl4 + q * 4);
        ffma2(p[q], p[q + 1], __uint_as_float(r[q]), __uint_as_float(r[q + 1]), cc,
              pack_f32x2(l.x, l.y));
        ffma2(p[q + 2], p[q + 3], __uint_as_float(r[q + 2]), __uint_as_float(r[q + 3]), cc,
              pack_f32x2(l.z, l.w));
      }
      uint32_t pk[kCols / 2];
#pragma unroll
      for (int q = 0; q < kCols; q += 2) {
        p[q] = ex2_approx(p[q]);
        p[q + 1] = ex2_approx(p[q + 1]);
        pk[q >> 1] = pack_bf16x2(p[q], p[q + 1]);
      }
      tmem_store_part<kCols>(tS, pk);
      tmem_wait_st();
      tc_fence_before_sync();
      mbar_arrive(p_ready);
      ok = wait_bounded(dp_full, par, wc);
      if (!ok) break;
      tc_fence_after_sync();
      tmem_load_part<kCols>(tDP, r);
#pragma unroll
      for (int q = 0; q < kCols; q += 4) {
        const float4 d = lds_f32x4(d4 + q * 4);
        const float s0 = p[q] * (__uint_as_float(r[q]) - d.x);
        const float s1 = p[q + 1] * (__uint_as_float(r[q + 1]) - d.y);
        const float s2 = p[q + 2] * (__uint_as_float(r[q + 2]) - d.z);
        const float s3 = p[q + 3] * (__uint_as_float(r[q + 3]) - d.w);
        pk[q >> 1] = pack_bf16x2(s0, s1);
        pk[(q >> 1) + 1] = pack_bf16x2(s2, s3);
      }
      tmem_store_part<kCols>(tDP, pk);
      tmem_wait_st();
      tc_fence_before_sync();
      mbar_arrive(ds_ready);
    }
    // Epilogue: the first half of the parts write dV, the second half scale * dK, each part a
    // slice of the columns (rows past N_k are not stored).
    if (ok && wait_bounded(acc_done, 0, wc)) {
      tc_fence_after_sync();
      const bool valid = k0 + row < Nk;
      const size_t grow = size_t(bh) * Nk + size_t(k0 + row);
      constexpr int kHalf = kParts / 2;
      if (part < kHalf) {
        constexpr int w = DV / kHalf;
        store_row_bf16<w>(tmem + lanes + C::kTmemDV + part * w, 1.0f, dV + grow * DV + part * w,
                          valid);
      } else {
        constexpr int w = DK / kHalf;
        const int q = part - kHalf;
        store_row_bf16<w>(tmem + lanes + C::kTmemDK + q * w, scale, dK + grow * DK + q * w, valid);
      }
    }
  }

  if (warp == kMmaWarp) wait_quiesce(acc_done, 0, wait_limit_ns, &g_moa_bwd_status);
  tc_fence_before_sync();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ------------------------------------------------------------------------------------------
// dQ: one CTA per (b, h, 128-row query block)
// ------------------------------------------------------------------------------------------
template <int DK, int DV>
struct DqCfg : Warps<bwd_parts(DK, DV)> {
  static_assert((DK == 64 || DK == 128) && (DV == 64 || DV == 128), "d_k, d_v in {64, 128}");
  static constexpr int kQBytes = kBlk * DK * 2;
  static constexpr int kDOBytes = kBlk * DV * 2;
  static constexpr int kKBytes = kBlk * DK * 2;
  static constexpr int kVBytes = kBlk * DV * 2;
  static constexpr int kStageBytes = kKBytes + kVBytes;  // K tile, V tile
  static constexpr int kStages = ring_stages(DK, DV);
  static constexpr int kOffQ = 0;
  static constexpr int kOffDO = kQBytes;
  static constexpr int kOffStage = kQBytes + kDOBytes;
  // barriers: full[NS], empty[NS], q_full, s_full, dp_full, ds_ready, acc_done, s_free
  static constexpr int kNumBars = 2 * kStages + 6;
  static constexpr int kOffBar = kOffStage + kStages * kStageBytes;
  static constexpr int kOffMisc = kOffBar + kNumBars * 8;
  static constexpr int kSmemBytes = kOffMisc + 16 + 1024;
  static constexpr uint32_t kTmemS = 0, kTmemDP = 128, kTmemDQ = 256;
  static_assert(kTmemDQ + DK <= kTmemCols, "TMEM budget");
  static_assert(kSmemBytes <= 232448, "shared memory budget");
};

template <int DK, int DV>
__global__ void __launch_bounds__(DqCfg<DK, DV>::kThreads, 1)
attn_bwd_dq_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                   const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmDO,
                   const float* __restrict__ nL, const float* __restrict__ Dd,
                   __nv_bfloat16* __restrict__ dQ, int Nq, int Nk, int Nq_pad, int n_qblocks,
                   float c_log2, float scale, uint64_t wait_limit_ns) {
  using C = DqCfg<DK, DV>;
  constexpr int kCols = C::kCols, kComputeThreads = C::kComputeThreads;
  constexpr int kMmaWarp = C::kMmaWarp, kLoadWarp = C::kLoadWarp;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const uint32_t sQ = smem_u32(smem + C::kOffQ);
  const uint32_t sDO = smem_u32(smem + C::kOffDO);
  const uint32_t sStage = smem_u32(smem + C::kOffStage);
  const uint32_t bar0 = smem_u32(smem + C::kOffBar);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (C::kStages + s); };
  const uint32_t q_full = bar0 + 8u * (2 * C::kStages);
  const uint32_t s_full = q_full + 8, dp_full = q_full + 16, ds_ready = q_full + 24;
  const uint32_t acc_done = q_full + 32, s_free = q_full + 40;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::kOffMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::kOffMisc + 4);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int bh = blockIdx.x / n_qblocks;
  const int q0 = (blockIdx.x % n_qblocks) * kBlk;
  const int n_kb = (Nk + kBlk - 1) / kBlk;
  const WaitCtl wc{abort_flag, wait_limit_ns, 0u, &g_moa_bwd_status};

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(q_full, 1);
    mbar_init(s_full, 1);
    mbar_init(dp_full, 1);
    mbar_init(ds_ready, kComputeThreads);
    mbar_init(acc_done, 1);
    mbar_init(s_free, kComputeThreads);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  if (warp == kLoadWarp) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      tma_prefetch_desc(&tmDO);
      mbar_arrive_expect_tx(q_full, C::kQBytes + C::kDOBytes);
#pragma unroll
      for (int p = 0; p < DK / 64; ++p)
        tma_load_3d(sQ + p * kPanelBytes, &tmQ, q_full, p * 64, q0, bh);
#pragma unroll
      for (int p = 0; p < DV / 64; ++p)
        tma_load_3d(sDO + p * kPanelBytes, &tmDO, q_full, p * 64, q0, bh);
      int slot = 0;
      uint32_t phase = 0, issued = 0, issued_phase = 0;
      bool aborted = false;
      for (int j = 0; j < n_kb; ++j) {
        if (!wait_bounded(empty_bar(slot), phase ^ 1u, wc)) {
          aborted = true;
          break;
        }
        issued |= 1u << slot;
        issued_phase = (issued_phase & ~(1u << slot)) | (phase << slot);
        const uint32_t st = sStage + slot * C::kStageBytes;
        mbar_arrive_expect_tx(full_bar(slot), C::kStageBytes);
#pragma unroll
        for (int p = 0; p < DK / 64; ++p)
          tma_load_3d(st + p * kPanelBytes, &tmK, full_bar(slot), p * 64, j * kBlk, bh);
#pragma unroll
        for (int p = 0; p < DV / 64; ++p)
          tma_load_3d(st + C::kKBytes + p * kPanelBytes, &tmV, full_bar(slot), p * 64, j * kBlk,
                      bh);
        if (++slot == C::kStages) {
          slot = 0;
          phase ^= 1u;
        }
      }
      if (aborted || *abort_flag) {
        wait_quiesce(q_full, 0, wait_limit_ns, &g_moa_bwd_status);
        for (int sl = 0; sl < C::kStages; ++sl)
          if (issued & (1u << sl))
            wait_quiesce(full_bar(sl), (issued_phase >> sl) & 1u, wait_limit_ns, &g_moa_bwd_status);
      }
    }
  } else if (warp == kMmaWarp) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t kIdescS = make_idesc(kBlk, kBlk, false);
      constexpr uint32_t kIdescDQ = make_idesc(kBlk, DK, true);
      const uint32_t tS = tmem + C::kTmemS, tDP = tmem + C::kTmemDP, tDQ = tmem + C::kTmemDQ;
      int slot = 0;
      uint32_t phase = 0;
      auto stage = [&](int st) { return sStage + st * C::kStageBytes; };
      // S = Q K^T (M = 128 queries, N = 128 keys, K-major operands)
      auto issue_s = [&](uint32_t sK) {
#pragma unroll
        for (int kk = 0; kk < DK / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kPanelBytes + (kk & 3) * 32;
          mma_f16_ss(tS, make_sdesc_sw128(sQ + off, 16, 1024), make_sdesc_sw128(sK + off, 16, 1024),
                     kIdescS, kk > 0 ? 1u : 0u);
        }
        mma_commit(s_full);
      };
      // dP = dO V^T (reduction over d_v)
      auto issue_dp = [&](uint32_t sV) {
#pragma unroll
        for (int kk = 0; kk < DV / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kPanelBytes + (kk & 3) * 32;
          mma_f16_ss(tDP, make_sdesc_sw128(sDO + off, 16, 1024), make_sdesc_sw128(sV + off, 16, 1024),
                     kIdescS, kk > 0 ? 1u : 0u);
        }
        mma_commit(dp_full);
      };
      // Issue order S(0) dP(0) | S(1) dQ(0) dP(1) | S(2) dQ(1) dP(2) | ...: S(j+1) goes as soon as
      // the compute warps hold S(j) in registers (s_free), so they find it ready after dS(j);
      // dP(j+1) overwrites the columns of dS(j) only after dQ(j), issued earlier.
      bool ok = wait_bounded(q_full, 0, wc) && wait_bounded(full_bar(0), 0, wc);
      if (ok) {
        tc_fence_after_sync();
        issue_s(stage(0));
        issue_dp(stage(0) + C::kKBytes);
      }
      for (int j = 0; ok && j < n_kb; ++j) {
        const int st = slot;
        if (++slot == C::kStages) {
          slot = 0;
          phase ^= 1u;
        }
        const uint32_t par = uint32_t(j) & 1u;
        const bool more = j + 1 < n_kb;
        if (more) {
          ok = wait_bounded(full_bar(slot), phase, wc) && wait_bounded(s_free, par, wc);
          if (!ok) break;
          tc_fence_after_sync();
          issue_s(stage(slot));
        }
        // dQ += dS K (scale applied in the epilogue): A = dS (bf16, TMEM), B = K tile MN-major.
        ok = wait_bounded(ds_ready, par, wc);
        if (!ok) break;
        tc_fence_after_sync();
        const uint32_t sK = stage(st);
#pragma unroll
        for (int kk = 0; kk < kBlk / 16; ++kk)
          mma_f16_ts(tDQ, tDP + part_col<kCols>(kk),
                     make_sdesc_sw128(sK + kk * 2048, kPanelBytes, 1024), kIdescDQ,
                     (kk > 0 || j > 0) ? 1u : 0u);
        mma_commit(empty_bar(st));
        if (more) issue_dp(stage(slot) + C::kKBytes);
      }
      mma_commit(acc_done);
    }
  } else {
    // ---------------------------------------------------------------- compute warps
    const int part = warp >> 2;              // column part of the 128-key tiles
    const int lane_base = (warp & 3) * 32;   // TMEM lanes (query rows) of this warp
    const int row = lane_base + lane;
    const uint32_t lanes = uint32_t(lane_base) << 16;
    const uint32_t tS = tmem + lanes + C::kTmemS + part * kCols;
    const uint32_t tDP = tmem + lanes + C::kTmemDP + part * kCols;
    const size_t vrow = size_t(bh) * Nq_pad + size_t(q0 + row);  // padded: always in range
    const float nl = nL[vrow], dd = Dd[vrow];
    const uint64_t cc = pack_f32x2(c_log2, c_log2);
    const uint64_t nn = pack_f32x2(nl, nl);
    bool ok = true;
    for (int j = 0; j < n_kb; ++j) {
      const uint32_t par = uint32_t(j) & 1u;
      ok = wait_bounded(s_full, par, wc);
      if (!ok) break;
      tc_fence_after_sync();
      uint32_t r[kCols];
      tmem_load_part<kCols>(tS, r);
      // S(j) is in registers: the issuer may write S(j+1) over it
      tc_fence_before_sync();
      mbar_arrive(s_free);
      float p[kCols];
#pragma unroll
      for (int k = 0; k < kCols; k += 2) {
        ffma2(p[k], p[k + 1], __uint_as_float(r[k]), __uint_as_float(r[k + 1]), cc, nn);
        p[k] = ex2_approx(p[k]);
        p[k + 1] = ex2_approx(p[k + 1]);
      }
      ok = wait_bounded(dp_full, par, wc);
      if (!ok) break;
      tc_fence_after_sync();
      tmem_load_part<kCols>(tDP, r);
      uint32_t pk[kCols / 2];
#pragma unroll
      for (int k = 0; k < kCols; k += 2)
        pk[k >> 1] = pack_bf16x2(p[k] * (__uint_as_float(r[k]) - dd),
                                 p[k + 1] * (__uint_as_float(r[k + 1]) - dd));
      tmem_store_part<kCols>(tDP, pk);
      tmem_wait_st();
      tc_fence_before_sync();
      mbar_arrive(ds_ready);
    }
    // Epilogue: scale * dQ -> bf16; part p < DK/w writes columns [w*p, w*p + w),
    // w = max(32, DK / parts).
    constexpr int w = DK / C::kParts > 32 ? DK / C::kParts : 32;
    if (ok && wait_bounded(acc_done, 0, wc) && part < DK / w) {
      tc_fence_after_sync();
      const bool valid = q0 + row < Nq;
      __nv_bfloat16* dst = dQ + (size_t(bh) * Nq + size_t(valid ? q0 + row : 0)) * DK + part * w;
      store_row_bf16<w>(tmem + lanes + C::kTmemDQ + part * w, scale, dst, valid);
    }
  }

  if (warp == kMmaWarp) wait_quiesce(acc_done, 0, wait_limit_ns, &g_moa_bwd_status);
  tc_fence_before_sync();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, kTmemCols);
  }
}


// ------------------------------------------------------------------------------------------
// dK, dV and dQ in one kernel (d_k = d_v = 64): one CTA per (b, h, 128-key block)
// ------------------------------------------------------------------------------------------
// The dK/dV kernel's schedule plus the query gradient of the same tiles: dS^T of every query
// block goes to shared memory (bf16, key rows, query columns contiguous, 128-byte swizzle),
// where it is both the A operand of dK += dS^T Q (K-major) and, read transposed, the A operand
// of dQ_i = dS_i K (MN-major), so S and dP are formed once per tile pair (5 products, not 7).
// dQ_i lands in one of two TMEM buffers; the compute warps copy it into a shared-memory tile
// (fp32, 128-byte swizzle) and a reduction warp adds that tile to an fp32 accumulator in global
// memory with TMA reductions (cp.reduce.async.bulk.tensor ... add), while the tensor core works
// on the next query block.  The order of the key blocks' additions varies from run to run, so
// dQ may differ in its last bits between runs; dK and dV are accumulated in one CTA each and
// are reproducible.
template <int DK, int DV>
struct FusedCfg : Warps<4> {
  static_assert(DK == 64 && DV == 64, "fused backward: d_k = d_v = 64");
  // warps: 16 compute, MMA, TMA loads, TMA reductions of dQ
  static constexpr int kReduceWarp = Warps<4>::kComputeWarps + 2;
  static constexpr int kThreads = Warps<4>::kComputeThreads + 96;
  static constexpr int kKBytes = kBlk * DK * 2;
  static constexpr int kVBytes = kBlk * DV * 2;
  static constexpr int kQBytes = kBlk * DK * 2;
  static constexpr int kDOBytes = kBlk * DV * 2;
  static constexpr int kStageBytes = kQBytes + kDOBytes + 2 * kVecBytes;
  static constexpr int kStages = 3;
  static constexpr int kDSBytes = 2 * kPanelBytes;  // 128 key rows x 128 queries, bf16
  static constexpr int kDQBytes = kBlk * DK * 4;    // staged dQ tile: 2 boxes of 32 fp32 columns
  static constexpr int kDQBoxBytes = kBlk * 128;
  static constexpr int kOffK = 0;
  static constexpr int kOffV = kKBytes;
  static constexpr int kOffStage = kKBytes + kVBytes;
  static constexpr int kOffDS = kOffStage + kStages * kStageBytes;
  static constexpr int kOffDQ = kOffDS + kDSBytes;
  // barriers: full[NS], empty[NS], kv_full, s_full, dp_full, p_ready, ds_ready, acc_done,
  //           ds_free, dq_full[2], dq_free[2], stg_full, stg_free
  static constexpr int kNumBars = 2 * kStages + 13;
  static constexpr int kOffBar = kOffDQ + kDQBytes;
  static constexpr int kOffMisc = kOffBar + kNumBars * 8;
  static constexpr int kSmemBytes = kOffMisc + 16 + 1024;
  static constexpr uint32_t kTmemS = 0, kTmemDP = 128, kTmemDV = 256, kTmemDK = 256 + DV;
  static constexpr uint32_t kTmemDQ0 = kTmemDK + DK, kTmemDQ1 = kTmemDQ0 + DK;
  static_assert(kStageBytes % 1024 == 0 && kOffDS % 1024 == 0 && kOffDQ % 1024 == 0,
                "stage alignment");
  static_assert(kTmemDQ1 + DK <= kTmemCols, "TMEM budget");
  static_assert(kSmemBytes <= 232448, "shared memory budget");
};

template <int DK, int DV>
__global__ void __launch_bounds__(FusedCfg<DK, DV>::kThreads, 1)
attn_bwd_fused_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                      const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmDO,
                      const __grid_constant__ CUtensorMap tmDQ, const float* __restrict__ nL,
                      const float* __restrict__ Dd, __nv_bfloat16* __restrict__ dK,
                      __nv_bfloat16* __restrict__ dV, int Nk, int Nq_pad, int n_kblocks,
                      float c_log2, float scale, uint64_t wait_limit_ns) {
  using C = FusedCfg<DK, DV>;
  constexpr int kParts = C::kParts, kCols = C::kCols, kComputeThreads = C::kComputeThreads;
  constexpr int kMmaWarp = C::kMmaWarp, kLoadWarp = C::kLoadWarp;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const uint32_t sK = smem_u32(smem + C::kOffK);
  const uint32_t sV = smem_u32(smem + C::kOffV);
  const uint32_t sStage = smem_u32(smem + C::kOffStage);
  const uint32_t sDS = smem_u32(smem + C::kOffDS);
  const uint32_t sDQ = smem_u32(smem + C::kOffDQ);
  const uint32_t bar0 = smem_u32(smem + C::kOffBar);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (C::kStages + s); };
  const uint32_t kv_full = bar0 + 8u * (2 * C::kStages);
  const uint32_t s_full = kv_full + 8, dp_full = kv_full + 16, p_ready = kv_full + 24;
  const uint32_t ds_ready = kv_full + 32, acc_done = kv_full + 40, ds_free = kv_full + 48;
  auto dq_full = [&](int b) { return kv_full + 56 + 8u * b; };
  auto dq_free = [&](int b) { return kv_full + 72 + 8u * b; };
  const uint32_t stg_full = kv_full + 88, stg_free = kv_full + 96;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::kOffMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::kOffMisc + 4);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int bh = blockIdx.x / n_kblocks;
  const int k0 = (blockIdx.x % n_kblocks) * kBlk;
  const int n_qb = Nq_pad / kBlk;
  const WaitCtl wc{abort_flag, wait_limit_ns, 0u, &g_moa_bwd_status};

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(kv_full, 1);
    mbar_init(s_full, 1);
    mbar_init(dp_full, 1);
    mbar_init(p_ready, kComputeThreads);
    mbar_init(ds_ready, kComputeThreads);
    mbar_init(acc_done, 1);
    mbar_init(ds_free, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(dq_full(b), 1);
      mbar_init(dq_free(b), kComputeThreads);
    }
    mbar_init(stg_full, kComputeThreads);
    mbar_init(stg_free, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  if (warp == C::kReduceWarp) {
    // ---------------------------------------------------------------- dQ reductions
    // Block j's staged dQ tile is added to the accumulator rows of query block j once every
    // compute thread has written its part; the tile is free again once the TMA has read it.
    if (lane == 0) {
      tma_prefetch_desc(&tmDQ);
      for (int j = 0; j < n_qb; ++j) {
        if (!wait_bounded(stg_full, uint32_t(j) & 1u, wc)) break;
        tma_reduce_add_3d(&tmDQ, sDQ, 0, j * kBlk, bh);
        tma_reduce_add_3d(&tmDQ, sDQ + C::kDQBoxBytes, 32, j * kBlk, bh);
        bulk_commit_group();
        bulk_wait_group_read_all();
        mbar_arrive(stg_free);
      }
      bulk_wait_group_all();
    }
  } else if (warp == kLoadWarp) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      tma_prefetch_desc(&tmDO);
      mbar_arrive_expect_tx(kv_full, C::kKBytes + C::kVBytes);
      tma_load_3d(sK, &tmK, kv_full, 0, k0, bh);
      tma_load_3d(sV, &tmV, kv_full, 0, k0, bh);
      int slot = 0;
      uint32_t phase = 0, issued = 0, issued_phase = 0;
      bool aborted = false;
      for (int i = 0; i < n_qb; ++i) {
        if (!wait_bounded(empty_bar(slot), phase ^ 1u, wc)) {
          aborted = true;
          break;
        }
        issued |= 1u << slot;
        issued_phase = (issued_phase & ~(1u << slot)) | (phase << slot);
        const uint32_t st = sStage + slot * C::kStageBytes;
        mbar_arrive_expect_tx(full_bar(slot), C::kStageBytes);
        tma_load_3d(st, &tmQ, full_bar(slot), 0, i * kBlk, bh);
        tma_load_3d(st + C::kQBytes, &tmDO, full_bar(slot), 0, i * kBlk, bh);
        const size_t vrow = size_t(bh) * Nq_pad + size_t(i) * kBlk;
        bulk_load(st + C::kQBytes + C::kDOBytes, nL + vrow, kVecBytes, full_bar(slot));
        bulk_load(st + C::kQBytes + C::kDOBytes + kVecBytes, Dd + vrow, kVecBytes, full_bar(slot));
        if (++slot == C::kStages) {
          slot = 0;
          phase ^= 1u;
        }
      }
      if (aborted || *abort_flag) {
        wait_quiesce(kv_full, 0, wait_limit_ns, &g_moa_bwd_status);
        for (int sl = 0; sl < C::kStages; ++sl)
          if (issued & (1u << sl))
            wait_quiesce(full_bar(sl), (issued_phase >> sl) & 1u, wait_limit_ns, &g_moa_bwd_status);
      }
    }
  } else if (warp == kMmaWarp) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t kIdescS = make_idesc(kBlk, kBlk, false);
      constexpr uint32_t kIdescDV = make_idesc(kBlk, DV, true);
      constexpr uint32_t kIdescDK = make_idesc(kBlk, DK, true);
      constexpr uint32_t kIdescDQ = make_idesc_a_mn(kBlk, DK, true);
      const uint32_t tS = tmem + C::kTmemS, tDP = tmem + C::kTmemDP;
      const uint32_t tDV = tmem + C::kTmemDV, tDK = tmem + C::kTmemDK;
      int slot = 0;
      uint32_t phase = 0;
      auto issue_s = [&](uint32_t sQ) {  // S^T = K Q^T (both K-major)
#pragma unroll
        for (int kk = 0; kk < DK / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kPanelBytes + (kk & 3) * 32;
          mma_f16_ss(tS, make_sdesc_sw128(sK + off, 16, 1024), make_sdesc_sw128(sQ + off, 16, 1024),
                     kIdescS, kk > 0 ? 1u : 0u);
        }
        mma_commit(s_full);
      };
      auto issue_dp = [&](uint32_t sDO) {  // dP^T = V dO^T
#pragma unroll
        for (int kk = 0; kk < DV / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kPanelBytes + (kk & 3) * 32;
          mma_f16_ss(tDP, make_sdesc_sw128(sV + off, 16, 1024), make_sdesc_sw128(sDO + off, 16, 1024),
                     kIdescS, kk > 0 ? 1u : 0u);
        }
        mma_commit(dp_full);
      };
      auto stage = [&](int st) { return sStage + st * C::kStageBytes; };
      // Issue order S(0) dP(0) | dV(0) S(1) dK(0) dP(1) dQ(0) | dV(1) S(2) dK(1) dP(2) dQ(1) | ...
      bool ok = wait_bounded(kv_full, 0, wc) && wait_bounded(full_bar(0), 0, wc);
      if (ok) {
        tc_fence_after_sync();
        issue_s(stage(0));
        issue_dp(stage(0) + C::kQBytes);
      }
      for (int i = 0; ok && i < n_qb; ++i) {
        const int st = slot;
        if (++slot == C::kStages) {
          slot = 0;
          phase ^= 1u;
        }
        const uint32_t sQ = stage(st), sDO = sQ + C::kQBytes;
        const uint32_t par = uint32_t(i) & 1u;
        // dV += P^T dO: A = P^T (bf16, TMEM), B = dO tile MN-major.
        ok = wait_bounded(p_ready, par, wc);
        if (!ok) break;
        tc_fence_after_sync();
#pragma unroll
        for (int kk = 0; kk < kBlk / 16; ++kk)
          mma_f16_ts(tDV, tS + part_col<kCols>(kk),
                     make_sdesc_sw128(sDO + kk * 2048, kPanelBytes, 1024), kIdescDV,
                     (kk > 0 || i > 0) ? 1u : 0u);
        const bool more = i + 1 < n_qb;
        if (more) {
          ok = wait_bounded(full_bar(slot), phase, wc);
          if (!ok) break;
          tc_fence_after_sync();
          issue_s(stage(slot));
        }
        // dK += dS^T Q: A = dS^T in shared memory (K-major: queries contiguous), B = Q MN-major.
        ok = wait_bounded(ds_ready, par, wc);
        if (!ok) break;
        tc_fence_after_sync();
#pragma unroll
        for (int kk = 0; kk < kBlk / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kPanelBytes + (kk & 3) * 32;
          mma_f16_ss(tDK, make_sdesc_sw128(sDS + off, 16, 1024),
                     make_sdesc_sw128(sQ + kk * 2048, kPanelBytes, 1024), kIdescDK,
                     (kk > 0 || i > 0) ? 1u : 0u);
        }
        // dP(i+1) before dQ(i): the compute warps wait for it next.
        if (more) issue_dp(stage(slot) + C::kQBytes);
        // dQ_i = dS K into TMEM buffer i % 2 (free once the compute warps read dQ_{i-2}):
        // A = the same dS^T tile read MN-major (query rows contiguous: 16 keys per step,
        // 64-query panels kPanelBytes apart), B = K tile MN-major.
        const int b = i & 1;
        if (i >= 2) {
          ok = wait_bounded(dq_free(b), uint32_t((i >> 1) - 1) & 1u, wc);
          if (!ok) break;
          tc_fence_after_sync();
        }
        const uint32_t tDQ = tmem + (b ? C::kTmemDQ1 : C::kTmemDQ0);
#pragma unroll
        for (int kk = 0; kk < kBlk / 16; ++kk)
          mma_f16_ss(tDQ, make_sdesc_sw128(sDS + kk * 2048, kPanelBytes, 1024),
                     make_sdesc_sw128(sK + kk * 2048, kPanelBytes, 1024), kIdescDQ,
                     kk > 0 ? 1u : 0u);
        mma_commit(dq_full(b));
        mma_commit(ds_free);        // dK(i) and dQ(i) have read dS(i)
        mma_commit(empty_bar(st));  // dV(i) read dO(i), dK(i) read Q(i)
      }
      // Always signal once everything issued has completed, so that TMEM is quiescent before
      // it is freed even on the abort path.
      mma_commit(acc_done);
    }
  } else {
    // ---------------------------------------------------------------- compute warps
    const int part = warp >> 2;              // column part of the 128-query tiles
    const int lane_base = (warp & 3) * 32;   // TMEM lanes (key rows; query rows of dQ)
    const int row = lane_base + lane;
    const uint32_t lanes = uint32_t(lane_base) << 16;
    const uint32_t tS = tmem + lanes + C::kTmemS + part * kCols;
    const uint32_t tDP = tmem + lanes + C::kTmemDP + part * kCols;
    const uint64_t cc = pack_f32x2(c_log2, c_log2);
    // This thread's 64 bytes of dS^T: key row `row`, queries [32 part, +32) = 16-byte chunks
    // 4(part % 2) .. +3 of panel part / 2, placed by the 128-byte swizzle (chunk ^ row % 8).
    uint8_t* ds_row = smem + C::kOffDS + (part >> 1) * kPanelBytes + row * 128;
    const int chunk0 = (part & 1) * 4;
    // dQ columns this thread stages for its query row: [16 part, +16) = 16-byte chunks
    // 4(part % 2) .. +3 of box part / 2 (32 columns, 128 bytes per row), swizzled like dS.
    constexpr int kDqCols = DK / kParts;
    uint8_t* dq_row = smem + C::kOffDQ + (part >> 1) * C::kDQBoxBytes + row * 128;
    auto drain_dq = [&](int j) -> bool {
      const int b = j & 1;
      if (!wait_bounded(dq_full(b), uint32_t(j >> 1) & 1u, wc)) return false;
      tc_fence_after_sync();
      uint32_t q[kDqCols];
      tmem_ld_32x32b_x16(tmem + lanes + (b ? C::kTmemDQ1 : C::kTmemDQ0) + part * kDqCols, q);
      tmem_wait_ld();
      reg_anchor_x16(q);
      tc_fence_before_sync();
      mbar_arrive(dq_free(b));
      // the staging tile is free once the previous block's reductions have read it
      if (j > 0 && !wait_bounded(stg_free, uint32_t(j - 1) & 1u, wc)) return false;
#pragma unroll
      for (int t = 0; t < kDqCols / 4; ++t)
        *reinterpret_cast<uint4*>(dq_row + (((chunk0 + t) ^ (row & 7)) << 4)) =
            make_uint4(q[4 * t], q[4 * t + 1], q[4 * t + 2], q[4 * t + 3]);
      fence_proxy_async_smem();  // the TMA reads the tile through the async proxy
      mbar_arrive(stg_full);
      return true;
    };
    int slot = 0;
    uint32_t phase = 0;
    bool ok = true;
    for (int i = 0; i < n_qb; ++i) {
      const int st = slot;
      const uint32_t par = uint32_t(i) & 1u;
      ok = wait_bounded(full_bar(st), phase, wc) && wait_bounded(s_full, par, wc);
      if (++slot == C::kStages) {
        slot = 0;
        phase ^= 1u;
      }
      if (!ok) break;
      tc_fence_after_sync();
      const float* vec = reinterpret_cast<const float*>(smem + C::kOffStage + st * C::kStageBytes +
                                                        C::kQBytes + C::kDOBytes);
      const float4* nl4 = reinterpret_cast<const float4*>(vec + part * kCols);
      const float4* d4 = reinterpret_cast<const float4*>(vec + kBlk + part * kCols);
      uint32_t r[kCols];
      tmem_load_part<kCols>(tS, r);
      float p[kCols];
#pragma unroll
      for (int q = 0; q < kCols; q += 4) {
        const float4 l = nl4[q >> 2];
        ffma2(p[q], p[q + 1], __uint_as_float(r[q]), __uint_as_float(r[q + 1]), cc,
              pack_f32x2(l.x, l.y));
        ffma2(p[q + 2], p[q + 3], __uint_as_float(r[q + 2]), __uint_as_float(r[q + 3]), cc,
              pack_f32x2(l.z, l.w));
      }
      uint32_t pk[kCols / 2];
#pragma unroll
      for (int q = 0; q < kCols; q += 2) {
        p[q] = ex2_approx(p[q]);
        p[q + 1] = ex2_approx(p[q + 1]);
        pk[q >> 1] = pack_bf16x2(p[q], p[q + 1]);
      }
      tmem_store_part<kCols>(tS, pk);
      tmem_wait_st();
      tc_fence_before_sync();
      mbar_arrive(p_ready);
      ok = wait_bounded(dp_full, par, wc);
      if (!ok) break;
      tc_fence_after_sync();
      // dP^T in two 16-column halves: all 32 columns beside P in registers spill at the
      // 96-register cap of 19 warps.
#pragma unroll
      for (int h = 0; h < kCols; h += 16) {
        tmem_ld_32x32b_x16(tDP + h, r);
        tmem_wait_ld();
        reg_anchor_x16(r);
#pragma unroll
        for (int q = 0; q < 16; q += 4) {
          const float4 d = d4[(h + q) >> 2];
          const float s0 = p[h + q] * (__uint_as_float(r[q]) - d.x);
          const float s1 = p[h + q + 1] * (__uint_as_float(r[q + 1]) - d.y);
          const float s2 = p[h + q + 2] * (__uint_as_float(r[q + 2]) - d.z);
          const float s3 = p[h + q + 3] * (__uint_as_float(r[q + 3]) - d.w);
          pk[(h + q) >> 1] = pack_bf16x2(s0, s1);
          pk[((h + q) >> 1) + 1] = pack_bf16x2(s2, s3);
        }
      }
      // dS(i) overwrites dS(i-1) once dK(i-1) and dQ(i-1) have read it.
      if (i > 0) {
        ok = wait_bounded(ds_free, uint32_t(i - 1) & 1u, wc);
        if (!ok) break;
      }
#pragma unroll
      for (int t = 0; t < 4; ++t)
        *reinterpret_cast<uint4*>(ds_row + (((chunk0 + t) ^ (row & 7)) << 4)) =
            make_uint4(pk[4 * t], pk[4 * t + 1], pk[4 * t + 2], pk[4 * t + 3]);
      fence_proxy_async_smem();  // the tensor core reads dS through the async proxy
      mbar_arrive(ds_ready);
      // The previous block's dQ: TMEM -> fp32 additions into the accumulator.
      if (i > 0 && !drain_dq(i - 1)) {
        ok = false;
        break;
      }
    }
    if (ok && n_qb > 0) ok = drain_dq(n_qb - 1);
    // Epilogue: the first half of the parts write dV, the second half scale * dK.
    if (ok && wait_bounded(acc_done, 0, wc)) {
      tc_fence_after_sync();
      const bool valid = k0 + row < Nk;
      const size_t grow = size_t(bh) * Nk + size_t(k0 + row);
      constexpr int kHalf = kParts / 2;
      if (part < kHalf) {
        constexpr int w = DV / kHalf;
        store_row_bf16<w>(tmem + lanes + C::kTmemDV + part * w, 1.0f, dV + grow * DV + part * w,
                          valid);
      } else {
        constexpr int w = DK / kHalf;
        const int q = part - kHalf;
        store_row_bf16<w>(tmem + lanes + C::kTmemDK + q * w, scale, dK + grow * DK + q * w, valid);
      }
    }
  }

  if (warp == kMmaWarp) wait_quiesce(acc_done, 0, wait_limit_ns, &g_moa_bwd_status);
  tc_fence_before_sync();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// dQ = scale * the fused kernel's fp32 accumulator, as bf16 (rows past N_q are not stored).
// One thread per 8 consecutive values of a row.
template <int DK>
__global__ void __launch_bounds__(256)
attn_bwd_dq_convert_kernel(const float* __restrict__ dq_acc, __nv_bfloat16* __restrict__ dQ,
                           int Nq, int Nq_pad, long long n_items, float scale) {
  const long long t = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= n_items) return;
  constexpr int kPerRow = DK / 8;
  const long long r = t / kPerRow;  // row of the real (unpadded) rows, head-major
  const int c = int(t % kPerRow) * 8;
  const long long bh = r / Nq, i = r % Nq;
  const float4* src = reinterpret_cast<const float4*>(dq_acc + (bh * Nq_pad + i) * DK + c);
  const float4 a = src[0], b = src[1];
  uint4 out;
  out.x = pack_bf16x2(a.x * scale, a.y * scale);
  out.y = pack_bf16x2(a.z * scale, a.w * scale);
  out.z = pack_bf16x2(b.x * scale, b.y * scale);
  out.w = pack_bf16x2(b.z * scale, b.w * scale);
  *reinterpret_cast<uint4*>(dQ + r * DK + c) = out;
}

// ------------------------------------------------------------------------------------------
// Host side
// ------------------------------------------------------------------------------------------
int64_t padded_rows(int64_t Nq) { return (Nq + kBlk - 1) / kBlk * kBlk; }

template <int DK, int DV>
int launch_bwd(const BwdArgs& a, const CUtensorMap& mq, const CUtensorMap& mk,
               const CUtensorMap& mv, const CUtensorMap& mdo, char* msg, size_t msglen) {
  using A = DkDvCfg<DK, DV>;
  using B = DqCfg<DK, DV>;
  cudaError_t attr_err =
      ensure_smem_limit(reinterpret_cast<const void*>(attn_bwd_dkdv_kernel<DK, DV>), A::kSmemBytes);
  if (attr_err == cudaSuccess)
    attr_err =
        ensure_smem_limit(reinterpret_cast<const void*>(attn_bwd_dq_kernel<DK, DV>), B::kSmemBytes);
  if (attr_err != cudaSuccess) {
    snprintf(msg, msglen, "cudaFuncSetAttribute (bf16 backward): %s", cudaGetErrorString(attr_err));
    return 5;
  }
  const int64_t BH = a.B * a.H;
  const int64_t nq_pad = padded_rows(a.Nq);
  const int64_t n_kb = (a.Nk + kBlk - 1) / kBlk, n_qb = nq_pad / kBlk;
  if (BH * n_kb > 0x7fffffffLL || BH * n_qb > 0x7fffffffLL || BH * nq_pad / 8 > 0x7fffffffLL ||
      nq_pad > 0x7fffffffLL) {
    snprintf(msg, msglen, "bf16 backward: grid too large");
    return 3;
  }
  float* nL = static_cast<float*>(a.ws);
  float* Dd = nL + BH * nq_pad;
  const float c_log2 = a.scale * kLog2e;
  const long long rows_pad = BH * nq_pad;
  constexpr int kPreRowsPerBlock = 8 * (32 / (DV / 8));
  attn_bwd_pre_kernel<DV><<<dim3(unsigned((rows_pad + kPreRowsPerBlock - 1) / kPreRowsPerBlock)),
                            dim3(256), 0, a.stream>>>(
      static_cast<const __nv_bfloat16*>(a.O), static_cast<const __nv_bfloat16*>(a.dO), a.lse, nL,
      Dd, int(a.Nq), int(nq_pad), rows_pad);
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) {
    attn_bwd_dkdv_kernel<DK, DV><<<dim3(unsigned(BH * n_kb)), dim3(A::kThreads), A::kSmemBytes,
                                   a.stream>>>(
        mq, mk, mv, mdo, nL, Dd, static_cast<__nv_bfloat16*>(a.dK),
        static_cast<__nv_bfloat16*>(a.dV), int(a.Nk), int(nq_pad), int(n_kb), c_log2, a.scale,
        wait_limit_ns());
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) {
    attn_bwd_dq_kernel<DK, DV><<<dim3(unsigned(BH * n_qb)), dim3(B::kThreads), B::kSmemBytes,
                                 a.stream>>>(mq, mk, mv, mdo, nL, Dd,
                                             static_cast<__nv_bfloat16*>(a.dQ), int(a.Nq),
                                             int(a.Nk), int(nq_pad), int(n_qb), c_log2, a.scale,
                                             wait_limit_ns());
    e = cudaGetLastError();
  }
  if (e != cudaSuccess) {
    snprintf(msg, msglen, "bf16 backward launch: %s", cudaGetErrorString(e));
    return 5;
  }
  return 0;
}

template <int DK, int DV>
int launch_bwd_fused(const BwdArgs& a, const CUtensorMap& mq, const CUtensorMap& mk,
                     const CUtensorMap& mv, const CUtensorMap& mdo, char* msg, size_t msglen) {
  using F = FusedCfg<DK, DV>;
  const cudaError_t attr_err =
      ensure_smem_limit(reinterpret_cast<const void*>(attn_bwd_fused_kernel<DK, DV>), F::kSmemBytes);
  if (attr_err != cudaSuccess) {
    snprintf(msg, msglen, "cudaFuncSetAttribute (fused backward): %s", cudaGetErrorString(attr_err));
    return 5;
  }
  const int64_t BH = a.B * a.H;
  const int64_t nq_pad = padded_rows(a.Nq);
  const int64_t n_kb = (a.Nk + kBlk - 1) / kBlk;
  const long long rows_pad = BH * nq_pad;
  const long long n_conv = BH * a.Nq * (DK / 8);
  if (BH * n_kb > 0x7fffffffLL || rows_pad / 8 > 0x7fffffffLL || nq_pad > 0x7fffffffLL ||
      (n_conv + 255) / 256 > 0x7fffffffLL) {
    snprintf(msg, msglen, "fused backward: grid too large");
    return 3;
  }
  float* nL = static_cast<float*>(a.ws);
  float* Dd = nL + rows_pad;
  float* dq_acc = Dd + rows_pad;  // 16-byte aligned: rows_pad is a multiple of 128
  CUtensorMap mdq;
  if (!encode_f32_map_sw128(&mdq, dq_acc, BH, nq_pad, DK, 32, kBlk, msg, msglen)) return 5;
  const float c_log2 = a.scale * kLog2e;
  constexpr int kPreRowsPerBlock = 8 * (32 / (DV / 8));
  attn_bwd_pre_kernel<DV, DK><<<dim3(unsigned((rows_pad + kPreRowsPerBlock - 1) / kPreRowsPerBlock)),
                                dim3(256), 0, a.stream>>>(
      static_cast<const __nv_bfloat16*>(a.O), static_cast<const __nv_bfloat16*>(a.dO), a.lse, nL,
      Dd, int(a.Nq), int(nq_pad), rows_pad, dq_acc);
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) {
    attn_bwd_fused_kernel<DK, DV><<<dim3(unsigned(BH * n_kb)), dim3(F::kThreads), F::kSmemBytes,
                                    a.stream>>>(
        mq, mk, mv, mdo, mdq, nL, Dd, static_cast<__nv_bfloat16*>(a.dK),
        static_cast<__nv_bfloat16*>(a.dV), int(a.Nk), int(nq_pad), int(n_kb), c_log2, a.scale,
        wait_limit_ns());
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) {
    attn_bwd_dq_convert_kernel<DK><<<dim3(unsigned((n_conv + 255) / 256)), dim3(256), 0,
                                     a.stream>>>(dq_acc, static_cast<__nv_bfloat16*>(a.dQ),
                                                 int(a.Nq), int(nq_pad), n_conv, a.scale);
    e = cudaGetLastError();
  }
  if (e != cudaSuccess) {
    snprintf(msg, msglen, "fused backward launch: %s", cudaGetErrorString(e));
    return 5;
  }
  return 0;
}

}  // namespace

size_t bwd_fused_workspace_bytes(int64_t B, int64_t H, int64_t Nq, int64_t dk) {
  return size_t(B) * size_t(H) * size_t(padded_rows(Nq)) * sizeof(float) * size_t(2 + dk);
}

int launch_attn_bwd_bf16_fused(const BwdArgs& a, char* msg, size_t msglen) {
  if (a.dk != 64 || a.dv != 64) {
    snprintf(msg, msglen, "the fused backward supports d_k = d_v = 64; got d_k=%lld d_v=%lld",
             (long long)a.dk, (long long)a.dv);
    return 3;
  }
  const int64_t BH = a.B * a.H;
  CUtensorMap mq, mk, mv, mdo;
  if (!encode_bf16_map(&mq, a.Q, BH, a.Nq, a.dk, msg, msglen)) return 5;
  if (!encode_bf16_map(&mk, a.K, BH, a.Nk, a.dk, msg, msglen)) return 5;
  if (!encode_bf16_map(&mv, a.V, BH, a.Nk, a.dv, msg, msglen)) return 5;
  if (!encode_bf16_map(&mdo, a.dO, BH, a.Nq, a.dv, msg, msglen)) return 5;
  return launch_bwd_fused<64, 64>(a, mq, mk, mv, mdo, msg, msglen);
}

size_t bwd_workspace_bytes(int64_t B, int64_t H, int64_t Nq) {
  return size_t(2) * size_t(B) * size_t(H) * size_t(padded_rows(Nq)) * sizeof(float);
}

int launch_attn_bwd_bf16(const BwdArgs& a, char* msg, size_t msglen) {
  const int64_t BH = a.B * a.H;
  CUtensorMap mq, mk, mv, mdo;
  if (!encode_bf16_map(&mq, a.Q, BH, a.Nq, a.dk, msg, msglen)) return 5;
  if (!encode_bf16_map(&mk, a.K, BH, a.Nk, a.dk, msg, msglen)) return 5;
  if (!encode_bf16_map(&mv, a.V, BH, a.Nk, a.dv, msg, msglen)) return 5;
  if (!encode_bf16_map(&mdo, a.dO, BH, a.Nq, a.dv, msg, msglen)) return 5;
  if (a.dk == 64 && a.dv == 64) return launch_bwd<64, 64>(a, mq, mk, mv, mdo, msg, msglen);
  if (a.dk == 128 && a.dv == 128) return launch_bwd<128, 128>(a, mq, mk, mv, mdo, msg, msglen);
  if (a.dk == 128 && a.dv == 64) return launch_bwd<128, 64>(a, mq, mk, mv, mdo, msg, msglen);
  if (a.dk == 64 && a.dv == 128) return launch_bwd<64, 128>(a, mq, mk, mv, mdo, msg, msglen);
  snprintf(msg, msglen, "bf16 backward supports d_k, d_v in {64, 128}; got d_k=%lld d_v=%lld",
           (long long)a.dk, (long long)a.dv);
  return 3;
}

cudaError_t bwd_read_and_clear_status(unsigned* value) {
  cudaError_t e = cudaMemcpyFromSymbol(value, g_moa_bwd_status, sizeof(unsigned));
  if (e != cudaSuccess) return e;
  const unsigned zero = 0;
  return cudaMemcpyToSymbol(g_moa_bwd_status, &zero, sizeof(unsigned));
}

}  // namespace moa
