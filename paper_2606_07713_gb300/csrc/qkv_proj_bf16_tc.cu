// Fused input projections on the fifth-generation tensor cores (tcgen05 + TMEM + TMA), sm_103a.
//
// What it computes (paper Section 4.1): Q = X W_Q, K = X W_K, V = X W_V for one input X
// [B, N, d] and the three weight matrices side by side in W [d, 2 H d_k + H d_v] (row-major,
// columns W_Q | W_K | W_V; column h*d_k + j of W_Q gives feature j of head h).  One GEMM
// C = X W over all B*N tokens reads X once for all three products, and its epilogue stores
// every 32-column chunk of C directly at its place in the head-major Q, K, V arrays
// [B, H, N, d] that the attention entry points read: no [B, N, 3, H, d] intermediate and no
// permute copy exists.
//
// Tiling: persistent CTAs (one per SM) walk the 128-token x 256-column tiles of C; d in steps
// of 64 through a 4-stage TMA ring (X tile 128 x 64 K-major, W tile 64 x 256 MN-major: the
// weights are read as stored).  Two 256-column TMEM accumulators alternate between tiles, so the
// epilogue of one tile overlaps the main loop of the next.  Warps: 0 TMA, 1 TMEM allocation +
// MMA issue, 2-5 epilogue (warp w owns TMEM lanes 32*(w%4): the 128 token rows).  Waits are
// bounded (status word g_moa_proj_status).
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdio>

#include "internal.h"
#include "ptx.cuh"
#include "tc_common.cuh"

namespace moa {

__device__ unsigned int g_moa_proj_status = 0;

namespace {

using namespace ptx;
using namespace tc;

constexpr int kBM = 128;        // tokens per tile (= TMEM lanes)
constexpr int kBN = 256;        // output columns per tile (= TMEM columns per accumulator)
constexpr int kBK = 64;         // model features per stage (one 128-byte swizzle panel of X)
constexpr int kStages = 4;
constexpr int kAccs = 2;        // TMEM accumulators (2 x 256 = 512 columns)
constexpr int kThreads = 192;
constexpr int kLoadWarp = 0;
constexpr int kMmaWarp = 1;
constexpr int kEpiThreads = 128;
constexpr int kXBytes = kBM * kBK * 2;       // 16 KB: 128 rows x 128 B
constexpr int kWPanelBytes = kBK * 64 * 2;   // 8 KB: 64 rows x 64 columns
constexpr int kWBytes = (kBN / 64) * kWPanelBytes;
constexpr int kStageBytes = kXBytes + kWBytes;
constexpr int kOffBar = kStages * kStageBytes;
// full[NS], empty[NS], acc_full[2], acc_empty[2], drain
constexpr int kNumBars = 2 * kStages + 2 * kAccs + 1;
constexpr int kOffMisc = kOffBar + kNumBars * 8;
constexpr int kSmemBytes = kOffMisc + 16 + 1024;
static_assert(kSmemBytes <= 232448, "shared memory budget");

struct ProjDims {
  int N;        // tokens per batch entry (rows of one head's Q/K/V)
  int M;        // B * N
  int H, dk, dv;
  int ncol;     // 2 H dk + H dv
  int n_ktiles; // ceil(d / 64)
  int n_ntiles; // ceil(ncol / 256)
};

__global__ void __launch_bounds__(kThreads, 1)
qkv_proj_bf16_tc_kernel(const __grid_constant__ CUtensorMap tmX,
                        const __grid_constant__ CUtensorMap tmW, __nv_bfloat16* __restrict__ Q,
                        __nv_bfloat16* __restrict__ K, __nv_bfloat16* __restrict__ V, ProjDims p,
                        int n_tiles, uint64_t wait_limit_ns) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar0 = smem_u32(smem + kOffBar);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (kStages + s); };
  auto acc_full = [&](int a) { return bar0 + 8u * (2 * kStages + a); };
  auto acc_empty = [&](int a) { return bar0 + 8u * (2 * kStages + kAccs + a); };
  const uint32_t drain = bar0 + 8u * (2 * kStages + 2 * kAccs);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + kOffMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + kOffMisc + 4);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const WaitCtl wc{abort_flag, wait_limit_ns, 0u, &g_moa_proj_status};
  // Tile t -> (token block t / n_ntiles, column block t % n_ntiles): CTAs running together
  // share X tiles (and the small W) through L2.

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int a = 0; a < kAccs; ++a) {
      mbar_init(acc_full(a), 1);
      mbar_init(acc_empty(a), kEpiThreads);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(smem_u32(tmem_slot), kAccs * kBN);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  if (warp == kLoadWarp) {
    if (lane == 0) {
      tma_prefetch_desc(&tmX);
      tma_prefetch_desc(&tmW);
      int slot = 0;
      uint32_t phase = 0, issued = 0, issued_phase = 0;
      bool ok = true;
      for (int t = blockIdx.x; ok && t < n_tiles; t += gridDim.x) {
        const int m0 = (t / p.n_ntiles) * kBM, c0 = (t % p.n_ntiles) * kBN;
        for (int kt = 0; kt < p.n_ktiles; ++kt) {
          if (!wait_bounded(empty_bar(slot), phase ^ 1u, wc)) {
            ok = false;
            break;
          }
          issued |= 1u << slot;
          issued_phase = (issued_phase & ~(1u << slot)) | (phase << slot);
          const uint32_t st = sbase + slot * kStageBytes;
          mbar_arrive_expect_tx(full_bar(slot), kStageBytes);
          // X: columns [kt*64, +64) of rows [m0, +128); W: rows [kt*64, +64), columns [c0, +256)
          // as four 64-column panels (rows past M or d and columns past ncol read as 0)
          tma_load_3d(st, &tmX, full_bar(slot), kt * kBK, m0, 0);
#pragma unroll
          for (int q = 0; q < kBN / 64; ++q)
            tma_load_3d(st + kXBytes + q * kWPanelBytes, &tmW, full_bar(slot), c0 + 64 * q,
                        kt * kBK, 0);
          if (++slot == kStages) {
            slot = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok || *abort_flag)
        for (int sl = 0; sl < kStages; ++sl)
          if (issued & (1u << sl))
            wait_quiesce(full_bar(sl), (issued_phase >> sl) & 1u, wait_limit_ns, &g_moa_proj_status);
    }
  } else if (warp == kMmaWarp) {
    if (lane == 0) {
      // C (+)= X W: M = 128 tokens, N = 256 columns, K = 16 per MMA.  A = X tile K-major (32 B
      // per step inside the 128-byte panel).  B = W tile MN-major: groups of 8 rows 1024 B
      // apart (stride byte offset), 64-column panels kWPanelBytes apart (leading byte offset),
      // 16 rows = 2048 B per step.
      constexpr uint32_t kIdesc = make_idesc(kBM, kBN, true);
      int slot = 0;
      uint32_t phase = 0;
      bool ok = true;
      int it = 0;
      for (int t = blockIdx.x; ok && t < n_tiles; t += gridDim.x, ++it) {
        const int a = it & 1;
        const uint32_t tacc = tmem + a * kBN;
        // the epilogue has drained this accumulator (its use before last)
        ok = wait_bounded(acc_empty(a), (uint32_t(it >> 1) & 1u) ^ 1u, wc);
        if (!ok) break;
        tc_fence_after_sync();
        for (int kt = 0; kt < p.n_ktiles; ++kt) {
          ok = wait_bounded(full_bar(slot), phase, wc);
          if (!ok) break;
          tc_fence_after_sync();
          const uint32_t st = sbase + slot * kStageBytes;
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk)
            mma_f16_ss(tacc, make_sdesc_sw128(st + kk * 32, 16, 1024),
                       make_sdesc_sw128(st + kXBytes + kk * 2048, kWPanelBytes, 1024), kIdesc,
                       (kt > 0 || kk > 0) ? 1u : 0u);
          mma_commit(empty_bar(slot));
          if (++slot == kStages) {
            slot = 0;
            phase ^= 1u;
          }
        }
        if (ok) mma_commit(acc_full(a));
      }
      mma_commit(drain);  // TMEM quiescent before it is freed, also on the abort path
    }
  } else {
    // Epilogue: token row m0 + r; every 32-column chunk of C goes to one head row of Q, K or V.
    const int lane_base = (warp & 3) * 32;
    const int r = lane_base + lane;
    const int hq = p.H * p.dk;
    int it = 0;
    for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++it) {
      const int a = it & 1;
      if (!wait_bounded(acc_full(a), uint32_t(it >> 1) & 1u, wc)) break;
      tc_fence_after_sync();
      const int m = (t / p.n_ntiles) * kBM + r, c0 = (t % p.n_ntiles) * kBN;
      const bool row_ok = m < p.M;
      const int b = row_ok ? m / p.N : 0, n = row_ok ? m % p.N : 0;
#pragma unroll 2
      for (int c = 0; c < kBN; c += 32) {
        uint32_t o[32];
        tmem_ld_32x32b_x32(tmem + (uint32_t(lane_base) << 16) + a * kBN + c, o);
        tmem_wait_ld();
        reg_anchor_x32(o);
        const int col = c0 + c;
        if (!row_ok || col >= p.ncol) continue;
        __nv_bfloat16* dst;
        if (col < hq) {
          dst = Q + ((size_t(b) * p.H + col / p.dk) * p.N + n) * p.dk + col % p.dk;
        } else if (col < 2 * hq) {
          const int cc = col - hq;
          dst = K + ((size_t(b) * p.H + cc / p.dk) * p.N + n) * p.dk + cc % p.dk;
        } else {
          const int cc = col - 2 * hq;
          dst = V + ((size_t(b) * p.H + cc / p.dv) * p.N + n) * p.dv + cc % p.dv;
        }
        uint4 pkt[4];
        uint32_t* w = reinterpret_cast<uint32_t*>(pkt);
#pragma unroll
        for (int i = 0; i < 16; ++i)
          w[i] = pack_bf16x2(__uint_as_float(o[2 * i]), __uint_as_float(o[2 * i + 1]));
        uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
        for (int i = 0; i < 4; ++i) d4[i] = pkt[i];
      }
      // this accumulator may now take the tile after next
      tc_fence_before_sync();
      mbar_arrive(acc_empty(a));
    }
  }

  if (warp == kMmaWarp) wait_quiesce(drain, 0, wait_limit_ns, &g_moa_proj_status);
  tc_fence_before_sync();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, kAccs * kBN);
  }
}


}  // namespace

int launch_qkv_proj_bf16(const ProjArgs& a, char* msg, size_t msglen) {
  cudaError_t attr_err =
      ensure_smem_limit(reinterpret_cast<const void*>(qkv_proj_bf16_tc_kernel), kSmemBytes);
  if (attr_err != cudaSuccess) {
    snprintf(msg, msglen, "cudaFuncSetAttribute (projection): %s", cudaGetErrorString(attr_err));
    return 5;
  }
  ProjDims p;
  p.N = int(a.N);
  p.M = int(a.B * a.N);
  p.H = int(a.H);
  p.dk = int(a.dk);
  p.dv = int(a.dv);
  p.ncol = int(2 * a.H * a.dk + a.H * a.dv);
  p.n_ktiles = int((a.d + kBK - 1) / kBK);
  p.n_ntiles = (p.ncol + kBN - 1) / kBN;
  const int64_t n_mtiles = (int64_t(p.M) + kBM - 1) / kBM;
  const int64_t n_tiles = n_mtiles * p.n_ntiles;
  int sm_count = 0;
  cudaError_t se = device_sm_count(&sm_count);
  if (se != cudaSuccess) {
    snprintf(msg, msglen, "projection: SM count: %s", cudaGetErrorString(se));
    return 5;
  }
  CUtensorMap mx, mw;
  // X as [1, M, d] (box 64 x 128 rows); W as [1, d, ncol] (box 64 columns x 64 rows)
  if (!encode_bf16_map_box(&mx, a.X, 1, p.M, a.d, 128, msg, msglen)) return 5;
  if (!encode_bf16_map_box(&mw, a.W, 1, a.d, p.ncol, 64, msg, msglen)) return 5;
  const int grid = int(n_tiles < sm_count ? n_tiles : sm_count);
  if (n_tiles > 0x7fffffffLL) {
    snprintf(msg, msglen, "projection: too many tiles");
    return 3;
  }
  qkv_proj_bf16_tc_kernel<<<dim3(unsigned(grid)), dim3(kThreads), kSmemBytes, a.stream>>>(
      mx, mw, static_cast<__nv_bfloat16*>(a.Q), static_cast<__nv_bfloat16*>(a.K),
      static_cast<__nv_bfloat16*>(a.V), p, int(n_tiles), wait_limit_ns());
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    snprintf(msg, msglen, "projection launch: %s", cudaGetErrorString(e));
    return 5;
  }
  return 0;
}

cudaError_t proj_read_and_clear_status(unsigned* value) {
  cudaError_t e = cudaMemcpyFromSymbol(value, g_moa_proj_status, sizeof(unsigned));
  if (e != cudaSuccess) return e;
  const unsigned zero = 0;
  return cudaMemcpyToSymbol(g_moa_proj_status, &zero, sizeof(unsigned));
}

}  // namespace moa
