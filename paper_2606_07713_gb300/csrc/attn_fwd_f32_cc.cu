// fp32 attention forward on CUDA cores (no TF32), for the MOA_FP32 element type.
//
// Computes O = softmax(scale * Q K^T) V (paper Section 4.1, Eq. attention) in
// the DNF's memory pattern: one CTA owns BM query rows of one (b, h) slice
// (the independent 2-D problems of the Remark in Section 4.2), streams K and V
// through shared memory in BN-key tiles, and keeps the scores of one tile, the
// running row maximum and the running denominator in registers.  The row max
// (Step I, Section 4.3), the exponentials (Step II, Section 4.4) and their sum
// (Step III, Section 4.5) are combined online: when a tile raises the running
// maximum from m to m', the partial sums are rescaled by exp(m - m'), which is
// the exact identity exp(s - m') = exp(s - m) * exp(m - m').  The division of
// Step IV happens once per row at the end.  Nothing but O is written to global
// memory.
//
// Layout: Q, K, V, O contiguous row-major [B,H,N,d] float32.
// Two kernels:
//   attn_fwd_f32_cc_kernel   CTA of 128 threads = 4 warps, BM = 32 rows (8 per warp), BN = 64
//                            keys; K and V tiles shared by the CTA's 32 rows through smem.
//   attn_fwd_f32_small_kernel  8 query rows of one (b, h) per CTA, one warp per row, for
//                            problems too small to give every SM a 32-row CTA: 64-key chunks of
//                            K and V are copied with cp.async, every piece of a chunk in flight
//                            at once, double-buffered, which matters when the call is bound by
//                            memory latency.
#include <cuda_runtime.h>
#include <math.h>
#include <cstdio>

#include "internal.h"

namespace moa {
namespace {

constexpr int kThreads = 128;
constexpr int kWarps = kThreads / 32;
constexpr int kRowsPerWarp = 8;
constexpr int kBM = kWarps * kRowsPerWarp;  // 32 query rows per CTA
constexpr int kBN = 64;                     // keys per tile
constexpr int kMaxD = 128;
constexpr int kMaxColGroups = kMaxD / 32;    // output columns per lane: c = lane + 32*g

struct F32Smem {
  // K tile padded by one float per row so that lane-strided reads hit distinct banks.
  static size_t bytes(int dk, int dv) {
    return sizeof(float) * (size_t(kBM) * dk + size_t(kBN) * (dk + 1) + size_t(kBN) * dv +
                            size_t(kWarps) * kRowsPerWarp * kBN);
  }
};

__global__ void __launch_bounds__(kThreads)
attn_fwd_f32_cc_kernel(const float* __restrict__ Q, const float* __restrict__ K,
                       const float* __restrict__ V, float* __restrict__ O,
                       float* __restrict__ lse, int Nq, int Nk, int dk, int dv, int n_qtiles,
                       float scale) {
  extern __shared__ float smem[];
  float* sQ = smem;                          // [kBM][dk]
  float* sK = sQ + kBM * dk;                 // [kBN][dk+1]
  float* sV = sK + kBN * (dk + 1);           // [kBN][dv]
  float* sP = sV + kBN * dv;                 // [kWarps][kRowsPerWarp][kBN]
  const int ldk = dk + 1;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const long long bh = blockIdx.x / n_qtiles;
  const int qt = blockIdx.x % n_qtiles;
  const int q0 = qt * kBM;

  const float* Qh = Q + bh * (long long)Nq * dk;
  const float* Kh = K + bh * (long long)Nk * dk;
  const float* Vh = V + bh * (long long)Nk * dv;
  float* Oh = O + bh * (long long)Nq * dv;

  // Q tile -> shared memory (rows past N_q are zero; they are computed but never stored).
  for (int idx = threadIdx.x; idx < kBM * dk; idx += kThreads) {
    const int r = idx / dk, j = idx % dk;
    sQ[idx] = (q0 + r < Nq) ? Qh[(long long)(q0 + r) * dk + j] : 0.f;
  }

  float m[kRowsPerWarp], l[kRowsPerWarp];
  float acc[kRowsPerWarp][kMaxColGroups];
#pragma unroll
  for (int r = 0; r < kRowsPerWarp; ++r) {
    m[r] = -INFINITY;
    l[r] = 0.f;
#pragma unroll
    for (int g = 0; g < kMaxColGroups; ++g) acc[r][g] = 0.f;
  }
  const int ngroups = (dv + 31) / 32;
  float* myP = sP + warp * kRowsPerWarp * kBN;
  const float* myQ = sQ + warp * kRowsPerWarp * dk;

  for (int k0 = 0; k0 < Nk; k0 += kBN) {
    __syncthreads();  // previous tile fully consumed (and Q visible on the first pass)
    for (int idx = threadIdx.x; idx < kBN * dk; idx += kThreads) {
      const int r = idx / dk, j = idx % dk;
      sK[r * ldk + j] = (k0 + r < Nk) ? Kh[(long long)(k0 + r) * dk + j] : 0.f;
    }
    for (int idx = threadIdx.x; idx < kBN * dv; idx += kThreads) {
      const int r = idx / dv;
      sV[idx] = (k0 + r < Nk) ? Vh[(long long)k0 * dv + idx] : 0.f;
    }
    __syncthreads();

    // Scores of this warp's 8 rows against keys (lane) and (lane + 32) of the tile.
    float s0[kRowsPerWarp], s1[kRowsPerWarp];
#pragma unroll
    for (int r = 0; r < kRowsPerWarp; ++r) s0[r] = s1[r] = 0.f;
    const float* k0p = sK + lane * ldk;
    const float* k1p = sK + (lane + 32) * ldk;
    for (int j = 0; j < dk; ++j) {
      const float ka = k0p[j], kb = k1p[j];
#pragma unroll
      for (int r = 0; r < kRowsPerWarp; ++r) {
        const float q = myQ[r * dk + j];
        s0[r] = fmaf(q, ka, s0[r]);
        s1[r] = fmaf(q, kb, s1[r]);
      }
    }
    const bool v0 = (k0 + lane) < Nk, v1 = (k0 + lane + 32) < Nk;
    float alpha[kRowsPerWarp];
#pragma unroll
    for (int r = 0; r < kRowsPerWarp; ++r) {
      const float x0 = v0 ? s0[r] * scale : -INFINITY;
      const float x1 = v1 ? s1[r] * scale : -INFINITY;
      float tmax = fmaxf(x0, x1);
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, off));
      const float mnew = fmaxf(m[r], tmax);   // finite: every tile has at least one key
      alpha[r] = expf(m[r] - mnew);           // exp(-inf) = 0 on the first tile
      const float p0 = expf(x0 - mnew), p1 = expf(x1 - mnew);
      float psum = p0 + p1;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) psum += __shfl_xor_sync(0xffffffffu, psum, off);
      l[r] = l[r] * alpha[r] + psum;
      m[r] = mnew;
      myP[r * kBN + lane] = p0;
      myP[r * kBN + lane + 32] = p1;
    }
    __syncwarp();
    // acc = alpha * acc + P V for this warp's rows and this lane's output columns.
#pragma unroll
    for (int r = 0; r < kRowsPerWarp; ++r)
#pragma unroll
      for (int g = 0; g < kMaxColGroups; ++g) acc[r][g] *= alpha[r];
    const int kn = min(kBN, Nk - k0);
    for (int kk = 0; kk < kn; ++kk) {
      float vv[kMaxColGroups];
#pragma unroll
      for (int g = 0; g < kMaxColGroups; ++g) {
        const int c = lane + 32 * g;
        vv[g] = (g < ngroups && c < dv) ? sV[kk * dv + c] : 0.f;
      }
#pragma unroll
      for (int r = 0; r < kRowsPerWarp; ++r) {
        const float p = myP[r * kBN + kk];
#pragma unroll
        for (int g = 0; g < kMaxColGroups; ++g) acc[r][g] = fmaf(p, vv[g], acc[r][g]);
      }
    }
    __syncwarp();
  }

#pragma unroll
  for (int r = 0; r < kRowsPerWarp; ++r) {
    const int row = q0 + warp * kRowsPerWarp + r;
    if (row >= Nq) continue;
    const float inv = 1.0f / l[r];
    // ln sum_k exp(scale s_k) = m + ln l (m is the exact row maximum here).
    if (lse != nullptr && lane == 0) lse[bh * Nq + row] = m[r] + logf(l[r]);
#pragma unroll
    for (int g = 0; g < kMaxColGroups; ++g) {
      const int c = lane + 32 * g;
      if (g < ngroups && c < dv) Oh[(long long)row * dv + c] = acc[r][g] * inv;
    }
  }
}

// Small problems: 8 query rows of one (b, h) per CTA, one warp per row.  The CTA's 256
// threads copy 64-key chunks of K and V into shared memory with cp.async (16-byte pieces, all
// in flight at once), double-buffered: chunk c+1 is requested before chunk c is used, so a call
// that is bound by memory latency pays it about once per chunk pair instead of once per
// dependent load.  Per chunk, lane = key for the scores (keys lane and lane + 32), lane =
// output column for the sum over V.
constexpr int kSmallRows = 8;     // rows (= warps) per CTA
constexpr int kSmallKeys = 64;    // keys per chunk
constexpr int kSmallThreads = 32 * kSmallRows;

struct SmallSmem {
  // K rows padded by 4 floats: 16-byte aligned, and the float4 reads of 8 consecutive key rows
  // fall on disjoint banks.
  __host__ __device__ static int ldk(int dk) { return dk + 4; }
  static size_t bytes(int dk, int dv) {
    return sizeof(float) * (size_t(kSmallRows) * dk + 2 * size_t(kSmallKeys) * ldk(dk) +
                            2 * size_t(kSmallKeys) * dv + size_t(kSmallRows) * kSmallKeys);
  }
};

// 16 bytes global -> shared, asynchronous; src_bytes = 0 writes zeros (the source is not read).
__device__ __forceinline__ void cp_async16(float* dst, const float* src, int src_bytes) {
  const unsigned d = static_cast<unsigned>(__cvta_generic_to_shared(dst));
  const size_t g = __cvta_generic_to_global(src);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(g), "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__global__ void __launch_bounds__(kSmallThreads)
attn_fwd_f32_small_kernel(const float* __restrict__ Q, const float* __restrict__ K,
                          const float* __restrict__ V, float* __restrict__ O,
                          float* __restrict__ lse, int Nq, int Nk, int dk, int dv, int n_qtiles,
                          float scale) {
  extern __shared__ __align__(16) float smem[];
  const int ldk = SmallSmem::ldk(dk);
  float* sQ = smem;                                   // [8][dk]
  float* sK = sQ + kSmallRows * dk;                   // [2][64][dk + 4]
  float* sV = sK + 2 * kSmallKeys * ldk;              // [2][64][dv]
  float* sP = sV + 2 * kSmallKeys * dv;               // [8][64]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long bh = blockIdx.x / n_qtiles;
  const int row = (blockIdx.x % n_qtiles) * kSmallRows + warp;  // query row of this warp
  const bool active = row < Nq;
  const float* Kh = K + bh * (long long)Nk * dk;
  const float* Vh = V + bh * (long long)Nk * dv;

  const int kseg = dk / 4, vseg = dv / 4;  // 16-byte pieces per row (d is a multiple of 4)
  auto request = [&](int c) {             // chunk c -> buffer c % 2
    const int k0 = c * kSmallKeys, b = c & 1;
    float* dK = sK + b * kSmallKeys * ldk;
    float* dV = sV + b * kSmallKeys * dv;
    for (int i = threadIdx.x; i < kSmallKeys * kseg; i += kSmallThreads) {
      const int r = i / kseg, j = i - r * kseg;
      const bool in = k0 + r < Nk;
      cp_async16(dK + r * ldk + 4 * j, in ? Kh + (long long)(k0 + r) * dk + 4 * j : Kh, in ? 16 : 0);
    }
    for (int i = threadIdx.x; i < kSmallKeys * vseg; i += kSmallThreads) {
      const int r = i / vseg, j = i - r * vseg;
      const bool in = k0 + r < Nk;
      cp_async16(dV + r * dv + 4 * j, in ? Vh + (long long)(k0 + r) * dv + 4 * j : Vh, in ? 16 : 0);
    }
    cp_async_commit();
  };

  request(0);
  if (active)
    for (int j = lane; j < dk; j += 32) sQ[warp * dk + j] = Q[(bh * Nq + row) * (long long)dk + j];
  const float* q = sQ + warp * dk;
  float* p_row = sP + warp * kSmallKeys;

  float m = -INFINITY, l = 0.f;
  float acc[kMaxColGroups];
#pragma unroll
  for (int g = 0; g < kMaxColGroups; ++g) acc[g] = 0.f;
  const int n_chunks = (Nk + kSmallKeys - 1) / kSmallKeys;
  for (int c = 0; c < n_chunks; ++c) {
    if (c + 1 < n_chunks) {
      request(c + 1);  // its buffer was released by the barrier at the end of chunk c - 1
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();  // chunk c (and the Q rows) visible to every warp
    if (active) {
      const int k0 = c * kSmallKeys, b = c & 1;
      const float* cK = sK + b * kSmallKeys * ldk;
      const float* cV = sV + b * kSmallKeys * dv;
      // scores of keys k0 + lane and k0 + lane + 32
      const float* ka = cK + lane * ldk;
      const float* kb = cK + (lane + 32) * ldk;
      float s0 = 0.f, s1 = 0.f;
      for (int j = 0; j < dk; j += 4) {
        const float4 qv = *reinterpret_cast<const float4*>(q + j);
        const float4 a4 = *reinterpret_cast<const float4*>(ka + j);
        const float4 b4 = *reinterpret_cast<const float4*>(kb + j);
        s0 = fmaf(qv.x, a4.x, s0);
        s1 = fmaf(qv.x, b4.x, s1);
        s0 = fmaf(qv.y, a4.y, s0);
        s1 = fmaf(qv.y, b4.y, s1);
        s0 = fmaf(qv.z, a4.z, s0);
        s1 = fmaf(qv.z, b4.z, s1);
        s0 = fmaf(qv.w, a4.w, s0);
        s1 = fmaf(qv.w, b4.w, s1);
      }
      const float x0 = k0 + lane < Nk ? s0 * scale : -INFINITY;
      const float x1 = k0 + lane + 32 < Nk ? s1 * scale : -INFINITY;
      float cmax = fmaxf(x0, x1);
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) cmax = fmaxf(cmax, __shfl_xor_sync(0xffffffffu, cmax, off));
      const float mnew = fmaxf(m, cmax);  // finite: every chunk has at least one key
      const float alpha = expf(m - mnew);  // exp(-inf) = 0 on the first chunk
      const float p0 = expf(x0 - mnew), p1 = expf(x1 - mnew);
      float psum = p0 + p1;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) psum += __shfl_xor_sync(0xffffffffu, psum, off);
      l = l * alpha + psum;
      m = mnew;
      p_row[lane] = p0;
      p_row[lane + 32] = p1;
      __syncwarp();
      // lane = output column: acc = alpha * acc + sum over the chunk's keys of p_k V[k, c]
#pragma unroll
      for (int g = 0; g < kMaxColGroups; ++g) acc[g] *= alpha;
      const int kn = min(kSmallKeys, Nk - k0);
      for (int k = 0; k < kn; k += 4) {
        float pv[4], vv[4][kMaxColGroups];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          pv[u] = k + u < kn ? p_row[k + u] : 0.f;  // zero-filled rows past N_k also read 0
#pragma unroll
          for (int g = 0; g < kMaxColGroups; ++g) {
            const int col = lane + 32 * g;
            vv[u][g] = col < dv ? cV[(k + u) * dv + col] : 0.f;
          }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u)
#pragma unroll
          for (int g = 0; g < kMaxColGroups; ++g) acc[g] = fmaf(pv[u], vv[u][g], acc[g]);
      }
    }
    __syncthreads();  // buffer c % 2 and the P rows are free again
  }
  if (active) {
    const float inv = 1.0f / l;
    float* orow = O + (bh * Nq + row) * (long long)dv;
#pragma unroll
    for (int g = 0; g < kMaxColGroups; ++g) {
      const int col = lane + 32 * g;
      if (col < dv) orow[col] = acc[g] * inv;
    }
    // ln sum_k exp(scale s_k) = m + ln l (m is the exact row maximum here)
    if (lse != nullptr && lane == 0) lse[bh * Nq + row] = m + logf(l);
  }
}

}  // namespace

int launch_attn_fwd_f32(const AttnArgs& a, char* msg, size_t msglen) {
  // Few 32-row CTAs (fewer than two per SM): 8-row CTAs instead, each with its K/V chunks
  // requested all at once.
  int dev = 0, sms = 148;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if ((long long)a.B * a.H * ((a.Nq + kBM - 1) / kBM) < 2LL * sms) {
    const int n_qtiles = int((a.Nq + kSmallRows - 1) / kSmallRows);
    const long long grid = (long long)a.B * a.H * n_qtiles;
    if (grid > 0x7fffffffLL) {
      snprintf(msg, msglen, "fp32 path: too many rows");
      return 3;
    }
    const cudaError_t attr_err =
        ensure_smem_limit(reinterpret_cast<const void*>(attn_fwd_f32_small_kernel),
                          int(SmallSmem::bytes(kMaxD, kMaxD)));
    if (attr_err != cudaSuccess) {
      snprintf(msg, msglen, "cudaFuncSetAttribute (fp32 small kernel): %s",
               cudaGetErrorString(attr_err));
      return 5;
    }
    attn_fwd_f32_small_kernel<<<dim3(unsigned(grid)), dim3(kSmallThreads),
                                SmallSmem::bytes(int(a.dk), int(a.dv)), a.stream>>>(
        static_cast<const float*>(a.Q), static_cast<const float*>(a.K),
        static_cast<const float*>(a.V), static_cast<float*>(a.O), a.lse, int(a.Nq), int(a.Nk),
        int(a.dk), int(a.dv), n_qtiles, a.scale);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) {
      snprintf(msg, msglen, "fp32 small kernel launch: %s", cudaGetErrorString(e));
      return 5;
    }
    return 0;
  }
  const int n_qtiles = int((a.Nq + kBM - 1) / kBM);
  const long long grid = (long long)a.B * a.H * n_qtiles;
  if (grid > 0x7fffffffLL) {
    snprintf(msg, msglen, "fp32 path: B*H*ceil(N_q/%d) = %lld CTAs exceeds the grid limit", kBM, grid);
    return 3;
  }
  const size_t smem = F32Smem::bytes(int(a.dk), int(a.dv));
  cudaError_t e = ensure_smem_limit(reinterpret_cast<const void*>(attn_fwd_f32_cc_kernel), int(smem));
  if (e != cudaSuccess) {
    snprintf(msg, msglen, "cudaFuncSetAttribute (fp32 kernel): %s", cudaGetErrorString(e));
    return 5;
  }
  attn_fwd_f32_cc_kernel<<<dim3(unsigned(grid)), dim3(kThreads), smem, a.stream>>>(
      static_cast<const float*>(a.Q), static_cast<const float*>(a.K),
      static_cast<const float*>(a.V), static_cast<float*>(a.O), a.lse, int(a.Nq), int(a.Nk),
      int(a.dk), int(a.dv), n_qtiles, a.scale);
  e = cudaGetLastError();
  if (e != cudaSuccess) {
    snprintf(msg, msglen, "fp32 kernel launch: %s", cudaGetErrorString(e));
    return 5;
  }
  return 0;
}

}  // namespace moa
