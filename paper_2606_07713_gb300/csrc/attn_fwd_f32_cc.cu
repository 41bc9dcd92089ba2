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
// CTA: 128 threads = 4 warps, BM = 32 rows (8 per warp), BN = 64 keys.
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

}  // namespace

int launch_attn_fwd_f32(const AttnArgs& a, char* msg, size_t msglen) {
  const int n_qtiles = int((a.Nq + kBM - 1) / kBM);
  const long long grid = (long long)a.B * a.H * n_qtiles;
  if (grid > 0x7fffffffLL) {
    snprintf(msg, msglen, "fp32 path: B*H*ceil(N_q/%d) = %lld CTAs exceeds the grid limit", kBM, grid);
    return 3;
  }
  const size_t smem = F32Smem::bytes(int(a.dk), int(a.dv));
  cudaError_t e = cudaFuncSetAttribute(attn_fwd_f32_cc_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
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
