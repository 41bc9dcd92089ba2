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
//   attn_fwd_f32_row_kernel  one warp per query row (lane = key of a 32-key chunk for the
//                            scores, lane = output column for the sum over V), for problems too
//                            small to give every SM a 32-row CTA: the work spreads over up to
//                            32x as many warps, which matters when the call is latency-bound.
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

// One warp per query row r = (b*H + h)*N_q + i; 8 rows per CTA.
__global__ void __launch_bounds__(256)
attn_fwd_f32_row_kernel(const float* __restrict__ Q, const float* __restrict__ K,
                        const float* __restrict__ V, float* __restrict__ O,
                        float* __restrict__ lse, int Nq, int Nk, int dk, int dv, float scale,
                        long long rows) {
  __shared__ float sq[8][kMaxD];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long r = (long long)blockIdx.x * 8 + warp;
  if (r >= rows) return;  // whole warps leave together
  const long long bh = r / Nq;
  const float* q = Q + r * dk;
  const float* Kh = K + bh * (long long)Nk * dk;
  const float* Vh = V + bh * (long long)Nk * dv;
  for (int j = lane; j < dk; j += 32) sq[warp][j] = q[j];
  __syncwarp();
  float m = -INFINITY, l = 0.f;
  float acc[kMaxColGroups];
#pragma unroll
  for (int g = 0; g < kMaxColGroups; ++g) acc[g] = 0.f;
  for (int k0 = 0; k0 < Nk; k0 += 32) {
    // lane = key k0 + lane: its score (rows past N_k: -inf)
    const int key = k0 + lane;
    float s = -INFINITY;
    if (key < Nk) {
      const float* kr = Kh + (long long)key * dk;
      float d = 0.f;
      // groups of 4 float4 loads in flight before their products
      for (int j0 = 0; j0 < dk; j0 += 16) {
        float4 kv[4];
#pragma unroll
        for (int u = 0; u < 4; ++u)
          kv[u] = j0 + 4 * u < dk ? *reinterpret_cast<const float4*>(kr + j0 + 4 * u)
                                  : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int j = j0 + 4 * u;
          if (j < dk) {
            d = fmaf(sq[warp][j], kv[u].x, d);
            d = fmaf(sq[warp][j + 1], kv[u].y, d);
            d = fmaf(sq[warp][j + 2], kv[u].z, d);
            d = fmaf(sq[warp][j + 3], kv[u].w, d);
          }
        }
      }
      s = d * scale;
    }
    float cmax = s;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) cmax = fmaxf(cmax, __shfl_xor_sync(0xffffffffu, cmax, off));
    const float mnew = fmaxf(m, cmax);       // finite: every chunk has at least one key
    const float alpha = expf(m - mnew);      // exp(-inf) = 0 on the first chunk
    const float p = expf(s - mnew);          // 0 for keys past N_k
    float psum = p;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) psum += __shfl_xor_sync(0xffffffffu, psum, off);
    l = l * alpha + psum;
    m = mnew;
    // lane = output column: acc = alpha * acc + sum over the chunk's keys of p_k V[k, c]
    const int kn = min(32, Nk - k0);
#pragma unroll
    for (int g = 0; g < kMaxColGroups; ++g) acc[g] *= alpha;
    // eight value rows loaded before their products (keys past N_k read as 0 with p = 0)
    for (int kb = 0; kb < kn; kb += 8) {
      float vv[8][kMaxColGroups];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const float* vr = Vh + (long long)(k0 + kb + u) * dv;
#pragma unroll
        for (int g = 0; g < kMaxColGroups; ++g) {
          const int c = lane + 32 * g;
          vv[u][g] = (kb + u < kn && c < dv) ? vr[c] : 0.f;
        }
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const float pk = __shfl_sync(0xffffffffu, p, (kb + u) & 31);
#pragma unroll
        for (int g = 0; g < kMaxColGroups; ++g) acc[g] = fmaf(pk, vv[u][g], acc[g]);
      }
    }
  }
  const float inv = 1.0f / l;
#pragma unroll
  for (int g = 0; g < kMaxColGroups; ++g) {
    const int c = lane + 32 * g;
    if (c < dv) O[r * dv + c] = acc[g] * inv;
  }
  if (lse != nullptr && lane == 0) lse[r] = m + logf(l);
}

}  // namespace

int launch_attn_fwd_f32(const AttnArgs& a, char* msg, size_t msglen) {
  // Few 32-row CTAs (fewer than two per SM): one warp per row instead.
  int dev = 0, sms = 148;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const long long rows = (long long)a.B * a.H * a.Nq;
  if ((long long)a.B * a.H * ((a.Nq + kBM - 1) / kBM) < 2LL * sms) {
    if ((rows + 7) / 8 > 0x7fffffffLL) {
      snprintf(msg, msglen, "fp32 path: too many rows");
      return 3;
    }
    attn_fwd_f32_row_kernel<<<dim3(unsigned((rows + 7) / 8)), dim3(256), 0, a.stream>>>(
        static_cast<const float*>(a.Q), static_cast<const float*>(a.K),
        static_cast<const float*>(a.V), static_cast<float*>(a.O), a.lse, int(a.Nq), int(a.Nk),
        int(a.dk), int(a.dv), a.scale, rows);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) {
      snprintf(msg, msglen, "fp32 row kernel launch: %s", cudaGetErrorString(e));
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
