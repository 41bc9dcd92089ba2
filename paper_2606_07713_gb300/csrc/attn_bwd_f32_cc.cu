// fp32 attention backward on CUDA cores (no TF32), for the MOA_FP32 element type.
//
// Computes the same gradients as the bf16 backward (paper Stage 5, Section 9):
//     dS = W * (dO V^T - D),  D_i = sum_c dO_ic O_ic,
//     dQ = scale * dS K,  dK = scale * dS^T Q,  dV = W^T dO,
// with the weights rebuilt from the forward's log-sum-exp, W_ik = exp(scale * s_ik - LSE_i), so
// that no N_q x N_k array is written to global memory.  Three kernels, all fp32 with expf:
//   attn_bwd_f32_pre_kernel   one warp per query row: D_i (and LSE_i copied) into the padded
//                             workspace layout of the bf16 path;
//   attn_bwd_f32_dkdv_kernel  one CTA per (b, h, 32 keys): streams the query rows in chunks of
//                             32 through shared memory; warp w owns keys 8w..8w+7, lane = query
//                             for S, P, dP, dS; then lane = output column for dV and dK;
//   attn_bwd_f32_dq_kernel    one CTA per (b, h, 32 query rows): streams the keys in chunks of
//                             32; warp w owns rows 8w..8w+7, lane = key, then lane = column.
// Layout: Q, K, V, O, dO, dQ, dK, dV contiguous row-major [B,H,N,d] float32; d <= 128, d % 4 == 0.
#include <cuda_runtime.h>
#include <math.h>
#include <cstdio>

#include "internal.h"

namespace moa {
namespace {

constexpr int kThreads = 128;
constexpr int kWarps = kThreads / 32;
constexpr int kRowsPerWarp = 8;
constexpr int kTile = kWarps * kRowsPerWarp;  // 32 keys (dK/dV) or 32 query rows (dQ) per CTA
constexpr int kChunk = 32;                    // rows of the streamed axis per step
constexpr int kMaxD = 128;
constexpr int kMaxGroups = kMaxD / 32;        // output columns per lane: c = lane + 32 g

// Padded-row workspace (shared with the bf16 path): row r = bh * Nq_pad + i.
int64_t f32_padded_rows(int64_t Nq) { return (Nq + 127) / 128 * 128; }

// One warp per query row: D = sum_c dO * O; LSE copied beside it.
__global__ void __launch_bounds__(256)
attn_bwd_f32_pre_kernel(const float* __restrict__ O, const float* __restrict__ dO,
                        const float* __restrict__ lse, float* __restrict__ Lw,
                        float* __restrict__ Dw, int Nq, int Nq_pad, int dv, long long rows) {
  const long long t = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (t >= rows) return;
  const long long bh = t / Nq;
  const int i = int(t % Nq);
  const float* o = O + t * dv;
  const float* g = dO + t * dv;
  float acc = 0.f;
  for (int c = lane; c < dv; c += 32) acc = fmaf(o[c], g[c], acc);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
  if (lane == 0) {
    const long long r = bh * Nq_pad + i;
    Lw[r] = lse[t];
    Dw[r] = acc;
  }
}

// dK and dV for 32 keys of one (b, h).
__global__ void __launch_bounds__(kThreads)
attn_bwd_f32_dkdv_kernel(const float* __restrict__ Q, const float* __restrict__ K,
                         const float* __restrict__ V, const float* __restrict__ dO,
                         const float* __restrict__ Lw, const float* __restrict__ Dw,
                         float* __restrict__ dK, float* __restrict__ dV, int Nq, int Nk,
                         int Nq_pad, int dk, int dv, int n_ktiles, float scale) {
  extern __shared__ float smem[];
  const int ldk = dk + 1, ldv = dv + 1;
  float* sK = smem;                       // [kTile][dk+1]
  float* sV = sK + kTile * ldk;           // [kTile][dv+1]
  float* sQ = sV + kTile * ldv;           // [kChunk][dk+1]
  float* sG = sQ + kChunk * ldk;          // [kChunk][dv+1]  (dO)
  float* sP = sG + kChunk * ldv;          // [kWarps][8][kChunk]
  float* sS = sP + kWarps * kRowsPerWarp * kChunk;  // [kWarps][8][kChunk]  (dS)
  float* sL = sS + kWarps * kRowsPerWarp * kChunk;  // [kChunk]
  float* sD = sL + kChunk;                          // [kChunk]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long bh = blockIdx.x / n_ktiles;
  const int k0 = (blockIdx.x % n_ktiles) * kTile;
  const float* Qh = Q + bh * (long long)Nq * dk;
  const float* Kh = K + bh * (long long)Nk * dk;
  const float* Vh = V + bh * (long long)Nk * dv;
  const float* Gh = dO + bh * (long long)Nq * dv;
  const float* Lh = Lw + bh * (long long)Nq_pad;
  const float* Dh = Dw + bh * (long long)Nq_pad;

  for (int idx = threadIdx.x; idx < kTile * dk; idx += kThreads) {
    const int r = idx / dk, j = idx % dk;
    sK[r * ldk + j] = (k0 + r < Nk) ? Kh[(long long)(k0 + r) * dk + j] : 0.f;
  }
  for (int idx = threadIdx.x; idx < kTile * dv; idx += kThreads) {
    const int r = idx / dv, j = idx % dv;
    sV[r * ldv + j] = (k0 + r < Nk) ? Vh[(long long)(k0 + r) * dv + j] : 0.f;
  }
  float accV[kRowsPerWarp][kMaxGroups], accK[kRowsPerWarp][kMaxGroups];
#pragma unroll
  for (int r = 0; r < kRowsPerWarp; ++r)
#pragma unroll
    for (int g = 0; g < kMaxGroups; ++g) accV[r][g] = accK[r][g] = 0.f;
  float* myP = sP + warp * kRowsPerWarp * kChunk;
  float* myS = sS + warp * kRowsPerWarp * kChunk;
  const float* myK = sK + warp * kRowsPerWarp * ldk;
  const float* myV = sV + warp * kRowsPerWarp * ldv;

  for (int q0 = 0; q0 < Nq; q0 += kChunk) {
    __syncthreads();  // previous chunk consumed (and the K/V tile visible on the first pass)
    for (int idx = threadIdx.x; idx < kChunk * dk; idx += kThreads) {
      const int r = idx / dk, j = idx % dk;
      sQ[r * ldk + j] = (q0 + r < Nq) ? Qh[(long long)(q0 + r) * dk + j] : 0.f;
    }
    for (int idx = threadIdx.x; idx < kChunk * dv; idx += kThreads) {
      const int r = idx / dv, j = idx % dv;
      sG[r * ldv + j] = (q0 + r < Nq) ? Gh[(long long)(q0 + r) * dv + j] : 0.f;
    }
    if (threadIdx.x < kChunk) {
      const int q = q0 + threadIdx.x;
      sL[threadIdx.x] = q < Nq ? Lh[q] : INFINITY;  // padded query rows weigh exp(-inf) = 0
      sD[threadIdx.x] = q < Nq ? Dh[q] : 0.f;
    }
    __syncthreads();
    // lane = query q0 + lane: s, p, dp, ds for this warp's 8 keys
    const float* qrow = sQ + lane * ldk;
    const float* grow = sG + lane * ldv;
    const float L = sL[lane], D = sD[lane];
#pragma unroll
    for (int r = 0; r < kRowsPerWarp; ++r) {
      float s = 0.f, dp = 0.f;
      for (int j = 0; j < dk; ++j) s = fmaf(myK[r * ldk + j], qrow[j], s);
      for (int c = 0; c < dv; ++c) dp = fmaf(myV[r * ldv + c], grow[c], dp);
      const float p = expf(s * scale - L);
      myP[r * kChunk + lane] = p;
      myS[r * kChunk + lane] = p * (dp - D);
    }
    __syncwarp();
    // lane = output column: dV += P^T dO, dK += dS^T Q over the chunk's queries
    const int qn = min(kChunk, Nq - q0);
    for (int q = 0; q < qn; ++q) {
      float gq[kMaxGroups], qq[kMaxGroups];
#pragma unroll
      for (int g = 0; g < kMaxGroups; ++g) {
        const int c = lane + 32 * g;
        gq[g] = c < dv ? sG[q * ldv + c] : 0.f;
        qq[g] = c < dk ? sQ[q * ldk + c] : 0.f;
      }
#pragma unroll
      for (int r = 0; r < kRowsPerWarp; ++r) {
        const float p = myP[r * kChunk + q], ds = myS[r * kChunk + q];
#pragma unroll
        for (int g = 0; g < kMaxGroups; ++g) {
          accV[r][g] = fmaf(p, gq[g], accV[r][g]);
          accK[r][g] = fmaf(ds, qq[g], accK[r][g]);
        }
      }
    }
    __syncwarp();
  }
#pragma unroll
  for (int r = 0; r < kRowsPerWarp; ++r) {
    const int key = k0 + warp * kRowsPerWarp + r;
    if (key >= Nk) continue;
#pragma unroll
    for (int g = 0; g < kMaxGroups; ++g) {
      const int c = lane + 32 * g;
      if (c < dv) dV[(bh * Nk + key) * dv + c] = accV[r][g];
      if (c < dk) dK[(bh * Nk + key) * dk + c] = accK[r][g] * scale;
    }
  }
}

// dQ for 32 query rows of one (b, h).
__global__ void __launch_bounds__(kThreads)
attn_bwd_f32_dq_kernel(const float* __restrict__ Q, const float* __restrict__ K,
                       const float* __restrict__ V, const float* __restrict__ dO,
                       const float* __restrict__ Lw, const float* __restrict__ Dw,
                       float* __restrict__ dQ, int Nq, int Nk, int Nq_pad, int dk, int dv,
                       int n_qtiles, float scale) {
  extern __shared__ float smem[];
  const int ldk = dk + 1, ldv = dv + 1;
  float* sQ = smem;                       // [kTile][dk]
  float* sG = sQ + kTile * dk;            // [kTile][dv]
  float* sK = sG + kTile * dv;            // [kChunk][dk+1]
  float* sV = sK + kChunk * ldk;          // [kChunk][dv+1]
  float* sS = sV + kChunk * ldv;          // [kWarps][8][kChunk]  (dS)

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long bh = blockIdx.x / n_qtiles;
  const int q0 = (blockIdx.x % n_qtiles) * kTile;
  const float* Qh = Q + bh * (long long)Nq * dk;
  const float* Kh = K + bh * (long long)Nk * dk;
  const float* Vh = V + bh * (long long)Nk * dv;
  const float* Gh = dO + bh * (long long)Nq * dv;

  for (int idx = threadIdx.x; idx < kTile * dk; idx += kThreads) {
    const int r = idx / dk, j = idx % dk;
    sQ[idx] = (q0 + r < Nq) ? Qh[(long long)(q0 + r) * dk + j] : 0.f;
  }
  for (int idx = threadIdx.x; idx < kTile * dv; idx += kThreads) {
    const int r = idx / dv, j = idx % dv;
    sG[idx] = (q0 + r < Nq) ? Gh[(long long)(q0 + r) * dv + j] : 0.f;
  }
  float L[kRowsPerWarp], D[kRowsPerWarp];
#pragma unroll
  for (int r = 0; r < kRowsPerWarp; ++r) {
    const int q = q0 + warp * kRowsPerWarp + r;
    const long long w = bh * (long long)Nq_pad + (q < Nq ? q : 0);
    L[r] = q < Nq ? Lw[w] : INFINITY;
    D[r] = q < Nq ? Dw[w] : 0.f;
  }
  float acc[kRowsPerWarp][kMaxGroups];
#pragma unroll
  for (int r = 0; r < kRowsPerWarp; ++r)
#pragma unroll
    for (int g = 0; g < kMaxGroups; ++g) acc[r][g] = 0.f;
  float* myS = sS + warp * kRowsPerWarp * kChunk;
  const float* myQ = sQ + warp * kRowsPerWarp * dk;
  const float* myG = sG + warp * kRowsPerWarp * dv;

  for (int c0 = 0; c0 < Nk; c0 += kChunk) {
    __syncthreads();
    for (int idx = threadIdx.x; idx < kChunk * dk; idx += kThreads) {
      const int r = idx / dk, j = idx % dk;
      sK[r * ldk + j] = (c0 + r < Nk) ? Kh[(long long)(c0 + r) * dk + j] : 0.f;
    }
    for (int idx = threadIdx.x; idx < kChunk * dv; idx += kThreads) {
      const int r = idx / dv, j = idx % dv;
      sV[r * ldv + j] = (c0 + r < Nk) ? Vh[(long long)(c0 + r) * dv + j] : 0.f;
    }
    __syncthreads();
    // lane = key c0 + lane (keys past N_k have K = V = 0: their dS multiplies K = 0 below)
    const float* krow = sK + lane * ldk;
    const float* vrow = sV + lane * ldv;
#pragma unroll
    for (int r = 0; r < kRowsPerWarp; ++r) {
      float s = 0.f, dp = 0.f;
      for (int j = 0; j < dk; ++j) s = fmaf(myQ[r * dk + j], krow[j], s);
      for (int c = 0; c < dv; ++c) dp = fmaf(myG[r * dv + c], vrow[c], dp);
      const float p = c0 + lane < Nk ? expf(s * scale - L[r]) : 0.f;
      myS[r * kChunk + lane] = p * (dp - D[r]);
    }
    __syncwarp();
    const int kn = min(kChunk, Nk - c0);
    for (int k = 0; k < kn; ++k) {
      float kk[kMaxGroups];
#pragma unroll
      for (int g = 0; g < kMaxGroups; ++g) {
        const int c = lane + 32 * g;
        kk[g] = c < dk ? sK[k * ldk + c] : 0.f;
      }
#pragma unroll
      for (int r = 0; r < kRowsPerWarp; ++r) {
        const float ds = myS[r * kChunk + k];
#pragma unroll
        for (int g = 0; g < kMaxGroups; ++g) acc[r][g] = fmaf(ds, kk[g], acc[r][g]);
      }
    }
    __syncwarp();
  }
#pragma unroll
  for (int r = 0; r < kRowsPerWarp; ++r) {
    const int q = q0 + warp * kRowsPerWarp + r;
    if (q >= Nq) continue;
#pragma unroll
    for (int g = 0; g < kMaxGroups; ++g) {
      const int c = lane + 32 * g;
      if (c < dk) dQ[(bh * Nq + q) * dk + c] = acc[r][g] * scale;
    }
  }
}

}  // namespace

int launch_attn_bwd_f32(const BwdArgs& a, char* msg, size_t msglen) {
  const int64_t BH = a.B * a.H;
  const int64_t nq_pad = f32_padded_rows(a.Nq);
  const int n_kt = int((a.Nk + kTile - 1) / kTile), n_qt = int((a.Nq + kTile - 1) / kTile);
  if (BH * n_kt > 0x7fffffffLL || BH * n_qt > 0x7fffffffLL || BH * a.Nq / 8 > 0x7fffffffLL) {
    snprintf(msg, msglen, "fp32 backward: grid too large");
    return 3;
  }
  float* Lw = static_cast<float*>(a.ws);
  float* Dw = Lw + BH * nq_pad;
  const int dk = int(a.dk), dv = int(a.dv);
  const long long rows = BH * a.Nq;
  attn_bwd_f32_pre_kernel<<<dim3(unsigned((rows + 7) / 8)), dim3(256), 0, a.stream>>>(
      static_cast<const float*>(a.O), static_cast<const float*>(a.dO), a.lse, Lw, Dw,
      int(a.Nq), int(nq_pad), dv, rows);
  cudaError_t e = cudaGetLastError();
  const size_t smem_kv = sizeof(float) * (size_t(kTile) * (dk + 1) + size_t(kTile) * (dv + 1) +
                                          size_t(kChunk) * (dk + 1) + size_t(kChunk) * (dv + 1) +
                                          2 * size_t(kWarps) * kRowsPerWarp * kChunk + 2 * kChunk);
  const size_t smem_q = sizeof(float) * (size_t(kTile) * dk + size_t(kTile) * dv +
                                         size_t(kChunk) * (dk + 1) + size_t(kChunk) * (dv + 1) +
                                         size_t(kWarps) * kRowsPerWarp * kChunk);
  if (e == cudaSuccess)
    e = ensure_smem_limit(reinterpret_cast<const void*>(attn_bwd_f32_dkdv_kernel), int(smem_kv));
  if (e == cudaSuccess)
    e = ensure_smem_limit(reinterpret_cast<const void*>(attn_bwd_f32_dq_kernel), int(smem_q));
  if (e == cudaSuccess) {
    attn_bwd_f32_dkdv_kernel<<<dim3(unsigned(BH * n_kt)), dim3(kThreads), smem_kv, a.stream>>>(
        static_cast<const float*>(a.Q), static_cast<const float*>(a.K),
        static_cast<const float*>(a.V), static_cast<const float*>(a.dO), Lw, Dw,
        static_cast<float*>(a.dK), static_cast<float*>(a.dV), int(a.Nq), int(a.Nk), int(nq_pad),
        dk, dv, n_kt, a.scale);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) {
    attn_bwd_f32_dq_kernel<<<dim3(unsigned(BH * n_qt)), dim3(kThreads), smem_q, a.stream>>>(
        static_cast<const float*>(a.Q), static_cast<const float*>(a.K),
        static_cast<const float*>(a.V), static_cast<const float*>(a.dO), Lw, Dw,
        static_cast<float*>(a.dQ), int(a.Nq), int(a.Nk), int(nq_pad), dk, dv, n_qt, a.scale);
    e = cudaGetLastError();
  }
  if (e != cudaSuccess) {
    snprintf(msg, msglen, "fp32 backward launch: %s", cudaGetErrorString(e));
    return 5;
  }
  return 0;
}

}  // namespace moa
