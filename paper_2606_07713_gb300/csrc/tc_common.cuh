// Device helpers shared by the tensor-core kernels (forward and backward): tcgen05 instruction
// and shared-memory descriptors, bounded mbarrier waits, packed fp32 arithmetic, bf16 packing and
// TMEM row loads.  Header-only; every function is inlined into the kernel that uses it.
#pragma once
#include <cuda_bf16.h>
#include <cstdint>

#include "ptx.cuh"

namespace moa {
namespace tc {

using namespace ptx;

// Instruction descriptor of tcgen05.mma kind::f16: D fp32, A and B bf16, dense.
//   bits 4-5 D format (1 = f32), 7-9 A format (1 = bf16), 10-12 B format (1 = bf16),
//   15 A major (0 = K-major), 16 B major (1 = MN-major), 17-22 N >> 3, 24-28 M >> 4.
__host__ __device__ constexpr uint32_t make_idesc(int M, int N, bool b_mn_major) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (0u << 15) | ((b_mn_major ? 1u : 0u) << 16) |
         (uint32_t(N >> 3) << 17) | (uint32_t(M >> 4) << 24);
}
// Same with the A operand (from shared memory) MN-major as well (bit 15: A transposed).
__host__ __device__ constexpr uint32_t make_idesc_a_mn(int M, int N, bool b_mn_major) {
  return make_idesc(M, N, b_mn_major) | (1u << 15);
}

// Shared-memory matrix descriptor, 128-byte swizzle (layout code 2 in bits 61-63), version 1
// (bits 46-47).  Start address, leading and stride byte offsets in 16-byte units.
__device__ __forceinline__ uint64_t make_sdesc_sw128(uint32_t addr, uint32_t lbo, uint32_t sbo) {
  return uint64_t((addr & 0x3FFFFu) >> 4) | (uint64_t((lbo >> 4) & 0x3FFFu) << 16) |
         (uint64_t((sbo >> 4) & 0x3FFFu) << 32) | (uint64_t(1) << 46) | (uint64_t(2) << 61);
}

struct WaitCtl {
  volatile int* abort_flag;
  uint64_t limit_ns;
  uint32_t hint_ns;  // 0: poll; otherwise let a not-yet-complete test suspend the thread
  unsigned* status;  // the translation unit's device status word
};

// Bounded mbarrier wait.  Returns false (and raises the CTA abort flag and writes
// MOA_ERR_DEVICE_TIMEOUT to the status word) if the phase did not complete within limit_ns, or
// if another role already aborted.
__device__ __forceinline__ bool wait_bounded(uint32_t bar, uint32_t parity, const WaitCtl& w) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 1;; ++it) {
    if (w.hint_ns ? mbar_try_wait_hint(bar, parity, w.hint_ns) : mbar_try_wait(bar, parity))
      return true;
    if ((it & 63u) == 0) {
      if (*w.abort_flag) return false;
      if (globaltimer_ns() - t0 > w.limit_ns) {
        *w.abort_flag = 1;
        atomicExch(w.status, 6u);  // MOA_ERR_DEVICE_TIMEOUT
        return false;
      }
    }
  }
}

// Time-limited wait that ignores the abort flag: used on the way out so that no TMA copy or
// tensor-core operation is still writing shared or tensor memory when the CTA exits.
__device__ __forceinline__ void wait_quiesce(uint32_t bar, uint32_t parity, uint64_t limit_ns,
                                             unsigned* status) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > limit_ns) {
      atomicExch(status, 6u);
      return;
    }
  }
}

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// log2 by the MUFU lg2 instruction (absolute error about 2^-22 for the row sums l >= 1 used here).
__device__ __forceinline__ float lg2_approx(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);  // .x (low 16 bits) = lo
  return *reinterpret_cast<uint32_t*>(&v);
}

// Packed fp32 pairs (Blackwell f32x2 ALU forms): one instruction for two lanes of data.
__device__ __forceinline__ uint64_t pack_f32x2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
// (d0, d1) = (a0, a1) * b + c, with b and c packed pairs.
__device__ __forceinline__ void ffma2(float& d0, float& d1, float a0, float a1, uint64_t b,
                                      uint64_t c) {
  asm("{\n\t.reg .b64 ra, rd;\n\tmov.b64 ra, {%2, %3};\n\t"
      "fma.rn.f32x2 rd, ra, %4, %5;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d0), "=f"(d1)
      : "f"(a0), "f"(a1), "l"(b), "l"(c));
}
// (a0, a1) += (b0, b1).
__device__ __forceinline__ void fadd2(float& a0, float& a1, float b0, float b1) {
  asm("{\n\t.reg .b64 ra, rb, rd;\n\tmov.b64 ra, {%0, %1};\n\tmov.b64 rb, {%2, %3};\n\t"
      "add.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "+f"(a0), "+f"(a1)
      : "f"(b0), "f"(b1));
}
__device__ __forceinline__ float max3f(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
// Loads 128 fp32 columns of this thread's TMEM lane into s[] and waits for completion.
__device__ __forceinline__ void tmem_load_row128(uint32_t taddr, uint32_t* s) {
  tmem_ld_32x32b_x32(taddr + 0, s + 0);
  tmem_ld_32x32b_x32(taddr + 32, s + 32);
  tmem_ld_32x32b_x32(taddr + 64, s + 64);
  tmem_ld_32x32b_x32(taddr + 96, s + 96);
  tmem_wait_ld();
  reg_anchor_x32(s + 0);
  reg_anchor_x32(s + 32);
  reg_anchor_x32(s + 64);
  reg_anchor_x32(s + 96);
}

}  // namespace tc
}  // namespace moa
