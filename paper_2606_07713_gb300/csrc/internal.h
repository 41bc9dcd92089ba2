// Declarations shared by the translation units of libmoa_attn.so (host side only).
#pragma once
#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

namespace moa {

// Validated arguments of one attention call (see include/moa_attn.h).
struct AttnArgs {
  const void* Q;
  const void* K;
  const void* V;
  void* O;
  int64_t B, H, Nq, Nk, dk, dv;
  float scale;
  cudaStream_t stream;
};

// Both launchers return a moa_status code and, on failure, write a message into msg.
int launch_attn_fwd_f32(const AttnArgs& a, char* msg, size_t msglen);
int launch_attn_fwd_bf16(const AttnArgs& a, char* msg, size_t msglen);

// Launches the bounded-wait self test (a wait that nothing completes) on `stream`.
cudaError_t launch_wait_timeout_selftest(uint64_t limit_ns, cudaStream_t stream);

// Reads and clears the status word of the bf16 kernel's bounded waits (after a sync).
cudaError_t bf16_read_and_clear_status(unsigned* value);

// Limit of one bounded wait inside a kernel, in nanoseconds (env MOA_WAIT_LIMIT_NS, default 1 s).
uint64_t wait_limit_ns();

}  // namespace moa
