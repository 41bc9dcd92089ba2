// Declarations shared by the translation units of libmoa_attn.so (host side only).
#pragma once
#include <cstddef>
#include <cstdint>
#include <cuda.h>
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
  // Optional per-row log-sum-exp output, fp32 [B*H*N_q] (nullptr: not written).
  float* lse = nullptr;
};

// Query rows per CTA of the bf16 forward (one "query block", the unit of its grid).
constexpr int64_t kQBlockRows = 256;

// How the key axis of the bf16 kernel is split: n_splits contiguous ranges of kv_per_split
// 128-key blocks (the last may be shorter); n_splits == 1 means no split.
struct SplitPlan {
  int n_splits = 1;
  int kv_per_split = 0x7fffffff;
};

// At most `requested` splits, each of at least one key block.
SplitPlan plan_splits(int64_t Nk, int requested);

// The library's own choice for `units` query blocks on `sms` SMs (one CTA per SM): when the
// blocks fill less than one wave, every block's key axis is split so that the CTAs fill the
// SMs; otherwise no split (see the model in the definition).
SplitPlan plan_splits_auto(int64_t units, int64_t Nk, int sms);

// Workspace of a split bf16 call: fp32 partial rows and (m, l) per split and output row.
size_t splitkv_workspace_bytes(int64_t rows, int64_t dv, const SplitPlan& sp);

// SM count of the current device, asked once per device.
cudaError_t device_sm_count(int* sms);

// Raises `func`'s dynamic shared-memory limit to `bytes` on the current device.  The attribute is
// per device, so the call is made once per (kernel, device, size) and its result remembered.
cudaError_t ensure_smem_limit(const void* func, int bytes);

// Size of the fixed device array behind the allocation-free split entry point (16 MiB).
constexpr size_t kNoallocScratchBytes = size_t(16) << 20;

// The launchers return a moa_status code and, on failure, write a message into msg.
int launch_attn_fwd_f32(const AttnArgs& a, char* msg, size_t msglen);
int launch_attn_fwd_bf16(const AttnArgs& a, char* msg, size_t msglen);
// `ws` must hold splitkv_workspace_bytes(B*H*N_q, d_v, sp) bytes (unused when n_splits == 1).
int launch_attn_fwd_bf16_split(const AttnArgs& a, const SplitPlan& sp, void* ws, char* msg,
                               size_t msglen);
// Same, with the partial rows in the library's fixed device array (no allocation; rejects a
// split whose partials exceed kNoallocScratchBytes with MOA_ERR_UNSUPPORTED_SHAPE).
int launch_attn_fwd_bf16_split_noalloc(const AttnArgs& a, const SplitPlan& sp, char* msg,
                                       size_t msglen);

// Tensor map over a contiguous bf16 [BH, N, d] tensor: box of 64 columns x 128 rows, 128-byte
// swizzle, rows past N of a slice read as zero.  False (and a message) on failure.
bool encode_bf16_map(CUtensorMap* map, const void* base, int64_t BH, int64_t N, int64_t d,
                     char* msg, size_t msglen);
// Map over a contiguous fp32 [BH, N, d] tensor: box of box_cols columns (at most 32) x box_rows
// rows, 128-byte swizzle.
bool encode_f32_map_sw128(CUtensorMap* map, const void* base, int64_t BH, int64_t N, int64_t d,
                          int box_cols, int box_rows, char* msg, size_t msglen);
// Same with a box of box_rows rows (64 columns, 128-byte swizzle).
bool encode_bf16_map_box(CUtensorMap* map, const void* base, int64_t BH, int64_t N, int64_t d,
                         int box_rows, char* msg, size_t msglen);

// Validated arguments of one projection call (see include/moa_attn.h, moa_qkv_proj).
struct ProjArgs {
  const void* X;  // [B, N, d]
  const void* W;  // [d, 2*H*dk + H*dv]
  void* Q;
  void* K;
  void* V;
  int64_t B, N, d, H, dk, dv;
  cudaStream_t stream;
};
int launch_qkv_proj_bf16(const ProjArgs& a, char* msg, size_t msglen);
cudaError_t proj_read_and_clear_status(unsigned* value);

// Validated arguments of one backward call (see include/moa_attn.h, moa_attn_bwd).
struct BwdArgs {
  const void* Q;
  const void* K;
  const void* V;
  const void* O;
  const void* dO;
  const float* lse;
  void* dQ;
  void* dK;
  void* dV;
  int64_t B, H, Nq, Nk, dk, dv;
  float scale;
  void* ws;  // bwd_workspace_bytes(...) bytes, 16-byte aligned
  cudaStream_t stream;
};

// Workspace of the backward: per (b,h) and padded query row, D = rowsum(dO * O) and the
// log-sum-exp (bf16 path: in log2 units, negated), fp32.
size_t bwd_workspace_bytes(int64_t B, int64_t H, int64_t Nq);
int launch_attn_bwd_bf16(const BwdArgs& a, char* msg, size_t msglen);
// One kernel for dK, dV and dQ (bf16, d_k = d_v = 64); the workspace adds an fp32 dQ
// accumulator of padded rows x d_k after the two per-row vectors.
size_t bwd_fused_workspace_bytes(int64_t B, int64_t H, int64_t Nq, int64_t dk);
int launch_attn_bwd_bf16_fused(const BwdArgs& a, char* msg, size_t msglen);
// fp32 backward on CUDA cores; same workspace layout (LSE instead of -LSE log2 e in the first half).
int launch_attn_bwd_f32(const BwdArgs& a, char* msg, size_t msglen);
// Reads and clears the status word of the backward kernels' bounded waits (after a sync).
cudaError_t bwd_read_and_clear_status(unsigned* value);

// Launches the bounded-wait self test (a wait that nothing completes) on `stream`.
cudaError_t launch_wait_timeout_selftest(uint64_t limit_ns, cudaStream_t stream);

// Reads and clears the status word of the bf16 kernel's bounded waits (after a sync).
cudaError_t bf16_read_and_clear_status(unsigned* value);

// Limit of one bounded wait inside a kernel, in nanoseconds (env MOA_WAIT_LIMIT_NS, default 1 s).
uint64_t wait_limit_ns();

}  // namespace moa
