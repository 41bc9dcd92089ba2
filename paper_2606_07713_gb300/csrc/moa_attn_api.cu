// C ABI of libmoa_attn.so: argument checks, dispatch to the kernels, status and helpers.
// The contract of every entry point is documented in include/moa_attn.h.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdarg>
#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <vector>

#include "../../include/moa_attn.h"
#include "internal.h"

namespace moa {

uint64_t wait_limit_ns() {
  static const uint64_t v = [] {
    const char* s = std::getenv("MOA_WAIT_LIMIT_NS");
    if (s && *s) {
      const unsigned long long x = std::strtoull(s, nullptr, 10);
      if (x > 0) return uint64_t(x);
    }
    return uint64_t(1000000000ull);  // 1 s
  }();
  return v;
}

namespace {
std::mutex g_sm_mu;
int g_sm_count[64] = {};

struct SmemLimit {
  const void* func;
  int dev;
  int bytes;
  cudaError_t result;
};
std::mutex g_smem_mu;
std::vector<SmemLimit> g_smem_limits;
}  // namespace

cudaError_t ensure_smem_limit(const void* func, int bytes) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(g_smem_mu);
  for (const SmemLimit& s : g_smem_limits)
    if (s.func == func && s.dev == dev && s.bytes >= bytes) return s.result;
  e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  g_smem_limits.push_back({func, dev, bytes, e});
  return e;
}

cudaError_t device_sm_count(int* sms) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_sm_mu);
  if (g_sm_count[dev] <= 0) {
    int n = 0;
    e = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    if (n <= 0) return cudaErrorInvalidDevice;
    g_sm_count[dev] = n;
  }
  *sms = g_sm_count[dev];
  return cudaSuccess;
}

namespace {

thread_local char t_last_error[512] = {0};

int fail(int code, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(t_last_error, sizeof(t_last_error), fmt, ap);
  va_end(ap);
  return code;
}

// a * b for non-negative values, or -1 on overflow of int64.
int64_t mul_checked(int64_t a, int64_t b) {
  if (a < 0 || b < 0) return -1;
  if (a != 0 && b > INT64_MAX / a) return -1;
  return a * b;
}

int64_t numel4(int64_t a, int64_t b, int64_t c, int64_t d) {
  int64_t x = mul_checked(a, b);
  x = x < 0 ? -1 : mul_checked(x, c);
  return x < 0 ? -1 : mul_checked(x, d);
}

bool overlaps(const void* a, int64_t abytes, const void* b, int64_t bbytes) {
  const uintptr_t a0 = reinterpret_cast<uintptr_t>(a), b0 = reinterpret_cast<uintptr_t>(b);
  return a0 < b0 + uintptr_t(bbytes) && b0 < a0 + uintptr_t(abytes);
}

// Checks everything that can be checked without touching the device.  On success fills *sz
// with the byte sizes of Q, K, V, O.
int validate(const void* Q, const void* K, const void* V, void* O, int64_t B, int64_t H,
             int64_t Nq, int64_t Nk, int64_t dk, int64_t dv, float scale, int dtype,
             int64_t sz[4]) {
  if (!Q || !K || !V || !O) return fail(MOA_ERR_INVALID_ARG, "null tensor pointer");
  if (B <= 0 || H <= 0 || Nq <= 0 || Nk <= 0 || dk <= 0 || dv <= 0)
    return fail(MOA_ERR_INVALID_ARG,
                "sizes must be >= 1 (B=%lld H=%lld N_q=%lld N_k=%lld d_k=%lld d_v=%lld)",
                (long long)B, (long long)H, (long long)Nq, (long long)Nk, (long long)dk,
                (long long)dv);
  if (!std::isfinite(scale)) return fail(MOA_ERR_INVALID_ARG, "scale must be finite");
  if (dtype != MOA_FP32 && dtype != MOA_BF16)
    return fail(MOA_ERR_UNSUPPORTED_DTYPE, "unknown dtype %d", dtype);
  const int64_t elt = dtype == MOA_FP32 ? 4 : 2;
  const int64_t nq = numel4(B, H, Nq, dk), nk = numel4(B, H, Nk, dk);
  const int64_t nv = numel4(B, H, Nk, dv), no = numel4(B, H, Nq, dv);
  if (nq < 0 || nk < 0 || nv < 0 || no < 0 || nq > INT64_MAX / 4 || nk > INT64_MAX / 4 ||
      nv > INT64_MAX / 4 || no > INT64_MAX / 4)
    return fail(MOA_ERR_UNSUPPORTED_SHAPE, "tensor sizes overflow 64-bit byte counts");
  if (B * H > 0x7fffffffLL || Nq > 0x7fffffffLL || Nk > 0x7fffffffLL)
    return fail(MOA_ERR_UNSUPPORTED_SHAPE, "B*H, N_q and N_k must each be below 2^31");
  if (dtype == MOA_BF16) {
    if ((dk != 64 && dk != 128) || (dv != 64 && dv != 128))
      return fail(MOA_ERR_UNSUPPORTED_SHAPE, "bf16 needs d_k, d_v in {64, 128}; got %lld, %lld",
                  (long long)dk, (long long)dv);
  } else {
    if (dk > 128 || dv > 128)
      return fail(MOA_ERR_UNSUPPORTED_SHAPE, "fp32 needs d_k, d_v <= 128; got %lld, %lld",
                  (long long)dk, (long long)dv);
    if (dk % 4 != 0 || dv % 4 != 0)
      return fail(MOA_ERR_MISALIGNED, "fp32 rows must be multiples of 16 bytes (d %% 4 == 0)");
  }
  const void* ptrs[4] = {Q, K, V, O};
  for (const void* p : ptrs)
    if (reinterpret_cast<uintptr_t>(p) % 16 != 0)
      return fail(MOA_ERR_MISALIGNED, "tensor pointer %p is not 16-byte aligned", p);
  sz[0] = nq * elt;
  sz[1] = nk * elt;
  sz[2] = nv * elt;
  sz[3] = no * elt;
  if (overlaps(O, sz[3], Q, sz[0]) || overlaps(O, sz[3], K, sz[1]) ||
      overlaps(O, sz[3], V, sz[2]))
    return fail(MOA_ERR_INVALID_ARG, "O overlaps an input tensor");
  return MOA_OK;
}

// MOA_DEBUG_SYNC=1: every entry point synchronises its stream after launching and reports a
// CUDA error or a recorded wait timeout from that call directly (debugging aid; off by default).
bool debug_sync() {
  static const bool v = [] {
    const char* s = std::getenv("MOA_DEBUG_SYNC");
    return s && *s && std::strcmp(s, "0") != 0;
  }();
  return v;
}

int debug_check(void* stream) {
  if (!debug_sync()) return MOA_OK;
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return fail(MOA_ERR_CUDA, "debug sync: %s", cudaGetErrorString(e));
  unsigned v = 0, vb = 0, vp = 0;
  e = bf16_read_and_clear_status(&v);
  if (e == cudaSuccess) e = bwd_read_and_clear_status(&vb);
  if (e == cudaSuccess) e = proj_read_and_clear_status(&vp);
  if (e != cudaSuccess) return fail(MOA_ERR_CUDA, "debug status read: %s", cudaGetErrorString(e));
  if ((v | vb | vp) != 0)
    return fail(MOA_ERR_DEVICE_TIMEOUT, "debug sync: a kernel wait ran out (status %u)", v | vb | vp);
  return MOA_OK;
}

int dispatch(const void* Q, const void* K, const void* V, void* O, int64_t B, int64_t H,
             int64_t Nq, int64_t Nk, int64_t dk, int64_t dv, float scale, int dtype,
             void* stream, float* lse = nullptr) {
  AttnArgs a{Q, K, V, O, B, H, Nq, Nk, dk, dv, scale, static_cast<cudaStream_t>(stream), lse};
  char msg[256] = {0};
  const int rc = dtype == MOA_BF16 ? launch_attn_fwd_bf16(a, msg, sizeof(msg))
                                   : launch_attn_fwd_f32(a, msg, sizeof(msg));
  if (rc != MOA_OK) return fail(rc, "%s", msg);
  t_last_error[0] = '\0';
  return debug_check(stream);
}

// Side streams and events of the pipelined staged call, one set per device, created on the
// device's first staged call.  The mutex is held while a call enqueues its work, so the events
// of two concurrent calls never interleave.
// Head ranges of the staged call: about kStageChunkBytes of inputs on average, 2 to
// kMaxStageChunks of them, the outer ones smaller (measured on a GB300, end to end, with kernels
// on two compute streams: equal ranges / weights 1, 2, 3, 3, ..., 3, 2, 1 gave 185 / 201 TFLOP/s
// on 4x16x2048^2 d=64, 912 / 955 on 2x32x8192^2 d=128, 1630 / 1678 on 1x16x32768^2 d=128; up to
// 16 ranges, 8 MiB ranges or weights capped at 2 or 4 were no better).
constexpr int kMaxStageChunks = 8;
constexpr int64_t kStageChunkBytes = int64_t(16) << 20;
// Range sizes: 0 = equal; R > 0 = weights min(c + 1, n - c, R), so that the first range (whose
// copy nothing hides) and the last (whose kernel and copy back nothing hides) are small.
constexpr int kStageRamp = 3;

// Head boundaries of the staged call's ranges: range c is [bound[c], bound[c + 1]).
void stage_bounds(int64_t BH, int chunks, int64_t* bound) {
  bound[0] = 0;
  if (kStageRamp <= 0) {
    const int64_t per = (BH + chunks - 1) / chunks;
    for (int c = 1; c <= chunks; ++c) bound[c] = c * per < BH ? c * per : BH;
    return;
  }
  int64_t w[kMaxStageChunks + 1], total = 0;
  for (int c = 0; c < chunks; ++c) {
    int64_t x = c + 1 < chunks - c ? c + 1 : chunks - c;
    w[c] = x < kStageRamp ? x : kStageRamp;
    total += w[c];
  }
  int64_t acc = 0;
  for (int c = 0; c < chunks; ++c) {
    acc += w[c];
    int64_t b = (BH * acc + total / 2) / total;
    const int64_t lo = bound[c] + 1, hi = BH - (chunks - 1 - c);  // at least one head each
    bound[c + 1] = b < lo ? lo : (b > hi ? hi : b);
  }
}
constexpr int kMaxDevices = 64;
struct StagePipe {
  // compute2 takes every other range's kernel, so that the last wave of one range's kernel
  // shares the GPU with the first CTAs of the next instead of leaving SMs idle.
  cudaStream_t copy_in = nullptr, copy_out = nullptr, compute2 = nullptr;
  cudaEvent_t start = nullptr, end = nullptr;
  cudaEvent_t in_done[kMaxStageChunks] = {}, kern_done[kMaxStageChunks] = {};
  bool ready = false;
};
StagePipe g_pipes[kMaxDevices];
std::mutex g_pipe_mu[kMaxDevices];

cudaError_t make_pipe(StagePipe& p) {
  cudaError_t e = cudaStreamCreateWithFlags(&p.copy_in, cudaStreamNonBlocking);
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&p.copy_out, cudaStreamNonBlocking);
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&p.compute2, cudaStreamNonBlocking);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&p.start, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&p.end, cudaEventDisableTiming);
  for (int c = 0; e == cudaSuccess && c < kMaxStageChunks; ++c) {
    e = cudaEventCreateWithFlags(&p.in_done[c], cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&p.kern_done[c], cudaEventDisableTiming);
  }
  p.ready = e == cudaSuccess;
  return e;
}

int current_sm_count(int* sms) {
  const cudaError_t e = device_sm_count(sms);
  if (e != cudaSuccess)
    return fail(MOA_ERR_CUDA, "SM count of the current device: %s", cudaGetErrorString(e));
  return MOA_OK;
}

// The split of a bf16 call: num_splits splits of every query block, or for MOA_SPLITS_AUTO the
// library's choice for `sms` SMs (sms <= 0: the current device's count).
int choose_plan(int64_t B, int64_t H, int64_t Nq, int64_t Nk, int num_splits, int sms,
                SplitPlan* sp) {
  if (num_splits < 0) return fail(MOA_ERR_INVALID_ARG, "num_splits must be >= 0");
  if (num_splits > 0) {
    *sp = plan_splits(Nk, num_splits);
    return MOA_OK;
  }
  if (sms <= 0) {
    const int rc = current_sm_count(&sms);
    if (rc != MOA_OK) return rc;
  }
  const int64_t units = numel4(B, H, (Nq + kQBlockRows - 1) / kQBlockRows, 1);
  if (units < 0) return fail(MOA_ERR_INVALID_ARG, "sizes overflow");
  *sp = plan_splits_auto(units, Nk, sms);
  return MOA_OK;
}

// Validation and dispatch of the two backward entry points.
int bwd_call(const void* Q, const void* K, const void* V, const void* O, const void* dO,
             const float* LSE, void* dQ, void* dK, void* dV, int64_t B, int64_t H, int64_t N_q,
             int64_t N_k, int64_t d_k, int64_t d_v, float scale, int dtype, void* workspace,
             size_t workspace_bytes, void* stream, bool fused) {
  if (!dO || !LSE || !dQ || !dK || !dV)
    return fail(MOA_ERR_INVALID_ARG, "null pointer among dO, LSE, dQ, dK, dV");
  int64_t sz[4];
  int rc = validate(Q, K, V, const_cast<void*>(O), B, H, N_q, N_k, d_k, d_v, scale, dtype, sz);
  if (rc != MOA_OK) return rc;
  if (fused && dtype != MOA_BF16)
    return fail(MOA_ERR_UNSUPPORTED_DTYPE, "the fused backward takes bf16 tensors only");
  if (fused && (d_k != 64 || d_v != 64))
    return fail(MOA_ERR_UNSUPPORTED_SHAPE, "the fused backward needs d_k = d_v = 64; got %lld, %lld",
                (long long)d_k, (long long)d_v);
  const void* al[5] = {dO, dQ, dK, dV, workspace};
  for (const void* p : al)
    if (reinterpret_cast<uintptr_t>(p) % 16 != 0)
      return fail(MOA_ERR_MISALIGNED, "pointer %p is not 16-byte aligned", p);
  if (reinterpret_cast<uintptr_t>(LSE) % 4 != 0)
    return fail(MOA_ERR_MISALIGNED, "LSE pointer is not 4-byte aligned");
  if (fused && numel4(B, H, N_q + 127, 2 + d_k) < 0)
    return fail(MOA_ERR_INVALID_ARG, "sizes overflow");
  const size_t need = fused ? bwd_fused_workspace_bytes(B, H, N_q, d_k)
                            : bwd_workspace_bytes(B, H, N_q);
  if (workspace == nullptr || workspace_bytes < need)
    return fail(MOA_ERR_INVALID_ARG, "workspace too small: need %zu bytes, got %zu", need,
                workspace == nullptr ? size_t(0) : workspace_bytes);
  // Read-only: Q, K, V, O, dO, LSE.  Written: dQ, dK, dV, workspace (no two may overlap, and
  // none may overlap a read-only buffer).
  const void* ro[6] = {Q, K, V, O, dO, LSE};
  const int64_t rosz[6] = {sz[0], sz[1], sz[2], sz[3], sz[3], B * H * N_q * 4};
  const void* wr[4] = {dQ, dK, dV, workspace};
  const int64_t wrsz[4] = {sz[0], sz[1], sz[2], int64_t(need)};
  for (int i = 0; i < 4; ++i) {
    for (int j = 0; j < 6; ++j)
      if (overlaps(wr[i], wrsz[i], ro[j], rosz[j]))
        return fail(MOA_ERR_INVALID_ARG, "an output or the workspace overlaps an input");
    for (int j = i + 1; j < 4; ++j)
      if (overlaps(wr[i], wrsz[i], wr[j], wrsz[j]))
        return fail(MOA_ERR_INVALID_ARG, "outputs or the workspace overlap each other");
  }
  BwdArgs a{Q, K, V, O, dO, LSE, dQ, dK, dV, B, H, N_q, N_k, d_k, d_v, scale, workspace,
            static_cast<cudaStream_t>(stream)};
  char msg[256] = {0};
  rc = fused ? launch_attn_bwd_bf16_fused(a, msg, sizeof(msg))
             : dtype == MOA_BF16 ? launch_attn_bwd_bf16(a, msg, sizeof(msg))
                                 : launch_attn_bwd_f32(a, msg, sizeof(msg));
  if (rc != MOA_OK) return fail(rc, "%s", msg);
  t_last_error[0] = '\0';
  return debug_check(stream);
}

}  // namespace
}  // namespace moa

extern "C" {

int moa_attn_fwd(const void* Q, const void* K, const void* V, void* O, int64_t B, int64_t H,
                 int64_t N_q, int64_t N_k, int64_t d_k, int64_t d_v, float scale, int dtype,
                 void* stream) {
  int64_t sz[4];
  const int rc = moa::validate(Q, K, V, O, B, H, N_q, N_k, d_k, d_v, scale, dtype, sz);
  if (rc != MOA_OK) return rc;
  return moa::dispatch(Q, K, V, O, B, H, N_q, N_k, d_k, d_v, scale, dtype, stream);
}

int moa_attn_fwd_lse(const void* Q, const void* K, const void* V, void* O, float* LSE, int64_t B,
                     int64_t H, int64_t N_q, int64_t N_k, int64_t d_k, int64_t d_v, float scale,
                     int dtype, void* stream) {
  int64_t sz[4];
  const int rc = moa::validate(Q, K, V, O, B, H, N_q, N_k, d_k, d_v, scale, dtype, sz);
  if (rc != MOA_OK) return rc;
  if (LSE == nullptr) return moa::fail(MOA_ERR_INVALID_ARG, "null LSE pointer");
  if (reinterpret_cast<uintptr_t>(LSE) % 4 != 0)
    return moa::fail(MOA_ERR_MISALIGNED, "LSE pointer is not 4-byte aligned");
  const int64_t lse_bytes = B * H * N_q * 4;  // validate() bounded B*H*N_q*d_q*4
  const void* ins[4] = {Q, K, V, O};
  for (int i = 0; i < 4; ++i)
    if (moa::overlaps(LSE, lse_bytes, ins[i], sz[i]))
      return moa::fail(MOA_ERR_INVALID_ARG, "LSE overlaps a tensor");
  return moa::dispatch(Q, K, V, O, B, H, N_q, N_k, d_k, d_v, scale, dtype, stream, LSE);
}

int moa_attn_fwd_staged(const void* hQ, const void* hK, const void* hV, void* hO, void* dQ,
                        void* dK, void* dV, void* dO, int64_t B, int64_t H, int64_t N_q,
                        int64_t N_k, int64_t d_k, int64_t d_v, float scale, int dtype,
                        void* stream) {
  if (!hQ || !hK || !hV || !hO) return moa::fail(MOA_ERR_INVALID_ARG, "null host pointer");
  int64_t sz[4];
  int rc = moa::validate(dQ, dK, dV, dO, B, H, N_q, N_k, d_k, d_v, scale, dtype, sz);
  if (rc != MOA_OK) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= moa::kMaxDevices)
    return moa::fail(MOA_ERR_CUDA, "no usable current device: %s", cudaGetErrorString(e));
  // The (b, h) problems are independent, so the call is pipelined over head ranges: the
  // host-to-device copies of range c+1 (side stream) overlap the kernel of range c (`stream`
  // for even c, a second compute stream for odd c, so that consecutive kernels may overlap),
  // whose output goes back on a third side stream while later ranges compute.
  std::lock_guard<std::mutex> lock(moa::g_pipe_mu[dev]);
  moa::StagePipe& p = moa::g_pipes[dev];
  if (!p.ready && (e = moa::make_pipe(p)) != cudaSuccess)
    return moa::fail(MOA_ERR_CUDA, "staged pipeline set-up: %s", cudaGetErrorString(e));
  const int64_t BH = B * H;
  const int64_t elt = dtype == MOA_FP32 ? 4 : 2;
  const int64_t row_bytes[4] = {N_q * d_k * elt, N_k * d_k * elt, N_k * d_v * elt, N_q * d_v * elt};
  const int64_t in_bytes = sz[0] + sz[1] + sz[2];
  int64_t want = (in_bytes + moa::kStageChunkBytes - 1) / moa::kStageChunkBytes;
  want = want < 2 ? 2 : (want > moa::kMaxStageChunks ? moa::kMaxStageChunks : want);
  const int chunks = int(BH < want ? BH : want);
  int64_t bound[moa::kMaxStageChunks + 1];
  moa::stage_bounds(BH, chunks, bound);
  const void* src[3] = {hQ, hK, hV};
  void* dst[3] = {dQ, dK, dV};
  auto chk = [&](cudaError_t err, const char* what) {
    if (err != cudaSuccess) moa::fail(MOA_ERR_CUDA, "%s: %s", what, cudaGetErrorString(err));
    return err == cudaSuccess;
  };
  // Work already queued on `stream` (e.g. a kernel still reading dQ) finishes before the copies.
  if (!chk(cudaEventRecord(p.start, s), "event record") ||
      !chk(cudaStreamWaitEvent(p.copy_in, p.start, 0), "stream wait") ||
      !chk(cudaStreamWaitEvent(p.compute2, p.start, 0), "stream wait"))
    return MOA_ERR_CUDA;
  for (int c = 0; c < chunks; ++c) {
    const int64_t h0 = bound[c], nh = bound[c + 1] - bound[c];
    if (nh <= 0) break;
    for (int t = 0; t < 3; ++t)
      if (!chk(cudaMemcpyAsync(static_cast<char*>(dst[t]) + h0 * row_bytes[t],
                               static_cast<const char*>(src[t]) + h0 * row_bytes[t],
                               size_t(nh * row_bytes[t]), cudaMemcpyHostToDevice, p.copy_in),
               "host-to-device copy"))
        return MOA_ERR_CUDA;
    if (!chk(cudaEventRecord(p.in_done[c], p.copy_in), "event record")) return MOA_ERR_CUDA;
  }
  for (int c = 0; c < chunks; ++c) {
    const int64_t h0 = bound[c], nh = bound[c + 1] - bound[c];
    if (nh <= 0) break;
    cudaStream_t cs = (c & 1) ? p.compute2 : s;
    if (!chk(cudaStreamWaitEvent(cs, p.in_done[c], 0), "stream wait")) return MOA_ERR_CUDA;
    rc = moa::dispatch(static_cast<const char*>(dQ) + h0 * row_bytes[0],
                       static_cast<const char*>(dK) + h0 * row_bytes[1],
                       static_cast<const char*>(dV) + h0 * row_bytes[2],
                       static_cast<char*>(dO) + h0 * row_bytes[3], 1, nh, N_q, N_k, d_k, d_v,
                       scale, dtype, cs);
    if (rc != MOA_OK) return rc;
    if (!chk(cudaEventRecord(p.kern_done[c], cs), "event record") ||
        !chk(cudaStreamWaitEvent(p.copy_out, p.kern_done[c], 0), "stream wait") ||
        !chk(cudaMemcpyAsync(static_cast<char*>(hO) + h0 * row_bytes[3],
                             static_cast<const char*>(dO) + h0 * row_bytes[3],
                             size_t(nh * row_bytes[3]), cudaMemcpyDeviceToHost, p.copy_out),
             "device-to-host copy"))
      return MOA_ERR_CUDA;
  }
  // `stream` completes only after the last copy back, which follows every range's kernel on
  // either compute stream: synchronising `stream` makes hO valid.
  if (!chk(cudaEventRecord(p.end, p.copy_out), "event record") ||
      !chk(cudaStreamWaitEvent(s, p.end, 0), "stream wait"))
    return MOA_ERR_CUDA;
  moa::t_last_error[0] = '\0';
  return MOA_OK;
}

size_t moa_attn_splitkv_workspace_bytes(int64_t B, int64_t H, int64_t N_q, int64_t N_k,
                                        int64_t d_k, int64_t d_v, int dtype, int num_splits) {
  (void)d_k;
  if (dtype != MOA_BF16 || B <= 0 || H <= 0 || N_q <= 0 || N_k <= 0 || d_v <= 0) return 0;
  if (moa::numel4(B, H, N_q, d_v) < 0) return 0;
  moa::SplitPlan sp;
  if (moa::choose_plan(B, H, N_q, N_k, num_splits, 0, &sp) != MOA_OK) return 0;
  return moa::splitkv_workspace_bytes(B * H * N_q, d_v, sp);
}

int moa_attn_split_plan(int64_t B, int64_t H, int64_t N_q, int64_t N_k, int num_splits,
                        int sm_count, int* splits, int* key_blocks_per_split,
                        int64_t* whole_query_blocks) {
  if (B <= 0 || H <= 0 || N_q <= 0 || N_k <= 0)
    return moa::fail(MOA_ERR_INVALID_ARG, "sizes must be positive");
  if (moa::numel4(B, H, N_q, 1) < 0) return moa::fail(MOA_ERR_INVALID_ARG, "sizes overflow");
  moa::SplitPlan sp;
  const int rc = moa::choose_plan(B, H, N_q, N_k, num_splits, sm_count, &sp);
  if (rc != MOA_OK) return rc;
  const int64_t units = B * H * ((N_q + moa::kQBlockRows - 1) / moa::kQBlockRows);
  const int64_t n_kt = (N_k + 127) / 128;
  if (splits) *splits = sp.n_splits;
  if (key_blocks_per_split)
    *key_blocks_per_split = int(sp.n_splits > 1 ? sp.kv_per_split : n_kt);
  if (whole_query_blocks) *whole_query_blocks = sp.n_splits > 1 ? 0 : units;
  moa::t_last_error[0] = '\0';
  return MOA_OK;
}

int moa_attn_fwd_splitkv(const void* Q, const void* K, const void* V, void* O, int64_t B,
                         int64_t H, int64_t N_q, int64_t N_k, int64_t d_k, int64_t d_v,
                         float scale, int dtype, int num_splits, void* workspace,
                         size_t workspace_bytes, void* stream) {
  int64_t sz[4];
  int rc = moa::validate(Q, K, V, O, B, H, N_q, N_k, d_k, d_v, scale, dtype, sz);
  if (rc != MOA_OK) return rc;
  if (num_splits < 0) return moa::fail(MOA_ERR_INVALID_ARG, "num_splits must be >= 0");
  if (dtype != MOA_BF16)  // the fp32 path has no split form; it computes the same result whole
    return moa::dispatch(Q, K, V, O, B, H, N_q, N_k, d_k, d_v, scale, dtype, stream);
  moa::SplitPlan sp;
  rc = moa::choose_plan(B, H, N_q, N_k, num_splits, 0, &sp);
  if (rc != MOA_OK) return rc;
  const size_t need = moa::splitkv_workspace_bytes(B * H * N_q, d_v, sp);
  if (need > 0) {
    if (workspace == nullptr || workspace_bytes < need)
      return moa::fail(MOA_ERR_INVALID_ARG, "workspace too small: need %zu bytes, got %zu", need,
                       workspace == nullptr ? size_t(0) : workspace_bytes);
    if (reinterpret_cast<uintptr_t>(workspace) % 16 != 0)
      return moa::fail(MOA_ERR_MISALIGNED, "workspace is not 16-byte aligned");
    const void* ins[4] = {Q, K, V, O};
    const int64_t insz[4] = {sz[0], sz[1], sz[2], sz[3]};
    for (int i = 0; i < 4; ++i)
      if (moa::overlaps(workspace, int64_t(need), ins[i], insz[i]))
        return moa::fail(MOA_ERR_INVALID_ARG, "workspace overlaps a tensor");
  }
  moa::AttnArgs a{Q, K, V, O, B, H, N_q, N_k, d_k, d_v, scale, static_cast<cudaStream_t>(stream)};
  char msg[256] = {0};
  rc = moa::launch_attn_fwd_bf16_split(a, sp, workspace, msg, sizeof(msg));
  if (rc != MOA_OK) return moa::fail(rc, "%s", msg);
  moa::t_last_error[0] = '\0';
  return moa::debug_check(stream);
}

int moa_attn_fwd_splitkv_noalloc(const void* Q, const void* K, const void* V, void* O, int64_t B,
                                 int64_t H, int64_t N_q, int64_t N_k, int64_t d_k, int64_t d_v,
                                 float scale, int dtype, int num_splits, void* stream) {
  int64_t sz[4];
  int rc = moa::validate(Q, K, V, O, B, H, N_q, N_k, d_k, d_v, scale, dtype, sz);
  if (rc != MOA_OK) return rc;
  if (num_splits < 0) return moa::fail(MOA_ERR_INVALID_ARG, "num_splits must be >= 0");
  if (dtype != MOA_BF16)  // no split form, no scratch: the whole fp32 computation
    return moa::dispatch(Q, K, V, O, B, H, N_q, N_k, d_k, d_v, scale, dtype, stream);
  moa::SplitPlan sp;
  rc = moa::choose_plan(B, H, N_q, N_k, num_splits, 0, &sp);
  if (rc != MOA_OK) return rc;
  // The library's own choice never fails for want of scratch: it runs unsplit instead.
  if (num_splits == MOA_SPLITS_AUTO &&
      moa::splitkv_workspace_bytes(B * H * N_q, d_v, sp) > moa::kNoallocScratchBytes)
    sp = moa::SplitPlan{};
  moa::AttnArgs a{Q, K, V, O, B, H, N_q, N_k, d_k, d_v, scale, static_cast<cudaStream_t>(stream)};
  char msg[256] = {0};
  rc = moa::launch_attn_fwd_bf16_split_noalloc(a, sp, msg, sizeof(msg));
  if (rc != MOA_OK) return moa::fail(rc, "%s", msg);
  moa::t_last_error[0] = '\0';
  return moa::debug_check(stream);
}

size_t moa_attn_bwd_workspace_bytes(int64_t B, int64_t H, int64_t N_q, int64_t N_k, int64_t d_k,
                                    int64_t d_v, int dtype) {
  (void)N_k;
  (void)d_k;
  (void)d_v;
  if ((dtype != MOA_BF16 && dtype != MOA_FP32) || B <= 0 || H <= 0 || N_q <= 0) return 0;
  if (moa::numel4(B, H, N_q + 127, 8) < 0) return 0;
  return moa::bwd_workspace_bytes(B, H, N_q);
}

int moa_attn_bwd(const void* Q, const void* K, const void* V, const void* O, const void* dO,
                 const float* LSE, void* dQ, void* dK, void* dV, int64_t B, int64_t H,
                 int64_t N_q, int64_t N_k, int64_t d_k, int64_t d_v, float scale, int dtype,
                 void* workspace, size_t workspace_bytes, void* stream) {
  return moa::bwd_call(Q, K, V, O, dO, LSE, dQ, dK, dV, B, H, N_q, N_k, d_k, d_v, scale, dtype,
                       workspace, workspace_bytes, stream, false);
}

int moa_attn_bwd_fused(const void* Q, const void* K, const void* V, const void* O,
                       const void* dO, const float* LSE, void* dQ, void* dK, void* dV, int64_t B,
                       int64_t H, int64_t N_q, int64_t N_k, int64_t d_k, int64_t d_v, float scale,
                       int dtype, void* workspace, size_t workspace_bytes, void* stream) {
  return moa::bwd_call(Q, K, V, O, dO, LSE, dQ, dK, dV, B, H, N_q, N_k, d_k, d_v, scale, dtype,
                       workspace, workspace_bytes, stream, true);
}

size_t moa_attn_bwd_fused_workspace_bytes(int64_t B, int64_t H, int64_t N_q, int64_t N_k,
                                          int64_t d_k, int64_t d_v, int dtype) {
  (void)N_k;
  if (dtype != MOA_BF16 || d_k != 64 || d_v != 64 || B < 1 || H < 1 || N_q < 1) return 0;
  if (moa::numel4(B, H, N_q + 127, 2 + d_k) < 0) return 0;
  return moa::bwd_fused_workspace_bytes(B, H, N_q, d_k);
}

int moa_qkv_proj(const void* X, const void* W, void* Q, void* K, void* V, int64_t B, int64_t N,
                 int64_t d_model, int64_t H, int64_t d_k, int64_t d_v, int dtype, void* stream) {
  if (!X || !W || !Q || !K || !V) return moa::fail(MOA_ERR_INVALID_ARG, "null tensor pointer");
  if (B <= 0 || N <= 0 || d_model <= 0 || H <= 0 || d_k <= 0 || d_v <= 0)
    return moa::fail(MOA_ERR_INVALID_ARG, "sizes must be >= 1");
  if (dtype != MOA_BF16)
    return moa::fail(MOA_ERR_UNSUPPORTED_DTYPE, "the projection takes bf16 tensors only (dtype %d)",
                     dtype);
  if ((d_k != 64 && d_k != 128) || (d_v != 64 && d_v != 128))
    return moa::fail(MOA_ERR_UNSUPPORTED_SHAPE, "d_k, d_v must be 64 or 128; got %lld, %lld",
                     (long long)d_k, (long long)d_v);
  if (d_model % 8 != 0)
    return moa::fail(MOA_ERR_MISALIGNED, "d_model must be a multiple of 8 (16-byte rows)");
  const int64_t ncol = 2 * H * d_k + H * d_v;
  const int64_t nx = moa::numel4(B, N, d_model, 1), nw = moa::numel4(d_model, ncol, 1, 1);
  const int64_t nq = moa::numel4(B, H, N, d_k), nv = moa::numel4(B, H, N, d_v);
  if (nx < 0 || nw < 0 || nq < 0 || nv < 0 || nx > INT64_MAX / 4 || nw > INT64_MAX / 4 ||
      nq > INT64_MAX / 4 || nv > INT64_MAX / 4)
    return moa::fail(MOA_ERR_UNSUPPORTED_SHAPE, "tensor sizes overflow 64-bit byte counts");
  if (B * N > 0x7fffffffLL || ncol > 0x7fffffffLL || d_model > 0x7fffffffLL)
    return moa::fail(MOA_ERR_UNSUPPORTED_SHAPE, "B*N, d_model and 2*H*d_k + H*d_v must be below 2^31");
  const void* ptrs[5] = {X, W, Q, K, V};
  for (const void* p : ptrs)
    if (reinterpret_cast<uintptr_t>(p) % 16 != 0)
      return moa::fail(MOA_ERR_MISALIGNED, "tensor pointer %p is not 16-byte aligned", p);
  const void* out[3] = {Q, K, V};
  const int64_t osz[3] = {nq * 2, nq * 2, nv * 2};
  for (int i = 0; i < 3; ++i) {
    if (moa::overlaps(out[i], osz[i], X, nx * 2) || moa::overlaps(out[i], osz[i], W, nw * 2))
      return moa::fail(MOA_ERR_INVALID_ARG, "an output overlaps X or W");
    for (int j = i + 1; j < 3; ++j)
      if (moa::overlaps(out[i], osz[i], out[j], osz[j]))
        return moa::fail(MOA_ERR_INVALID_ARG, "Q, K and V overlap");
  }
  moa::ProjArgs a{X, W, Q, K, V, B, N, d_model, H, d_k, d_v, static_cast<cudaStream_t>(stream)};
  char msg[256] = {0};
  const int rc = moa::launch_qkv_proj_bf16(a, msg, sizeof(msg));
  if (rc != MOA_OK) return moa::fail(rc, "%s", msg);
  moa::t_last_error[0] = '\0';
  return moa::debug_check(stream);
}

const char* moa_last_error(void) { return moa::t_last_error; }

int moa_get_device_status(void* stream) {
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess)
    return moa::fail(MOA_ERR_CUDA, "stream synchronize: %s", cudaGetErrorString(e));
  unsigned v = 0, vb = 0, vp = 0;
  e = moa::bf16_read_and_clear_status(&v);
  if (e == cudaSuccess) e = moa::bwd_read_and_clear_status(&vb);
  if (e == cudaSuccess) e = moa::proj_read_and_clear_status(&vp);
  if (e != cudaSuccess)
    return moa::fail(MOA_ERR_CUDA, "status word read: %s", cudaGetErrorString(e));
  v |= vb | vp;
  if (v != 0)
    return moa::fail(MOA_ERR_DEVICE_TIMEOUT, "a kernel wait ran out (status %u)", v);
  return MOA_OK;
}

int moa_selftest_wait_timeout(uint64_t limit_ns, void* stream) {
  if (limit_ns == 0 || limit_ns > 10000000000ull)
    return moa::fail(MOA_ERR_INVALID_ARG, "limit_ns must be in (0, 1e10]");
  cudaError_t e = moa::launch_wait_timeout_selftest(limit_ns, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess)
    return moa::fail(MOA_ERR_CUDA, "self-test launch: %s", cudaGetErrorString(e));
  return MOA_OK;
}

double moa_attn_flops(int64_t B, int64_t H, int64_t N_q, int64_t N_k, int64_t d_k, int64_t d_v) {
  return 2.0 * double(B) * double(H) * double(N_q) * double(N_k) * double(d_k + d_v);
}

double moa_attn_dnf_bytes(int64_t B, int64_t H, int64_t N_q, int64_t N_k, int64_t d_k,
                          int64_t d_v, int dtype) {
  const double elt = dtype == MOA_FP32 ? 4.0 : dtype == MOA_BF16 ? 2.0 : -1.0;
  if (elt < 0) return -1.0;
  return elt * double(B) * double(H) *
         (double(N_q) * d_k + double(N_k) * d_k + double(N_k) * d_v + double(N_q) * d_v);
}

int moa_attn_version(void) { return 100; }

}  // extern "C"
