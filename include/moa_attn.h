/*
 * moa_attn: forward pass of scaled dot-product attention on sm_103a (GB300),
 * computed in the paper's Denotational Normal Form: no score, probability or
 * transposed-K array ever exists in device memory, so Q, K and V are read once
 * and O is written once.
 *
 * Paper: "Attention at the Theoretical Minimum: A Mathematics of Arrays
 * Framework for Memory-Optimal Transformer Kernels" (Mullin, Hains).
 *
 * Shared library: libmoa_attn.so (plain C ABI, no C++ or PyTorch types).
 * Every entry point is thread-safe; moa_last_error() is per calling thread.
 *
 * Environment (read once per process):
 *   MOA_WAIT_LIMIT_NS  limit of one bounded wait inside a kernel (default 1e9 ns)
 *   MOA_DEBUG_SYNC=1   every entry point synchronises its stream after launching and returns
 *                      MOA_ERR_CUDA or MOA_ERR_DEVICE_TIMEOUT for that call itself (debugging;
 *                      off by default, when errors surface at moa_get_device_status)
 */
#ifndef MOA_ATTN_H
#define MOA_ATTN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Element types of Q, K, V and O (all four share one type). */
enum moa_dtype {
    MOA_FP32 = 0, /* IEEE binary32; computed on CUDA cores in fp32 (no TF32) */
    MOA_BF16 = 1  /* bfloat16; tensor-core products, fp32 accumulation and softmax */
};

/* Status codes returned by every int-valued entry point. */
enum moa_status {
    MOA_OK = 0,
    MOA_ERR_INVALID_ARG = 1,       /* null pointer, a size <= 0, non-finite scale, O overlaps an input */
    MOA_ERR_UNSUPPORTED_DTYPE = 2, /* dtype is not one of enum moa_dtype */
    MOA_ERR_UNSUPPORTED_SHAPE = 3, /* head dimensions or sizes outside what the kernels take */
    MOA_ERR_MISALIGNED = 4,        /* a pointer not 16-byte aligned, or a row not a multiple of 16 bytes */
    MOA_ERR_CUDA = 5,              /* a CUDA runtime/driver call failed (message in moa_last_error) */
    MOA_ERR_DEVICE_TIMEOUT = 6     /* a kernel gave up on a wait and recorded it in the status word */
};

/*
 * moa_attn_fwd -- O = softmax(scale * Q K^T) V, one independent problem per (b, h).
 *
 * Defines: paper Section 4.1, Eq. (attention) with the max-subtracted softmax of
 * Eq. (stable_softmax) and the contraction with V of Eq. (output_dnf), computed
 * per (batch, head) slice as in the Remark of Section 4.2 (Eq. batched_mm).
 * For every b < B, h < H, i < N_q, c < d_v:
 *     s_k        = scale * sum_{j < d_k} Q[b,h,i,j] * K[b,h,k,j]      (k < N_k)
 *     O[b,h,i,c] = sum_k exp(s_k - max_k' s_k') / (sum_k'' exp(s_k'' - max_k' s_k')) * V[b,h,k,c]
 * The softmax runs over the key axis N_k; N_q and N_k may differ, as may d_k
 * and d_v.  No mask, dropout or bias.
 *
 * Arguments:
 *   Q  device pointer, [B, H, N_q, d_k], contiguous row-major, element type dtype (read only)
 *   K  device pointer, [B, H, N_k, d_k], same layout, read as stored (no transpose copy)
 *   V  device pointer, [B, H, N_k, d_v], same layout
 *   O  device pointer, [B, H, N_q, d_v], same element type; written, must not overlap Q, K, V
 *   B, H, N_q, N_k, d_k, d_v   sizes, each >= 1
 *   scale   multiplier of the scores, any finite value (the paper uses 1/sqrt(d_k))
 *   dtype   MOA_FP32 or MOA_BF16
 *   stream  a cudaStream_t (NULL = legacy default stream) of the current device
 *
 * Supported sizes:
 *   MOA_BF16: d_k, d_v in {64, 128}; N_q, N_k < 2^31; B*H < 2^31.
 *   MOA_FP32: 1 <= d_k, d_v <= 128 and d_k, d_v multiples of 4.
 * Alignment: Q, K, V, O 16-byte aligned.
 *
 * Ownership and memory: the caller owns all four buffers.  The call allocates
 * no device memory and uses no workspace; the kernels keep every intermediate
 * (scores, probabilities, running max and sum) in registers, shared memory and
 * tensor memory.
 *
 * Behaviour: asynchronous on `stream`; returns after the launch.  Arguments
 * are checked before anything is launched; on a non-OK return nothing was
 * launched and moa_last_error() describes the problem.  Kernel waits are
 * bounded: a wait that runs out records MOA_ERR_DEVICE_TIMEOUT in a device
 * status word (see moa_get_device_status) and the kernel returns early.
 */
int moa_attn_fwd(const void* Q, const void* K, const void* V, void* O, int64_t B, int64_t H,
                 int64_t N_q, int64_t N_k, int64_t d_k, int64_t d_v, float scale, int dtype,
                 void* stream);

/*
 * moa_attn_fwd_lse -- moa_attn_fwd, and also the log-sum-exp of every row's scores.
 *
 * Defines: O as in moa_attn_fwd, plus, for every b, h, i,
 *     LSE[b,h,i] = ln sum_{k < N_k} exp(s_k) = m + ln sum_k exp(s_k - m),  m = max_k s_k,
 * i.e. the logarithm of the softmax denominator of Eq. (stable_softmax) before its
 * max shift.  It is the per-row quantity a backward pass needs to rebuild the
 * weights exp(s_k - LSE) without the N_q x N_k matrix (paper Stage 5, Section 9),
 * and the one a merge of key ranges computed apart needs.
 *
 * Arguments: those of moa_attn_fwd, plus
 *   LSE  device pointer, float32 [B, H, N_q] contiguous, natural logarithm; written,
 *        4-byte aligned, must not overlap Q, K, V or O.  Owned by the caller.
 * Accuracy: bf16 path, the kernel's exp2/log2 in fp32 of the fp32-accumulated
 * scores (absolute error about 1e-5 * |LSE| + 1e-5); fp32 path, fp32 expf/logf.
 * Behaviour: as moa_attn_fwd; LSE adds 4 bytes per output row of traffic.
 */
int moa_attn_fwd_lse(const void* Q, const void* K, const void* V, void* O, float* LSE, int64_t B,
                     int64_t H, int64_t N_q, int64_t N_k, int64_t d_k, int64_t d_v, float scale,
                     int dtype, void* stream);

/*
 * moa_attn_bwd -- gradients of a scalar loss through O = softmax(scale * Q K^T) V.
 *
 * Defines: paper Stage 5 (Section 9) gives the query gradient as
 *     dL/dQ = dL/dO . V^T . J . K * scale,  J the row-wise Jacobian of the softmax;
 * with W the attention weights and dP = dO V^T, J applied to a row of dP is
 * w * (dP - w.dP), so for every (b, h):
 *     dS = W * (dO V^T - D),  D_i = sum_c dO[i,c] O[i,c]  (= w_i . dP_i),
 *     dQ = scale * dS K,  dK = scale * dS^T Q,  dV = W^T dO.
 * (dK and dV are the derivatives of the same expression with respect to its other two
 * operands.)  W is rebuilt from the scores and LSE; no N_q x N_k array is written to
 * device memory.
 *
 * Arguments:
 *   Q, K, V  device, the forward inputs (layouts of moa_attn_fwd), read only
 *   O        device, [B, H, N_q, d_v], the forward output for these inputs, read only
 *   dO       device, [B, H, N_q, d_v], dL/dO, read only
 *   LSE      device, float32 [B, H, N_q], the forward pass's log-sum-exp (moa_attn_fwd_lse)
 *   dQ, dK, dV  device, written: [B, H, N_q, d_k], [B, H, N_k, d_k], [B, H, N_k, d_v]
 *   B, H, N_q, N_k, d_k, d_v, scale   as for moa_attn_fwd (the same scale as the forward)
 *   dtype    MOA_BF16 (tensor cores, bf16 gradients) or MOA_FP32 (CUDA cores, fp32
 *            gradients, no TF32); all eight tensors share it
 *   workspace, workspace_bytes  device scratch of at least moa_attn_bwd_workspace_bytes(...)
 *            bytes, 16-byte aligned, owned by the caller; its contents need no initial value
 *   stream   a cudaStream_t of the current device
 * Supported sizes: those of moa_attn_fwd for the dtype (bf16: d_k, d_v in {64, 128}; fp32:
 * d_k, d_v <= 128 and multiples of 4).  Alignment: every tensor 16-byte aligned (LSE 4-byte).
 * Outputs and workspace must not overlap each other or any input.
 * Behaviour: asynchronous; three kernel launches on `stream` (per-row D and LSE in log2
 * units, then dK/dV, then dQ).  Allocates nothing.  Bounded waits as for moa_attn_fwd
 * (moa_get_device_status reports a timeout).  bf16: accumulation is fp32 in tensor memory and
 * the weights W and dS enter the tensor-core products rounded to bf16.  fp32: every step in
 * fp32 (expf for the weights).
 */
int moa_attn_bwd(const void* Q, const void* K, const void* V, const void* O, const void* dO,
                 const float* LSE, void* dQ, void* dK, void* dV, int64_t B, int64_t H,
                 int64_t N_q, int64_t N_k, int64_t d_k, int64_t d_v, float scale, int dtype,
                 void* workspace, size_t workspace_bytes, void* stream);

/*
 * moa_attn_bwd_workspace_bytes -- scratch bytes moa_attn_bwd needs: two fp32 values per
 * (b, h) and query row, rows padded to a multiple of 128, for either dtype (0 for an unknown
 * dtype or sizes < 1).
 */
size_t moa_attn_bwd_workspace_bytes(int64_t B, int64_t H, int64_t N_q, int64_t N_k, int64_t d_k,
                                    int64_t d_v, int dtype);

/*
 * moa_attn_bwd_fused -- the gradients of moa_attn_bwd from one tile kernel (bf16, d_k = d_v = 64).
 *
 * Defines: the same dQ, dK, dV as moa_attn_bwd (paper Stage 5, Section 9).  Each CTA owns a
 * block of 128 keys and forms the scores and dP of every query block once, computing the three
 * products dV += W^T dO, dK += dS^T Q and dQ_i = dS_i K from them (5 tile products per block
 * pair instead of moa_attn_bwd's 7).  The dQ_i of the key blocks are summed in an fp32
 * accumulator in the workspace with atomic additions, then scaled and rounded to bf16.
 * Arguments, layouts, alignment and overlap rules: those of moa_attn_bwd, with
 * dtype MOA_BF16 and d_k = d_v = 64 only, and a workspace of at least
 * moa_attn_bwd_fused_workspace_bytes(...) bytes.
 * Reproducibility: dK and dV are bitwise reproducible; the order of the fp32 additions into dQ
 * varies between runs, so dQ may differ in its last bits from run to run.  Callers that need
 * bit-identical gradients from identical inputs call moa_attn_bwd, whose three gradients are
 * all bitwise reproducible.
 * Errors: those of moa_attn_bwd; MOA_ERR_UNSUPPORTED_DTYPE for fp32, MOA_ERR_UNSUPPORTED_SHAPE
 * for other head dimensions.
 * Behaviour: asynchronous; three kernel launches on `stream` (per-row D and LSE with the
 * accumulator zeroed, the tile kernel, the dQ conversion).  Allocates nothing.
 */
int moa_attn_bwd_fused(const void* Q, const void* K, const void* V, const void* O,
                       const void* dO, const float* LSE, void* dQ, void* dK, void* dV, int64_t B,
                       int64_t H, int64_t N_q, int64_t N_k, int64_t d_k, int64_t d_v, float scale,
                       int dtype, void* workspace, size_t workspace_bytes, void* stream);

/*
 * moa_attn_bwd_fused_workspace_bytes -- scratch bytes moa_attn_bwd_fused needs: (2 + d_k) fp32
 * values per (b, h) and query row, rows padded to a multiple of 128 (0 unless dtype is
 * MOA_BF16 and d_k = d_v = 64, or for sizes < 1).
 */
size_t moa_attn_bwd_fused_workspace_bytes(int64_t B, int64_t H, int64_t N_q, int64_t N_k,
                                          int64_t d_k, int64_t d_v, int dtype);

/*
 * moa_qkv_proj -- the input projections Q = X W_Q, K = X W_K, V = X W_V in one pass.
 *
 * Defines: paper Section 4.1 (the problem setup: Q, K, V are the input sequence X projected
 * by learned weight matrices).  With the three weight matrices side by side in W,
 *     Q[b,h,n,j] = sum_c X[b,n,c] W[c, h*d_k + j]
 *     K[b,h,n,j] = sum_c X[b,n,c] W[c, H*d_k + h*d_k + j]
 *     V[b,h,n,j] = sum_c X[b,n,c] W[c, 2*H*d_k + h*d_v + j]
 * One tensor-core GEMM over all B*N tokens (X read once for all three); its epilogue stores
 * each result in the head-major layout moa_attn_fwd takes, so no permute copy follows.
 *
 * Arguments:
 *   X  device, [B, N, d_model] row-major, bf16, read only
 *   W  device, [d_model, 2*H*d_k + H*d_v] row-major, bf16 (columns W_Q | W_K | W_V), read only
 *   Q, K  device, written: [B, H, N, d_k];  V  device, written: [B, H, N, d_v]
 *   dtype  MOA_BF16 only; fp32 accumulation, outputs rounded to bf16 once
 *   stream a cudaStream_t of the current device
 * Supported sizes: d_k, d_v in {64, 128}; d_model a multiple of 8; B*N < 2^31.  Alignment:
 * all pointers 16-byte aligned.  Q, K, V must not overlap each other, X or W.
 * Behaviour: asynchronous, one launch, allocates nothing; bounded waits as moa_attn_fwd.
 * (The paper has no bias term and none is added.)
 */
int moa_qkv_proj(const void* X, const void* W, void* Q, void* K, void* V, int64_t B, int64_t N,
                 int64_t d_model, int64_t H, int64_t d_k, int64_t d_v, int dtype, void* stream);

/*
 * moa_attn_fwd_staged -- the same computation with host-resident inputs and output.
 *
 * Defines: as moa_attn_fwd (paper Section 4.1, Eq. attention).  Copies hQ, hK,
 * hV (host memory, ideally page-locked) into the caller's device buffers dQ,
 * dK, dV, runs the attention on them and copies dO back into hO.  The (b, h)
 * problems are independent (Remark in Section 4.2), so the call is pipelined
 * over contiguous ranges of heads (2 to 8 of them, about 16 MiB of inputs each
 * on average, the first and last ones smaller, at least one (b, h) each): the
 * copies of range c+1 into the
 * device run on a library-owned side stream while the kernel of range c runs
 * (on `stream` for even c, on a library-owned second compute stream for odd c,
 * so that one range's last wave of CTAs and the next range's first can share the
 * GPU), and each range's output goes back on a third side stream.  Work
 * already queued on `stream` completes before the first copy or kernel starts,
 * and `stream` completes only after the last copy back, so hO holds the result
 * once `stream` has been synchronised.  Sizes, layouts, dtype and alignment rules
 * are those of moa_attn_fwd; d* are device pointers owned by the caller, h* host
 * pointers owned by the caller.  Allocates no memory; the first call on a device
 * creates the three side streams and their events (kept until the process
 * exits).  Calls on one device enqueue under a lock and share the side streams.
 */
int moa_attn_fwd_staged(const void* hQ, const void* hK, const void* hV, void* hO, void* dQ,
                        void* dK, void* dV, void* dO, int64_t B, int64_t H, int64_t N_q,
                        int64_t N_k, int64_t d_k, int64_t d_v, float scale, int dtype,
                        void* stream);

/*
 * moa_attn_fwd_splitkv -- the same O as moa_attn_fwd, with the key axis split.
 *
 * Defines: paper Section 4.1, Eq. (attention).  The key axis [0, N_k) is cut into up to
 * `num_splits` contiguous ranges of whole 128-key blocks; each range is reduced on its own
 * (its own running maximum and sum, the online form of Eq. stable_softmax) into an
 * unnormalised fp32 partial output, and a second kernel merges the partials with the identity
 *     M = max_s m_s,   O = sum_s e^(m_s - M) O_s / sum_s e^(m_s - M) l_s,
 * which is Eq. stable_softmax over the union of the ranges.  Useful when B*H*N_q gives too
 * few 256-row query blocks to fill the GPU (long keys, short queries).
 *
 * Arguments: as moa_attn_fwd, plus
 *   num_splits       requested number of key ranges for every 256-row query block (>= 1;
 *                    fewer are used when N_k has fewer 128-key blocks; 1 runs the unsplit
 *                    kernel), or MOA_SPLITS_AUTO (see below)
 *   workspace        device pointer, 16-byte aligned, not overlapping any tensor; owned by the
 *                    caller; contents on entry are ignored and undefined afterwards
 *   workspace_bytes  its size; must be >= moa_attn_splitkv_workspace_bytes(...) with the same
 *                    num_splits (and, for MOA_SPLITS_AUTO, the same current device)
 * MOA_SPLITS_AUTO: the library chooses from the current device's SM count.  When the
 * B*H*ceil(N_q/256) query blocks (one SM's worth of work each) leave SMs idle, every block's
 * key axis is split so that the CTAs fill the SMs (at least two key blocks per range), when a
 * model of the split's cost predicts a saving of at least 15 %; with a full wave of blocks or more
 * nothing is split and the call is moa_attn_fwd (same bits).  moa_attn_split_plan reports
 * the choice.
 * MOA_FP32 has no split form: the call then computes the same result with moa_attn_fwd.
 * Errors: those of moa_attn_fwd; MOA_ERR_INVALID_ARG for num_splits < 0 or a missing, too
 * small or overlapping workspace; MOA_ERR_MISALIGNED for a misaligned workspace;
 * MOA_ERR_CUDA when MOA_SPLITS_AUTO cannot read the current device's SM count.
 * Asynchronous on `stream`; allocates nothing.  Launches the split kernel and the merge, or
 * the unsplit kernel alone.
 */
#define MOA_SPLITS_AUTO 0

int moa_attn_fwd_splitkv(const void* Q, const void* K, const void* V, void* O, int64_t B,
                         int64_t H, int64_t N_q, int64_t N_k, int64_t d_k, int64_t d_v,
                         float scale, int dtype, int num_splits, void* workspace,
                         size_t workspace_bytes, void* stream);

/*
 * moa_attn_splitkv_workspace_bytes -- bytes of workspace moa_attn_fwd_splitkv needs for these
 * sizes and this num_splits: splits * B*H*N_q * (4*d_v + 8) (fp32 partial rows plus a
 * running maximum and sum per row and split).  0 when no split happens, for MOA_FP32, for
 * invalid sizes, and for MOA_SPLITS_AUTO without a usable current device.
 */
size_t moa_attn_splitkv_workspace_bytes(int64_t B, int64_t H, int64_t N_q, int64_t N_k,
                                        int64_t d_k, int64_t d_v, int dtype, int num_splits);

/*
 * moa_attn_split_plan -- the schedule moa_attn_fwd_splitkv would run (host only).
 *
 * For these sizes and num_splits (>= 1, or MOA_SPLITS_AUTO) on a GPU of sm_count SMs
 * (<= 0: the current device, which then must be usable), writes through each non-null
 * pointer: *splits, the key ranges per split query block (1: nothing is split);
 * *key_blocks_per_split, the 128-key blocks in each range (the last may hold fewer); and
 * *whole_query_blocks, how many 256-row query blocks run unsplit (all or none of them).
 * Launches nothing.  Errors: MOA_ERR_INVALID_ARG for non-positive or overflowing sizes or
 * num_splits < 0; MOA_ERR_CUDA when sm_count <= 0 and no device answers.
 */
int moa_attn_split_plan(int64_t B, int64_t H, int64_t N_q, int64_t N_k, int num_splits,
                        int sm_count, int* splits, int* key_blocks_per_split,
                        int64_t* whole_query_blocks);

/* Size in bytes of the fixed device array used by moa_attn_fwd_splitkv_noalloc (16 MiB). */
#define MOA_NOALLOC_SCRATCH_BYTES ((size_t)16 << 20)

/*
 * moa_attn_fwd_splitkv_noalloc -- moa_attn_fwd_splitkv for callers that cannot allocate.
 *
 * The paper has no counterpart to this entry point; it is a convenience of this library.
 * Some callers have no way to hand this library scratch memory: a framework that owns every
 * byte of device memory through its own pool and allows no other allocation, a serving loop
 * that must not call cudaMalloc because the call synchronises the device and stalls other
 * work, or a plugin interface that passes only the input and output buffers.  For them this
 * entry point takes no workspace and allocates nothing (no cudaMalloc, cudaFree or allocating
 * library routine): the fp32 partial rows and per-row maxima and sums of the split live in a
 * fixed array of MOA_NOALLOC_SCRATCH_BYTES inside the library, which every GPU that loads the
 * library holds until the process exits.
 *
 * Result and arguments: exactly those of moa_attn_fwd_splitkv without the workspace; the
 * caller still passes Q, K, V and O.  A split whose partials need more than
 * MOA_NOALLOC_SCRATCH_BYTES (splits * B*H*N_q * (4*d_v + 8) bytes) is rejected with
 * MOA_ERR_UNSUPPORTED_SHAPE and a message naming both sizes; nothing is launched.  With
 * MOA_SPLITS_AUTO a plan that would not fit runs unsplit instead.
 *
 * The first call on a device looks up that device's address of the array (once per device,
 * with the device current); make that first call before any stream capture on the device.
 * All calls on a device share the one array and it keeps the last call's contents: calls that
 * can run at the same time on the GPU (e.g. on unordered streams) race on it and must be
 * serialised by the caller.  Nothing in the array needs to start at zero.
 * Asynchronous on `stream`.
 */
int moa_attn_fwd_splitkv_noalloc(const void* Q, const void* K, const void* V, void* O,
                                 int64_t B, int64_t H, int64_t N_q, int64_t N_k, int64_t d_k,
                                 int64_t d_v, float scale, int dtype, int num_splits,
                                 void* stream);

/*
 * moa_last_error -- human-readable reason for the last non-OK status returned
 * on the calling thread ("" if none).  The string is owned by the library and
 * stays valid until the next call on the same thread.
 */
const char* moa_last_error(void);

/*
 * moa_get_device_status -- synchronises `stream`, then returns and clears the
 * device status word that bounded waits write on timeout: MOA_OK if no kernel
 * timed out since the last call, MOA_ERR_DEVICE_TIMEOUT otherwise,
 * MOA_ERR_CUDA if the synchronisation itself failed.
 */
int moa_get_device_status(void* stream);

/*
 * moa_selftest_wait_timeout -- diagnostic for the failure path of the kernels' bounded waits
 * (no counterpart in the paper; it exists so that timeout handling can be tested without
 * hanging or faulting a GPU).  Launches one warp on `stream` whose thread waits, with the same
 * bounded wait the attention kernel uses, on an mbarrier phase that nothing completes.  After
 * limit_ns nanoseconds (0 < limit_ns <= 1e10) the wait gives up and records
 * MOA_ERR_DEVICE_TIMEOUT in the device status word; the kernel then returns normally and the
 * context stays usable.  Read the result with moa_get_device_status.  Asynchronous; allocates
 * nothing.  Returns MOA_ERR_INVALID_ARG for a limit out of range, MOA_ERR_CUDA if the launch
 * failed.
 */
int moa_selftest_wait_timeout(uint64_t limit_ns, void* stream);

/*
 * moa_attn_flops -- floating-point operations of the two contractions,
 * 2*B*H*N_q*N_k*(d_k + d_v): the two matrix products of Eq. (attention),
 * Q K^T and the product of the weights with V (exponentials, maxima and the
 * division are not counted).
 */
double moa_attn_flops(int64_t B, int64_t H, int64_t N_q, int64_t N_k, int64_t d_k, int64_t d_v);

/*
 * moa_attn_dnf_bytes -- the memory-traffic lower bound of the paper (Theorem
 * lower_bound, Section 6.5): read Q, K, V once and write O once,
 *     elt * B * H * (N_q*d_k + N_k*d_k + N_k*d_v + N_q*d_v)
 * with elt = 4 (MOA_FP32) or 2 (MOA_BF16); returns -1 for an unknown dtype.
 */
double moa_attn_dnf_bytes(int64_t B, int64_t H, int64_t N_q, int64_t N_k, int64_t d_k,
                          int64_t d_v, int dtype);

/* moa_attn_version -- library version, major*10000 + minor*100 + patch. */
int moa_attn_version(void);

#ifdef __cplusplus
}
#endif

#endif /* MOA_ATTN_H */
