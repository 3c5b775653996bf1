/*
 * fal_kernels.h - kernel-level C ABI of the same library (libfal.so), used to
 * check and time single steps of the hot path in isolation.  Every call only
 * enqueues work on `stream` (a cudaStream_t, NULL = legacy default stream) and
 * returns a FAL_* status from fal.h; all pointers are device pointers owned
 * by the caller.
 */
#ifndef FAL_KERNELS_H
#define FAL_KERNELS_H

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

#define FAL_ENGINE_TCGEN05 0       /* tcgen05/TMEM GEMM fed by TMA, one CTA per 128x256 tile */
#define FAL_ENGINE_SIMT 1         /* plain fp32-FMA tiled GEMM */
#define FAL_ENGINE_TCGEN05_PAIR 2  /* tcgen05/TMEM GEMM fed by TMA, CTA pairs (cta_group::2, 256x256 tiles; used by the model) */

/* C[M,N] = sum_k A(m,k) B(n,k) (+ bias[n]) : the contraction of every linear map
 * of the blocks (Eq. 1, Eq. 2) and of their gradients.
 *   A(m,k) = A[m*lda + k] if !a_mn_major else A[k*lda + m]
 *   B(n,k) = B[n*ldb + k] if !b_mn_major else B[k*ldb + n]
 * A, B: bf16 (in_f32 = 0) or fp32 (in_f32 = 1; SIMT engine only).
 * C: bf16 (c_f32 = 0) or fp32 (c_f32 = 1), row-major with leading dim ldc.
 * bias: fp32 [N] or NULL.  tcgen05 engines: A, B, C, bias 16-byte aligned,
 * lda/ldb multiples of 8, ldc a multiple of 4.  dev_err: device int that
 * receives a nonzero code if a bounded wait inside the kernel expires (may be NULL).
 * Errors: FAL_ERR_ARG (shape/alignment), FAL_ERR_CUDA (launch). */
int fal_kernel_gemm(int M, int N, int K, const void* A, long lda, int a_mn_major, const void* B, long ldb,
                    int b_mn_major, int in_f32, const float* bias, void* C, long ldc, int c_f32, int engine,
                    int* dev_err, void* stream);

/* Causal multi-head attention forward (MHA_i of Eq. 1/2, scaled by 1/sqrt(head_dim)).
 * qkv: bf16 [B*T, 3*H*hd] = [q | k | v] rows (head h at columns h*hd of each third);
 * ctx: bf16 [B*T, H*hd]; lse: fp32 [B, H, T] log-sum-exp of S*log2(e) (base 2).
 * hd must be 64 or 128.  Errors: FAL_ERR_ARG, FAL_ERR_UNSUPPORTED, FAL_ERR_CUDA. */
int fal_kernel_attention_fwd(int B, int T, int H, int hd, const void* qkv, void* ctx, float* lse, void* stream);

/* Backward of fal_kernel_attention_fwd: dqkv (bf16 [B*T, 3*H*hd]) from qkv,
 * ctx, lse and dctx (bf16 [B*T, H*hd]).  scratch: fp32 device buffer of at
 * least fal_kernel_attention_bwd_scratch(B, T, H, hd) floats, 256-byte aligned
 * (B*H*T rounded up to a multiple of 64, plus 64): overwritten, it receives
 * D = rowsum(dO * O) per query and head and then the work counter of the
 * backward kernel, cleared on `stream` before each launch. */
size_t fal_kernel_attention_bwd_scratch(int B, int T, int H, int hd);
int fal_kernel_attention_bwd(int B, int T, int H, int hd, const void* qkv, const void* ctx, const float* lse,
                             const void* dctx, void* dqkv, float* scratch, void* stream);

/* Allocation-free variant of fal_kernel_attention_bwd (the paper has no
 * counterpart: this is a deployment convenience).  It is for callers that may
 * not allocate device memory themselves -- for instance code running inside a
 * host framework that owns every device byte through its own pool and forbids
 * stray cudaMalloc/cudaFree (which also synchronize the device), or callers
 * that simply cannot pass a scratch buffer.  Same arguments as
 * fal_kernel_attention_bwd minus `scratch`; same results.
 *
 * Scratch comes from one fixed array of FAL_NOALLOC_ATTN_SCRATCH_FLOATS fp32
 * values (16 MiB) compiled into libfal.so: every GPU that loads the library
 * holds it until the process exits.  The call needs
 * fal_kernel_attention_bwd_scratch(B, T, H, hd) <= FAL_NOALLOC_ATTN_SCRATCH_FLOATS
 * (about B*H*T) and returns FAL_ERR_WORKSPACE (launching nothing) above that.  It never calls cudaMalloc,
 * cudaFree or any allocating routine.  Every call made while `stream` is not
 * being captured looks up the array's device address in the current device's
 * context (cudaGetSymbolAddress), so the address stays right after a device
 * reset; a call made while `stream` is being captured uses the address found
 * by an earlier call on the same device and context, and returns
 * FAL_ERR_STATE if there was none: make one call before any stream capture.
 * All calls share the one array and each call rewrites what it reads, so calls
 * that overlap on the GPU (different streams, or several host threads on one
 * device) race: serialize them. */
#define FAL_NOALLOC_ATTN_SCRATCH_FLOATS (4u * 1024u * 1024u)
int fal_kernel_attention_bwd_noalloc(int B, int T, int H, int hd, const void* qkv, const void* ctx, const float* lse,
                                     const void* dctx, void* dqkv, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* FAL_KERNELS_H */
