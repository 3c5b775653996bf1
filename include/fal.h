/*
 * fal.h - C ABI of the GB300 (sm_103a) training hot path for decoder stacks of
 * GPT (Pre-LN), FAL and FAL+ blocks ("First Attentions Last", arXiv 2510.14614).
 *
 * Block equations implemented (paper section / equation):
 *   GPT  (Eq. 1, Sec. 2):   X_{i+1} = X_i + MHA_i(LN(X_i)) + MLP_i(LN(X_i + MHA_i(LN(X_i))))
 *   FAL  (Eq. 2, Sec. 4.1): X_{i+1} = X_i + MHA_i(LN(X_i)) + MLP_i(LN(X_i) + LN_F(MHA_1(LN(X_1))))
 *        LN(X_i) is the same LayerNorm output that feeds MHA_i; LN_F is one
 *        LayerNorm shared by all blocks (the first attention output is normalised
 *        a single time, Sec. 4.1).
 *   FAL+ (Sec. 5, App. D.1): block 1 is the standard block; block i >= 2 feeds
 *        MLP_i(LN(X_i + MHA_i(LN(X_i))) + LN_{F,i}(MHA_1(LN(X_1)))).
 * The paper's comparison blocks, built from the same kernels:
 *   Parallel (Sec. 5.1, GPT-J style): X_i + MHA_i(LN(X_i)) + MLP_i(LN(X_i)).
 *   Ablation1 (App. D): X_i + MHA_i(LN(X_i)) + MLP_i(LN(X_i) + LN_{A,i}(MHA_i(LN(X_i)))).
 *   Ablation2 (App. D): block 1 standard, every later block Parallel.
 *   FAL+ reusing block k (App. D, "Ablation with Other Layers"): blocks 1..k
 *        standard, block i > k adds LN_{F,i}(MHA_k(LN(X_k))) (reuse_layer = k).
 * GPT-2 conventions: learned positions, tied LM head, final LN, biases on every
 * linear map, tanh GELU, LN eps 1e-5, causal attention scaled by 1/sqrt(head_dim),
 * mean token cross-entropy; AdamW with bias correction and decoupled weight
 * decay on matrices and embeddings (App. A: lr 1e-4, weight decay 1e-3).
 *
 * Conventions for every entry point:
 *   - Return 0 (FAL_OK) or a positive FAL_ERR_* code; nothing aborts or throws.
 *   - A non-OK return leaves a message retrievable with fal_last_error().
 *   - "device or host" pointers are resolved through unified addressing
 *     (cudaMemcpyDefault); host memory should be pinned for asynchronous copies.
 *   - All work is enqueued on the caller's streams; only calls that return a
 *     host value (a loss, parameters, a tap) or fal_sync() synchronize.
 */
#ifndef FAL_H
#define FAL_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* status codes */
#define FAL_OK 0
#define FAL_ERR_ARG 1         /* null pointer, bad shape, bad alignment, token id out of range */
#define FAL_ERR_STATE 2       /* call order (e.g. backward without a forward) */
#define FAL_ERR_WORKSPACE 3   /* workspace smaller than fal_workspace_size(), or a problem larger than the
                                 fixed scratch of fal_kernel_attention_bwd_noalloc (fal_kernels.h) */
#define FAL_ERR_CUDA 4        /* a CUDA runtime/driver call failed */
#define FAL_ERR_TIMEOUT 5     /* a bounded device-side wait expired (kernel returned early) */
#define FAL_ERR_UNSUPPORTED 6 /* configuration valid but not implemented on this path */

/* block variants */
#define FAL_GPT 0
#define FAL_FAL 1
#define FAL_FALPLUS 2
#define FAL_PARALLEL 3
#define FAL_ABLATION1 4
#define FAL_ABLATION2 5

/* arithmetic of the path */
#define FAL_BF16 0        /* bf16 tensor-core GEMMs/attention, fp32 accumulation, fp32 residual */
#define FAL_FP32_DEBUG 1  /* plain fp32 FMA kernels everywhere (no TF32), for parity at 1e-4 */

/* schedule of the two branches of a FAL block (Sec. 4.2 "Single-GPU Acceleration") */
#define FAL_SCHED_SERIAL 0      /* one stream, MHA branch then MLP branch */
#define FAL_SCHED_TWO_STREAM 1  /* FAL blocks i >= 2: MHA branch on stream_side, MLP on stream_main */

typedef struct fal_config {
    int variant;      /* FAL_GPT | FAL_FAL | FAL_FALPLUS | FAL_PARALLEL | FAL_ABLATION1 | FAL_ABLATION2 */
    int layers;       /* L >= 1 */
    int d_model;      /* d, multiple of 8 (bf16) or 4 (fp32 debug) */
    int heads;        /* H, d % H == 0; bf16 needs head_dim in {64, 128} */
    int d_ff;         /* MLP width, multiple of 8 */
    int seq;          /* T >= 1 (positions table size) */
    int batch;        /* B >= 1 */
    int vocab;        /* V >= 2 */
    int precision;    /* FAL_BF16 | FAL_FP32_DEBUG */
    int schedule;     /* FAL_SCHED_* */
    float lr, beta1, beta2, eps, weight_decay;  /* AdamW */
    int reuse_layer;  /* FAL+ only: block k (1-based) whose attention output later blocks add;
                         0 or 1 = the first block (FAL+ as defined); other variants need 0 or 1 */
    float clip_norm;  /* > 0: before AdamW, scale the gradients so that their global L2 norm is
                         at most clip_norm (App. A clips at 1.0); 0 = no clipping.  With
                         clipping, fal_train_step cannot update weights inside the gradient
                         GEMMs (the norm needs every gradient first) and runs AdamW after
                         the backward, like fal_step. */
    int kv_heads;     /* grouped-query attention (App. E): key/value heads, each shared by
                         heads / kv_heads query heads; 0 = heads (multi-head attention).
                         The fused QKV matrix then has d_model + 2 * kv_heads * head_dim rows. */
    int head_chunk;   /* 0: the LM head stores the logits [B*T, vocab] once and the cross-entropy
                         reads them.  > 0 (a multiple of 64): the logits are never stored whole.
                         The forward's LM-head GEMM reduces each row to its log-sum-exp and
                         target logit in the epilogue; the backward recomputes the logits
                         head_chunk vocabulary columns at a time, turns them into the loss
                         gradient in the epilogue and feeds that chunk to the weight and input
                         gradients.  The workspace then holds two [B*T, head_chunk] chunks
                         instead of two [B*T, vocab] arrays, for one more LM-head GEMM per
                         step.  The "logits" tap is unavailable in this mode. */
} fal_config;

typedef struct fal_tensor_info {
    char name[48];   /* e.g. "wte", "h3.attn.w_qkv", "lnF.g" (layers numbered from 0); per-block
                        LayerNorms: ln1, ln2 (GPT-style MLP input), lnF (FAL+ first-attention
                        term), lnA (Ablation1 own-attention term) */
    size_t offset;   /* first element inside the flat fp32 parameter buffer */
    size_t numel;
    int ndim;        /* 1 or 2 */
    int shape[2];    /* matrices are [out, in], row-major */
    int decayed;     /* 1 if AdamW applies weight decay */
} fal_tensor_info;

typedef struct fal_handle fal_handle;

/* Bytes of device workspace a configuration needs (parameters, gradients,
 * AdamW moments, bf16 weight copy, activations, scratch).  Error: FAL_ERR_ARG. */
int fal_workspace_size(const fal_config* cfg, size_t* bytes);

/* Creates a model inside `workspace` (device memory owned by the caller, at
 * least fal_workspace_size() bytes, 256-byte aligned).  stream_main and
 * stream_side are cudaStream_t values owned by the caller (may be equal; NULL
 * means the legacy default stream).  Parameters start at zero: load them with
 * fal_set_params().  The handle owns only host memory, CUDA events and TMA
 * descriptors; fal_destroy() releases them. */
int fal_create(const fal_config* cfg, void* workspace, size_t bytes,
               void* stream_main, void* stream_side, fal_handle** out);
void fal_destroy(fal_handle* h);

/* Forward pass and mean cross-entropy loss over B*T positions.
 * tokens, targets: int32 [B, T] row-major, device or host.  loss_host may be
 * NULL (the loss stays on the device, see fal_get_loss); otherwise the call
 * synchronizes and writes it.  Token ids outside [0, V) are zeroed and
 * reported as FAL_ERR_ARG at the next synchronizing call. */
int fal_forward(fal_handle* h, const int32_t* tokens, const int32_t* targets, float* loss_host);

/* Forward-only pass for inference: App. E times the forward step without
 * gradients as the time to first token.  Runs the
 * stack over tokens [B, T] (int32 row-major, device or host), the final
 * LayerNorm, and the tied LM head for the last position of every sequence
 * only.  last_logits: fp32 [B, V] row-major, device or host, or NULL to leave
 * them on the device; a non-NULL pointer makes the call synchronize.  No loss
 * and no backward state: a following fal_backward returns FAL_ERR_STATE. */
int fal_prefill(fal_handle* h, const int32_t* tokens, float* last_logits);

/* Gradients of the last forward's loss into the flat fp32 gradient buffer
 * (overwritten, not accumulated).  FAL_ERR_STATE without a preceding forward. */
int fal_backward(fal_handle* h);

/* One AdamW step over the flat parameter buffer; also refreshes the bf16
 * weight copy.  FAL_ERR_STATE without a preceding backward. */
int fal_step(fal_handle* h);

/* forward + backward + step. */
int fal_train_step(fal_handle* h, const int32_t* tokens, const int32_t* targets, float* loss_host);

/* Global L2 norm of the gradients before clipping, as computed by the last
 * fal_step / fal_train_step with clip_norm > 0 (synchronizes).  FAL_ERR_STATE
 * if no clipped step ran yet. */
int fal_get_grad_norm(fal_handle* h, float* norm_host);

/* Waits for both streams and reports device-side errors (token range, wait timeouts). */
int fal_sync(fal_handle* h);

/* Loss of the last forward (synchronizes). */
int fal_get_loss(fal_handle* h, float* loss_host);

/* Parameter table: n_tensors entries describing the flat buffer of n_elems floats. */
int fal_param_count(fal_handle* h, int* n_tensors, size_t* n_elems);
int fal_param_info(fal_handle* h, int idx, fal_tensor_info* info);

/* Copy the whole flat fp32 buffer (n must equal n_elems); src/dst device or host.
 * fal_set_params also refreshes the bf16 weight copy and resets AdamW state. */
int fal_set_params(fal_handle* h, const float* src, size_t n);
int fal_get_params(fal_handle* h, float* dst, size_t n);
int fal_get_grads(fal_handle* h, float* dst, size_t n);

/* AdamW state, for checkpoint / resume: the first and second moments (flat
 * fp32 buffers laid out like the parameters, n == n_elems; src/dst device or
 * host, either pointer may be NULL to skip that buffer) and the number of
 * optimizer steps taken so far (the next step's bias corrections use
 * step + 1).  fal_set_opt_state does not touch the parameters; call it after
 * fal_set_params, which resets the state to zero. */
int fal_get_opt_state(fal_handle* h, float* m, float* v, size_t n, long long* step);
int fal_set_opt_state(fal_handle* h, const float* m, const float* v, size_t n, long long step);

/* Debug view of a saved activation of the last forward, converted to fp32.
 * name in {"X","u","m","qkv","ctx","h","g","Y","a1","xf","logits"}; layer is
 * ignored for the global ones ("a1","xf","logits"; "X" with layer==L is the
 * stack output).  n must equal the tensor's element count (logits: B*T*V). */
int fal_get_tap(fal_handle* h, const char* name, int layer, float* dst, size_t n);

/* Live kernel timing for roofline reports.  While enabled (enable = 1), every
 * GEMM and attention launch of this handle is bracketed by CUDA events on its
 * own stream (no synchronization is added); enable = 2 brackets every launch
 * (LayerNorm, column reductions, cross-entropy too) for fal_profile_timeline.  fal_profile_read() synchronizes,
 * sums the event intervals since the last read, and resets the counters.
 * FLOPs are algorithmic: 2*M*N*K per GEMM; causal attention counts half of
 * the dense 4*B*H*T^2*hd forward and twice that for the backward. */
typedef struct fal_profile {
    double gemm_ms, gemm_flops;
    long long gemm_launches;
    double attn_ms, attn_flops;
    long long attn_launches;
} fal_profile;
int fal_profile_enable(fal_handle* h, int enable);
int fal_profile_read(fal_handle* h, fal_profile* out);

/* Per-launch view of the same records (GEMM, attention, LayerNorm, column
 * reductions, cross-entropy), in issue order, times in ms relative to the
 * start of the first record; stream 0 is the main stream, 1 the side stream.
 * kind: 0 GEMM, 1 attention forward, 2 attention backward, 3 other.
 * Synchronizes; does not reset the records (fal_profile_read does).  Fills at
 * most cap entries of the caller's array and sets *n to their count. */
typedef struct fal_launch_record {
    double start_ms, end_ms, flops;
    int kind, stream;
    char label[48];
} fal_launch_record;
int fal_profile_timeline(fal_handle* h, fal_launch_record* out, int cap, int* n);

/* Number of kernels this library has launched in this process (all handles). */
long long fal_launch_count(void);

/* Test hook for the library's bounded device waits (the paper has no
 * counterpart).  With rows >= 0, every CTA of the row-streaming LayerNorm
 * kernels stops loading rows after `rows` of them, so that the kernel's
 * waits for the missing rows expire after wait_ns nanoseconds (the default
 * budget of about one second when wait_ns <= 0); the kernel then records a
 * timeout and returns, and the next synchronizing call reports
 * FAL_ERR_TIMEOUT.  rows < 0 restores normal operation (and the default
 * budget).  Process-wide; for tests only: results computed meanwhile are
 * invalid. */
int fal_debug_layernorm_stall(int rows, long long wait_ns);

/* Message for the last failed call on this handle (never NULL). */
const char* fal_last_error(const fal_handle* h);
const char* fal_status_string(int status);

#ifdef __cplusplus
}
#endif
#endif /* FAL_H */
