// Host-side interface between the translation units of libfal.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>
#include <string>

namespace fal {

// Device error word codes (written with atomicCAS so the first error sticks).
enum DevErr { DEV_OK = 0, DEV_ERR_TOKEN = 1, DEV_ERR_TIMEOUT = 2 };

// ---------------------------------------------------------------- GEMM
// Every GEMM of the path is C[M,N] = sum_k A(m,k) * B(n,k) followed by an
// epilogue.  A operand element (m,k) lives at A[m*ld + k] (K-major) or
// A[k*ld + m] (MN-major); B operand element (n,k) at B[n*ld + k] (K-major) or
// B[k*ld + n] (MN-major).  A group may chain two K segments (two operand pairs
// summed into one accumulator: the fused [ctx | g] x [W_o ; W_down] residual
// GEMM), and one launch may run up to four independent groups (tiles in group
// order).
// EPI_ADAMW: the GEMM computes the gradient of a weight matrix (stored to `out`,
// fp32, OUT_F32) and the epilogue also applies AdamW to that weight in place.
// EPI_CE_STATS / EPI_CE_GRAD: the LM head's cross-entropy without stored
// logits (fields ce_* below).
enum EpiOp { EPI_NONE = 0, EPI_GELU = 1, EPI_DGELU = 2, EPI_ADAMW = 3, EPI_CE_STATS = 4, EPI_CE_GRAD = 5 };
enum OutMode { OUT_ACT = 0, OUT_F32 = 1, OUT_F32_ACCUM = 2 };

struct EpiParams {
  int op;        // EpiOp
  int out_mode;  // OutMode for `out`
  void* out;  long ldo;
  void* out2; long ldo2;     // GELU: gelu(v) (activation type); pre_f32: fp32 copy of acc+bias
  int pre_f32;               // write out2 = acc + bias before the residual is added
  const float* bias;  const float* bias2;   // per-column (N) fp32 vectors, may be null
  const float* resid; long ldr;             // fp32 [M, N] added after pre_f32
  const float* resid2; long ldr2;
  const void* aux; long ldx;                // DGELU: pre-activation h (activation type)
  // ADAMW: fp32 master weights, moments and the bf16 copy the GEMMs read (or
  // null), all [M, N] with row pitch ldo; decoupled weight decay wd; rbc1 and
  // rbc2 are 1 / (1 - beta^t).
  float* opt_p; float* opt_m; float* opt_v; void* opt_sh;
  float opt_lr, opt_b1, opt_b2, opt_eps, opt_wd, opt_rbc1, opt_rbc2;
  // Optional per-head row dot products of the (activation-rounded) output with
  // rd_src (same [M, N] layout, row pitch rd_ld), for the attention backward's
  // D = rowsum(dO * O): rd_out[((r / rd_T) * rd_H + c / rd_hd) * rd_T + r % rd_T]
  // = sum over the head's columns c.  tcgen05 path only.
  const void* rd_src; long rd_ld; float* rd_out; int rd_hd, rd_T, rd_H;
  // Ordered split-K over one output (tcgen05 one-CTA engine, TMA outputs):
  // an ORD_SIGNAL group stores its tiles and then publishes, per tile and
  // epilogue warp, ord_flags[...] = ord_epoch; a later ORD_WAIT group of the
  // same launch and shape (OUT_F32_ACCUM) waits for that flag before it adds
  // its partial, so the sum is formed in a fixed order.  ord_cap: ints in
  // ord_flags; ord_epoch must differ from every value left by earlier launches.
  int ord_role; int* ord_flags; int ord_cap; int ord_epoch;
  // Cross-entropy of the LM head (C = logits, column c is vocabulary entry
  // ce_v0 + c; the target of row r is ce_tgt[r]):
  // EPI_CE_STATS stores nothing to `out`; for every row and slice of
  // kCeSliceTc (tcgen05) or kCeSliceSimt (SIMT) columns it writes
  // ce_stats[slice * ce_ld + r] = (max, sum of exp(x - max)) over the slice's
  // columns below N (ce_ld >= M), and the logit of the row's target, when it
  // lies in [ce_v0, ce_v0 + N), to ce_tlogit[r].  EPI_CE_GRAD stores out = (exp(x - ce_lse[r]) - [ce_v0 + c ==
  // ce_tgt[r]]) * ce_scale (activation type): the gradient of the mean loss.
  const int* ce_tgt; const float* ce_lse; float2* ce_stats; float* ce_tlogit; long ce_ld; int ce_v0; float ce_scale;
};
enum OrdRole { ORD_NONE = 0, ORD_SIGNAL = 1, ORD_WAIT = 2 };

struct GemmOperand { const void* ptr; long ld; int mn_major; };
struct GemmSeg { GemmOperand A, B; int K; };
struct GemmGroupDesc { int M, N; int nseg; GemmSeg seg[2]; EpiParams epi; };
constexpr int kMaxGemmGroups = 4;
struct GemmCall { int ngroups; GemmGroupDesc g[kMaxGemmGroups]; };

// Plain fp32-FMA tiled GEMM (debug precision; also a GPU cross-check).
// in_bf16: operands are bf16 (else fp32); act_bf16: activation outputs bf16.
int gemm_simt(const GemmCall& c, int in_bf16, int act_bf16, cudaStream_t s, std::string* msg);
// tcgen05/TMEM GEMM fed by TMA (bf16 operands, fp32 accumulation, bf16 activations).
int gemm_tc(const GemmCall& c, int* dev_err, cudaStream_t s, std::string* msg);
// TC_ONE: one CTA per 128x256 tile; TC_PAIR: CTA pairs (cta_group::2, 256x256
// tiles).
enum TcKind { TC_ONE = 0, TC_PAIR = 1 };
int gemm_tc_engine(const GemmCall& c, int kind, int* dev_err, cudaStream_t s, std::string* msg);
// Columns per EPI_CE_STATS slice: 128 for the tcgen05 engines (one epilogue
// warp's half of a 256-column tile), 64 for the SIMT GEMM (its tile width).
constexpr int kCeSliceTc = 128, kCeSliceSimt = 64;

// ---------------------------------------------------------------- attention
// qkv: activation [B*T, 3*H*hd] (q | k | v, head-major inside each third);
// ctx: activation [B*T, H*hd]; lse: fp32 [B, H, T] in log2 units of the scaled scores.
// bf16: tcgen05 kernel (dev_err receives DEV_ERR_TIMEOUT if a bounded wait expires);
// fp32 debug: one thread per query row.
// Hkv: key/value heads (grouped-query attention, qkv rows of (H + 2 Hkv) * hd);
// 0 means H (multi-head attention).
int attn_fwd(int act_bf16, int B, int T, int H, int hd, const void* qkv, void* ctx, float* lse, int* dev_err,
             cudaStream_t s, std::string* msg, int Hkv = 0);
// dvec: fp32 scratch of attn_bwd_scratch_floats(B, T, H) floats: D = rowsum(dO * O)
// in [B, H, T] layout, then the backward kernel's work counter; d_ready: dvec
// already holds D (computed by the GEMM that produced dctx).
inline size_t attn_bwd_scratch_floats(long B, long T, long H) {
  return (size_t)((B * H * T + 63) / 64 * 64 + 64);
}
int attn_bwd(int act_bf16, int B, int T, int H, int hd, const void* qkv, const void* ctx,
             const float* lse, const void* dctx, void* dqkv, float* dvec, int* dev_err,
             cudaStream_t s, std::string* msg, int d_ready = 0, int Hkv = 0);

// ---------------------------------------------------------------- elementwise
struct LnFwdArgs {
  int rows, d;
  const float* x;                       // fp32 [rows, d]
  const float* gamma; const float* beta;  // null => no affine
  void* out;                            // activation [rows, d] or null
  float* out_f32;                       // fp32 [rows, d] or null
  float* mean; float* rstd;             // [rows] or null
  // out2 = LN(x)*gamma+beta + add_src*add_g + add_b  (activation), if out2 != null
  void* out2; const float* add_src; const float* add_g; const float* add_b;
  int* err;                             // receives DEV_ERR_TIMEOUT if a bounded wait expires (may be null)
};
int ln_fwd(int act_bf16, const LnFwdArgs& a, cudaStream_t s);
// Sums nchunk per-chunk partial column sums [nchunk][nslot][d] into the
// outputs (slot 0 -> out0 and out0b, slot 1 -> out1, slot 2 -> out2 and out2b).
int colsum_finish(const float* partial, int nchunk, int d, float* out1, float* out0, float* out0b, int accumulate,
                  cudaStream_t s, int nslot = 2, float* out2 = nullptr, float* out2b = nullptr);

struct LnBwdArgs {
  int rows, d;
  const float* dy; const float* dy2;    // gradient of the LN output (dy2 may be null)
  const float* x; const float* mean; const float* rstd; const float* gamma;  // gamma null => 1
  const float* dres;                    // added to dx (residual branch), may be null
  float* dx;                            // fp32 out
  void* dx_act;                         // activation copy (may be null)
  // Optional fused column sums of the affine parameters' gradients over the
  // rows: cs_out1 (+)= sum (dy + dy2) * xhat, cs_out0 (+)= sum (dy + dy2).
  // cs_part: scratch of colsum_partial_floats(d) floats.
  float* cs_part; float* cs_out1; float* cs_out0; int cs_accumulate;
  // Optional column sums of the output dx itself (the bias gradients of the
  // linear maps that produced the LN input's gradient): dxs_out and dxs_out2
  // (+)= sum dx, with the same accumulate flag.  Needs cs_part.
  float* dxs_out; float* dxs_out2;
  int* err;                             // receives DEV_ERR_TIMEOUT if a bounded wait expires (may be null)
};

// Test hook for the bounded waits of the row-streaming LayerNorm kernels: when
// stall_rows >= 0 each CTA's producer stops after that many rows, so that the
// consumers' waits expire (after wait_ns, or the default budget when <= 0);
// the kernels then report DEV_ERR_TIMEOUT and return.  stall_rows < 0: off.
void ln_debug_stall(int stall_rows, long long wait_ns);
int ln_bwd(int act_bf16, const LnBwdArgs& a, cudaStream_t s);
// Row-streaming LayerNorm kernels (two persistent CTAs per SM, rows staged in
// shared memory by bulk copies); 1 when the shape or alignment does not fit
// them (the caller then uses the warp-per-row kernels).
int ln_fwd_bulk(int act_bf16, const LnFwdArgs& a, cudaStream_t s);
int ln_bwd_bulk(int act_bf16, const LnBwdArgs& a, cudaStream_t s);

// Column sums over rows: s1[c] = sum_r a(r,c)*b(r,c), s0[c] = sum_r a(r,c)
// with a = src (+ src2), b = LN-normalised x (bmode 1) or bsrc (bmode 2).
struct ColsumArgs {
  int rows, d;
  const void* src; int src_act;   // src_act: src is the activation type (else fp32)
  long ld;
  const float* src2;              // fp32, same layout, may be null
  int bmode; const float* x; const float* mean; const float* rstd; const float* bsrc;
  float* partial;                 // scratch [nchunk, 2, d]
  float* out1; float* out0; float* out0b;  // destinations (may be null)
  int accumulate;                 // add into destinations instead of storing
};
int colsum(int act_bf16, const ColsumArgs& a, cudaStream_t s);
size_t colsum_partial_floats(int d);  // = kMaxColsumChunks * 3 * d
constexpr int kMaxColsumChunks = 384;  // most per-chunk partials any column reduction writes

int embed_fwd(int rows, int T, int d, int V, const int32_t* tok, const float* wte, const float* wpe,
              float* X, int* err, cudaStream_t s);
int embed_bwd(int B, int T, int d, int V, const int32_t* tok, const float* dX, float* dwte, float* dwpe,
              cudaStream_t s);
// logits/dlogits: activation [rows, ld] with V valid columns; loss_rows fp32 [rows].
int cross_entropy(int act_bf16, int rows, int V, long ld, const void* logits, const int32_t* tgt,
                  void* dlogits, float* loss_rows, float* loss, int* err, cudaStream_t s);
// Loss of the chunked LM head from the EPI_CE_STATS output of the logits GEMM
// (nslices slices per row, slice-major with row pitch ld): lse and loss_rows
// fp32 [rows], loss = their mean; a target outside [0, V) sets DEV_ERR_TOKEN.
int ce_combine(int rows, int nslices, const float2* stats, long ld, const float* tlogit, const int32_t* tgt, int V,
               float* lse, float* loss_rows, float* loss, int* err, cudaStream_t s);
// dst += src * colvec (per column), fp32 [rows, d]
int add_scaled_cols(int rows, int d, const float* src, const float* colvec, float* dst, cudaStream_t s);
// gscale: device scalar multiplying every gradient (gradient clipping), or null.
int adamw(size_t n, size_t n_decay, float* p, const float* g, float* m, float* v, void* shadow_bf16,
          float lr, float beta1, float beta2, float eps, float wd, float bc1, float bc2, cudaStream_t s,
          const float* gscale = nullptr);
// Global L2 norm of g[0..n) (n a multiple of 4) and the clipping factor
// min(1, max_norm / norm), both written to device scalars; deterministic
// (fixed per-block partials summed in a fixed order).  partial: scratch of
// grad_norm_partials() floats.
int grad_norm_clip(size_t n, const float* g, float max_norm, float* partial, float* norm_out, float* scale_out,
                   cudaStream_t s);
int grad_norm_partials();
int f32_to_bf16(size_t n, const float* src, void* dst, cudaStream_t s);
int act_to_f32(int act_bf16, size_t n, const void* src, float* dst, cudaStream_t s);
// copy [rows, cols] from a strided activation into dense fp32
int act_to_f32_2d(int act_bf16, int rows, int cols, long ld, const void* src, float* dst, cudaStream_t s);

int num_sms();

// 2-D TMA descriptor over a row-major matrix (inner = contiguous extent, outer =
// rows, ld in elements), bf16 or fp32, box box_inner x box_outer, 128-byte
// swizzle or none.  False (with a message) when the driver rejects it.
bool tma_map_2d(void* map128, const void* ptr, int f32, unsigned long long inner, unsigned long long outer,
                unsigned long long ld, unsigned box_inner, unsigned box_outer, int swizzle128, std::string* msg);

// tcgen05 flash-attention forward (bf16, head_dim 64 or 128); Hkv key/value
// heads, each serving H / Hkv query heads (grouped-query attention; Hkv = H:
// multi-head attention), qkv rows of (H + 2 Hkv) * hd.
int attn_fwd_tc(int B, int T, int H, int Hkv, int hd, const void* qkv, void* ctx, float* lse, int* dev_err,
                cudaStream_t s, std::string* msg);
// tcgen05 attention backward: one persistent launch over key-block items
// (dK, dV) and query-block items (dQ), each accumulated in TMEM (no atomics, no
// fp32 dQ accumulator).  dvec = rowsum(dO * O); counter: one int of device
// memory that the launch uses as its work counter (cleared on the stream first).
int attn_bwd_tc(int B, int T, int H, int Hkv, int hd, const void* qkv, const void* dctx, const float* lse,
                const float* dvec, int* counter, void* dqkv, int* dev_err, cudaStream_t s, std::string* msg);

// Process-wide count of kernel launches made by the library.
void count_launches(long long n);
long long launches_total();

}  // namespace fal
