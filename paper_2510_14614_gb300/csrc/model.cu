// Runtime behind the C ABI: workspace layout, the forward/backward schedule of
// GPT (Eq. 1), FAL (Eq. 2) and FAL+ (App. D.1) decoder stacks and of the
// paper's comparison blocks (Parallel, Sec. 5.1; Ablation1 / Ablation2 and FAL+
// reusing block k, App. D), AdamW with optional gradient clipping, taps.
//
// Data layout (all carved from the caller's workspace, 256-byte aligned):
//   flat fp32 parameters / gradients / AdamW m, v   [n_params]
//   bf16 copy of the parameters                      [n_params]   (bf16 path)
//   residual stream X_0..X_L fp32 [B*T, d]; per block u, m (MLP input),
//   qkv [B*T, 3d], ctx, h, g [B*T, d_ff] (activation type), LN statistics,
//   attention log-sum-exp; GPT/FAL+ also Y = X + a (fp32).
//   First attention a_1 (fp32) and its normalised form a1hat = (a_1 - mu)/sigma
//   (fp32): FAL's F = LN_F(a_1) = a1hat * gamma_F + beta_F and FAL+'s
//   LN_{F,i}(a_1) = a1hat * gamma_{F,i} + beta_{F,i}, so a_1 is normalised once
//   and every later block only applies its affine parameters (Sec. 4.1).
// Weight matrices are [out, in]; the fused FAL residual GEMM reads W_o and
// W_down in place as two K segments of one contraction.
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>
#include <initializer_list>
#include <climits>
#include <vector>

#include "../../include/fal.h"
#include "internal.h"

using namespace fal;

namespace {

constexpr size_t ALIGN = 256;
constexpr size_t NPOS = (size_t)-1;

struct LayerP {
  size_t ln1_g = NPOS, ln1_b = NPOS, w_qkv = NPOS, b_qkv = NPOS, w_o = NPOS, b_o = NPOS;
  size_t ln2_g = NPOS, ln2_b = NPOS, lnF_g = NPOS, lnF_b = NPOS, lnA_g = NPOS, lnA_b = NPOS;
  size_t w_up = NPOS, b_up = NPOS, w_down = NPOS, b_down = NPOS;
};

struct LayerA {
  float* X = nullptr;  // block input X_i
  float *ln1_mean = nullptr, *ln1_rstd = nullptr;
  void *u = nullptr, *m = nullptr, *qkv = nullptr, *ctx = nullptr, *h = nullptr, *g = nullptr;
  float* lse = nullptr;
  float *Y = nullptr, *ln2_mean = nullptr, *ln2_rstd = nullptr;
  // Ablation1: the block's own attention output a_i and its normalised form
  float *a = nullptr, *ahat = nullptr, *a_mean = nullptr, *a_rstd = nullptr;
};

// How block i computes its MLP input.
enum BlockKind {
  BK_SEQ = 0,     // m = LN2(X + a) (+ LN_{F,i}(a_k) for FAL+ after block k): GPT-style, sequential
  BK_PAR = 1,     // m = LN1(X) (+ LN_F(a_1) for FAL): the branches run side by side (Eq. 2)
  BK_FIRST = 2,   // FAL block 1: m = LN1(X) + LN_F(a_1) with a_1 computed here
  BK_OWN = 3      // Ablation1: m = LN1(X) + LN_{A,i}(a_i), the block's own attention
};

struct Bump {
  uint8_t* base;
  size_t off = 0;
  explicit Bump(uint8_t* b) : base(b) {}
  template <typename T>
  T* take(size_t count, size_t elem = sizeof(T)) {
    off = (off + ALIGN - 1) / ALIGN * ALIGN;
    T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
    off += count * elem;
    return p;
  }
};

}  // namespace

struct fal_handle {
  fal_config cfg{};
  int bf = 1;          // activations bf16 (else fp32 debug)
  size_t asz = 2;      // activation element size
  int B = 0, T = 0, d = 0, H = 0, hd = 0, F = 0, L = 0, V = 0, Vp = 0;
  int Hkv = 0, DQ = 0;  // key/value heads (GQA groups) and the fused QKV width d + 2 Hkv hd
  long BT = 0;
  cudaStream_t sm = nullptr, ss = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr, ev_mid = nullptr;
  std::string err;
  int state = 0;  // 0 fresh, 1 after forward, 2 after backward
  bool has_loss = false;
  long step_t = 0;
  // fal_train_step: the weight-gradient GEMMs of the block matrices also apply
  // AdamW (bias corrections of step step_t).
  bool fuse_opt = false;
  float opt_rbc1 = 1.f, opt_rbc2 = 1.f;

  std::vector<fal_tensor_info> tensors;
  size_t n_params = 0, n_decay = 0;
  size_t wte = NPOS, wpe = NPOS, lnF_g = NPOS, lnF_b = NPOS, lnf_g = NPOS, lnf_b = NPOS;
  std::vector<LayerP> lp;

  // workspace views
  float *P = nullptr, *G = nullptr, *Mo = nullptr, *Vo = nullptr;
  // bf16 copies of the parameters read by the GEMMs (bf16 path), two buffers:
  // the forward and backward read Shb[sh_cur]; AdamW writes the updated copy
  // into the other one, which becomes current after the step.  With the
  // optimizer fused into the weight-gradient GEMMs, a data-gradient GEMM that
  // runs in the same launch still reads this step's weights.
  void* Shb[2] = {nullptr, nullptr};
  int sh_cur = 0;
  int32_t *tok = nullptr, *tgt = nullptr;
  int* dev_err = nullptr;
  // per-tile flags of the ordered split-K residual GEMM; one new epoch per launch
  int* ord_flags = nullptr;
  int ord_cap = 0, ord_epoch = 0;
  float *loss = nullptr, *loss_rows = nullptr;
  std::vector<LayerA> la;
  float* Xout = nullptr;
  float *a1 = nullptr, *a1hat = nullptr, *a1_mean = nullptr, *a1_rstd = nullptr;
  void* xf = nullptr;
  float *lnf_mean = nullptr, *lnf_rstd = nullptr;
  void *logits = nullptr, *dlogits = nullptr;
  // chunked LM head (head_chunk > 0): two [BT, hc] chunk buffers, the
  // epilogue's per-slice statistics, the target logits and the log-sum-exp
  int hc = 0, ce_nsl = 0;
  void* hbuf[2] = {nullptr, nullptr};
  float2* ce_stats = nullptr;
  float *ce_tlogit = nullptr, *ce_lse = nullptr;
  float *dX = nullptr, *dY = nullptr, *dA = nullptr, *dU = nullptr, *dU2 = nullptr, *dA1hat = nullptr;
  void *dX_act = nullptr, *dY_act = nullptr, *dA_act = nullptr, *dctx = nullptr, *dh = nullptr, *dqkv = nullptr;
  float *dvec = nullptr, *part0 = nullptr, *part1 = nullptr;
  // gradient clipping: per-block partials, the norm and the scale factor
  float *gn_part = nullptr, *gn_norm = nullptr, *gn_scale = nullptr;
  bool has_norm = false;
  int reuse = 0;  // 0-based block whose attention output FAL+ adds to later MLP inputs
  float* stage = nullptr;
  size_t stage_floats = 0;
  size_t total_bytes = 0;

  // live kernel timing (fal_profile_enable)
  struct ProfRec { cudaEvent_t a, b; int kind; double flops; const char* label; int stream; };
  int prof = 0;  // 0 off, 1 GEMM and attention launches, 2 every launch
  std::vector<cudaEvent_t> ev_pool;
  size_t ev_next = 0;
  std::vector<ProfRec> recs;
};

namespace {

int fail(fal_handle* h, int code, const std::string& msg) {
  if (h) h->err = msg;
  return code;
}

void add_tensor(fal_handle* h, std::vector<fal_tensor_info>& dec, std::vector<fal_tensor_info>& nodec,
                const std::string& name, int r, int c, int decayed) {
  fal_tensor_info t;
  memset(&t, 0, sizeof(t));
  snprintf(t.name, sizeof(t.name), "%s", name.c_str());
  t.ndim = c > 0 ? 2 : 1;
  t.shape[0] = r;
  t.shape[1] = c > 0 ? c : 0;
  t.numel = (size_t)r * (c > 0 ? c : 1);
  t.decayed = decayed;
  (decayed ? dec : nodec).push_back(t);
  (void)h;
}

// Parameter table in the canonical order (matrices and embeddings first, so
// weight decay applies to one prefix of the flat buffer).
void build_table(fal_handle* h) {
  const int d = h->d, F = h->F, L = h->L, V = h->V, T = h->T, var = h->cfg.variant;
  std::vector<fal_tensor_info> dec, nodec;
  add_tensor(h, dec, nodec, "wte", V, d, 1);
  add_tensor(h, dec, nodec, "wpe", T, d, 1);
  for (int i = 0; i < L; ++i) {
    const std::string p = "h" + std::to_string(i) + ".";
    add_tensor(h, nodec, nodec, p + "ln1.g", d, 0, 0);
    add_tensor(h, nodec, nodec, p + "ln1.b", d, 0, 0);
    add_tensor(h, dec, nodec, p + "attn.w_qkv", h->DQ, d, 1);
    add_tensor(h, dec, nodec, p + "attn.b_qkv", h->DQ, 0, 0);
    add_tensor(h, dec, nodec, p + "attn.w_o", d, d, 1);
    add_tensor(h, dec, nodec, p + "attn.b_o", d, 0, 0);
    if (var == FAL_GPT || var == FAL_FALPLUS || (var == FAL_ABLATION2 && i == 0)) {
      add_tensor(h, dec, nodec, p + "ln2.g", d, 0, 0);
      add_tensor(h, dec, nodec, p + "ln2.b", d, 0, 0);
    }
    if (var == FAL_FALPLUS && i > h->reuse) {
      add_tensor(h, dec, nodec, p + "lnF.g", d, 0, 0);
      add_tensor(h, dec, nodec, p + "lnF.b", d, 0, 0);
    }
    if (var == FAL_ABLATION1) {
      add_tensor(h, dec, nodec, p + "lnA.g", d, 0, 0);
      add_tensor(h, dec, nodec, p + "lnA.b", d, 0, 0);
    }
    add_tensor(h, dec, nodec, p + "mlp.w_up", F, d, 1);
    add_tensor(h, dec, nodec, p + "mlp.b_up", F, 0, 0);
    add_tensor(h, dec, nodec, p + "mlp.w_down", d, F, 1);
    add_tensor(h, dec, nodec, p + "mlp.b_down", d, 0, 0);
  }
  if (var == FAL_FAL) {
    add_tensor(h, dec, nodec, "lnF.g", d, 0, 0);
    add_tensor(h, dec, nodec, "lnF.b", d, 0, 0);
  }
  add_tensor(h, dec, nodec, "lnf.g", d, 0, 0);
  add_tensor(h, dec, nodec, "lnf.b", d, 0, 0);
  h->tensors.clear();
  size_t off = 0;
  auto place = [&](std::vector<fal_tensor_info>& v) {
    for (auto& t : v) {
      off = (off + 63) / 64 * 64;  // 256-byte aligned fp32, 128-byte aligned bf16
      t.offset = off;
      off += t.numel;
      h->tensors.push_back(t);
    }
  };
  place(dec);
  off = (off + 63) / 64 * 64;
  h->n_decay = off;
  place(nodec);
  h->n_params = (off + 63) / 64 * 64;
  h->lp.assign(L, LayerP());
  for (auto& t : h->tensors) {
    const std::string n = t.name;
    if (n == "wte") h->wte = t.offset;
    else if (n == "wpe") h->wpe = t.offset;
    else if (n == "lnF.g") h->lnF_g = t.offset;
    else if (n == "lnF.b") h->lnF_b = t.offset;
    else if (n == "lnf.g") h->lnf_g = t.offset;
    else if (n == "lnf.b") h->lnf_b = t.offset;
    else {
      const int i = atoi(n.c_str() + 1);
      const std::string leaf = n.substr(n.find('.') + 1);
      LayerP& q = h->lp[i];
      if (leaf == "ln1.g") q.ln1_g = t.offset;
      else if (leaf == "ln1.b") q.ln1_b = t.offset;
      else if (leaf == "attn.w_qkv") q.w_qkv = t.offset;
      else if (leaf == "attn.b_qkv") q.b_qkv = t.offset;
      else if (leaf == "attn.w_o") q.w_o = t.offset;
      else if (leaf == "attn.b_o") q.b_o = t.offset;
      else if (leaf == "ln2.g") q.ln2_g = t.offset;
      else if (leaf == "ln2.b") q.ln2_b = t.offset;
      else if (leaf == "lnF.g") q.lnF_g = t.offset;
      else if (leaf == "lnF.b") q.lnF_b = t.offset;
      else if (leaf == "lnA.g") q.lnA_g = t.offset;
      else if (leaf == "lnA.b") q.lnA_b = t.offset;
      else if (leaf == "mlp.w_up") q.w_up = t.offset;
      else if (leaf == "mlp.b_up") q.b_up = t.offset;
      else if (leaf == "mlp.w_down") q.w_down = t.offset;
      else if (leaf == "mlp.b_down") q.b_down = t.offset;
    }
  }
}

int validate(const fal_config* c, std::string* msg) {
  if (!c) { *msg = "null config"; return FAL_ERR_ARG; }
  if (c->variant < FAL_GPT || c->variant > FAL_ABLATION2) {
    *msg = "variant must be GPT, FAL, FAL+, Parallel, Ablation1 or Ablation2";
    return FAL_ERR_ARG;
  }
  if (c->layers < 1 || c->d_model < 1 || c->heads < 1 || c->d_ff < 1 || c->seq < 1 || c->batch < 1 || c->vocab < 2) {
    *msg = "layers, d_model, heads, d_ff, seq, batch must be >= 1 and vocab >= 2";
    return FAL_ERR_ARG;
  }
  if (c->d_model % c->heads) { *msg = "d_model must be a multiple of heads"; return FAL_ERR_ARG; }
  if (c->reuse_layer < 0 || c->reuse_layer > c->layers || (c->reuse_layer > 1 && c->variant != FAL_FALPLUS)) {
    *msg = "reuse_layer must be in [0, layers] and above 1 only for FAL+";
    return FAL_ERR_ARG;
  }
  if (!(c->clip_norm >= 0.f)) { *msg = "clip_norm must be >= 0"; return FAL_ERR_ARG; }
  if (c->kv_heads < 0 || (c->kv_heads > 0 && c->heads % c->kv_heads)) {
    *msg = "kv_heads must be 0 (one per head) or divide heads";
    return FAL_ERR_ARG;
  }
  if (c->head_chunk < 0 || c->head_chunk % 64) {
    *msg = "head_chunk must be 0 (stored logits) or a positive multiple of 64";
    return FAL_ERR_ARG;
  }
  if (c->precision != FAL_BF16 && c->precision != FAL_FP32_DEBUG) { *msg = "bad precision"; return FAL_ERR_ARG; }
  if (c->schedule != FAL_SCHED_SERIAL && c->schedule != FAL_SCHED_TWO_STREAM) { *msg = "bad schedule"; return FAL_ERR_ARG; }
  const int hd = c->d_model / c->heads;
  if (c->precision == FAL_BF16) {
    if (hd != 64 && hd != 128) { *msg = "bf16 path needs head_dim 64 or 128"; return FAL_ERR_ARG; }
    if (c->d_model % 8 || c->d_ff % 8) { *msg = "bf16 path needs d_model and d_ff multiples of 8"; return FAL_ERR_ARG; }
  } else {
    if (hd > 128) { *msg = "fp32 debug path needs head_dim <= 128"; return FAL_ERR_ARG; }
    if (c->d_model % 4 || c->d_ff % 4) { *msg = "d_model and d_ff must be multiples of 4"; return FAL_ERR_ARG; }
  }
  if (c->d_model > 4096) { *msg = "d_model above 4096 is not supported by the LayerNorm kernels"; return FAL_ERR_ARG; }
  if ((long)c->batch * c->seq > 65535) { *msg = "batch*seq above 65535 is not supported"; return FAL_ERR_ARG; }
  return FAL_OK;
}

void init_dims(fal_handle* h, const fal_config* c) {
  h->cfg = *c;
  h->bf = c->precision == FAL_BF16;
  h->asz = h->bf ? 2 : 4;
  h->B = c->batch; h->T = c->seq; h->d = c->d_model; h->H = c->heads; h->hd = c->d_model / c->heads;
  h->F = c->d_ff; h->L = c->layers; h->V = c->vocab;
  h->Vp = (c->vocab + 63) / 64 * 64;
  h->BT = (long)h->B * h->T;
  h->reuse = c->reuse_layer > 1 ? c->reuse_layer - 1 : 0;
  h->Hkv = c->kv_heads > 0 ? c->kv_heads : h->H;
  h->DQ = h->d + 2 * h->Hkv * h->hd;
  h->hc = c->head_chunk > 0 ? (c->head_chunk < h->Vp ? c->head_chunk : (int)h->Vp) : 0;
  h->ce_nsl = (c->vocab + (h->bf ? kCeSliceTc : kCeSliceSimt) - 1) / (h->bf ? kCeSliceTc : kCeSliceSimt);
}

// MLP-input rule of block i (the block equations of each variant).
int block_kind(const fal_handle* h, int i) {
  switch (h->cfg.variant) {
    case FAL_FAL: return i == 0 ? BK_FIRST : BK_PAR;
    case FAL_PARALLEL: return BK_PAR;
    case FAL_ABLATION1: return BK_OWN;
    case FAL_ABLATION2: return i == 0 ? BK_SEQ : BK_PAR;
    default: return BK_SEQ;  // GPT, FAL+
  }
}
// The tensor the MLP reads: m, or u itself where the MLP input is LN1(X) alone.
const void* mlp_in(const fal_handle* h, int i) {
  const int v = h->cfg.variant;
  return (block_kind(h, i) == BK_PAR && v != FAL_FAL) ? h->la[i].u : h->la[i].m;
}

// Carves every buffer; with base == nullptr it only measures.
void carve(fal_handle* h, uint8_t* base) {
  Bump b(base);
  const long BT = h->BT;
  const size_t d = h->d, F = h->F, a = h->asz;
  const int var = h->cfg.variant;
  h->P = b.take<float>(h->n_params);
  h->G = b.take<float>(h->n_params);
  h->Mo = b.take<float>(h->n_params);
  h->Vo = b.take<float>(h->n_params);
  h->Shb[0] = h->bf ? b.take<uint8_t>(h->n_params * 2) : nullptr;
  h->Shb[1] = h->bf ? b.take<uint8_t>(h->n_params * 2) : nullptr;
  h->tok = b.take<int32_t>(BT);
  h->tgt = b.take<int32_t>(BT);
  h->dev_err = b.take<int>(4);
  h->ord_cap = (int)(((BT + 127) / 128) * (((long)d + 255) / 256) * 16);
  h->ord_flags = b.take<int>(h->ord_cap);
  h->loss = b.take<float>(4);
  h->loss_rows = b.take<float>(BT);
  h->la.assign(h->L, LayerA());
  for (int i = 0; i < h->L; ++i) {
    LayerA& A = h->la[i];
    A.X = b.take<float>(BT * d);
    A.ln1_mean = b.take<float>(BT);
    A.ln1_rstd = b.take<float>(BT);
    A.u = b.take<uint8_t>(BT * d * a);
    A.m = b.take<uint8_t>(BT * d * a);
    A.qkv = b.take<uint8_t>(BT * h->DQ * a);
    A.ctx = b.take<uint8_t>(BT * d * a);
    A.lse = b.take<float>((size_t)h->B * h->H * h->T);
    A.h = b.take<uint8_t>(BT * F * a);
    A.g = b.take<uint8_t>(BT * F * a);
    if (var == FAL_GPT || var == FAL_FALPLUS || (var == FAL_ABLATION2 && i == 0)) {
      A.Y = b.take<float>(BT * d);
      A.ln2_mean = b.take<float>(BT);
      A.ln2_rstd = b.take<float>(BT);
    }
    if (var == FAL_ABLATION1) {
      A.a = b.take<float>(BT * d);
      A.ahat = b.take<float>(BT * d);
      A.a_mean = b.take<float>(BT);
      A.a_rstd = b.take<float>(BT);
    }
  }
  h->Xout = b.take<float>(BT * d);
  h->a1 = b.take<float>(BT * d);
  h->a1hat = b.take<float>(BT * d);
  h->a1_mean = b.take<float>(BT);
  h->a1_rstd = b.take<float>(BT);
  h->xf = b.take<uint8_t>(BT * d * a);
  h->lnf_mean = b.take<float>(BT);
  h->lnf_rstd = b.take<float>(BT);
  if (h->hc) {
    h->hbuf[0] = b.take<uint8_t>((size_t)BT * h->hc * a);
    h->hbuf[1] = b.take<uint8_t>((size_t)BT * h->hc * a);
    h->ce_stats = b.take<float2>((size_t)h->ce_nsl * BT);
    h->ce_tlogit = b.take<float>(BT);
    h->ce_lse = b.take<float>(BT);
  } else {
    h->logits = b.take<uint8_t>((size_t)BT * h->Vp * a);
    h->dlogits = b.take<uint8_t>((size_t)BT * h->Vp * a);
  }
  h->dX = b.take<float>(BT * d);
  h->dY = b.take<float>(BT * d);
  h->dA = b.take<float>(BT * d);
  h->dU = b.take<float>(BT * d);
  h->dU2 = b.take<float>(BT * d);
  h->dA1hat = b.take<float>(BT * d);
  h->dX_act = b.take<uint8_t>(BT * d * a);
  h->dY_act = b.take<uint8_t>(BT * d * a);
  h->dA_act = b.take<uint8_t>(BT * d * a);
  h->dctx = b.take<uint8_t>(BT * d * a);
  h->dh = b.take<uint8_t>(BT * F * a);
  h->dqkv = b.take<uint8_t>(BT * h->DQ * a);
  h->dvec = b.take<float>(attn_bwd_scratch_floats(h->B, h->T, h->H));
  const int cs_cols = h->DQ > h->F ? h->DQ : h->F;  // widest column reduction: b_qkv or b_up
  h->part0 = b.take<float>(colsum_partial_floats(cs_cols));
  h->part1 = b.take<float>(colsum_partial_floats(cs_cols));
  h->gn_part = b.take<float>(grad_norm_partials());
  h->gn_norm = b.take<float>(4);
  h->gn_scale = b.take<float>(4);
  h->stage_floats = (size_t)4 << 20;
  h->stage = b.take<float>(h->stage_floats);
  h->total_bytes = b.off + ALIGN;
}

// ------------------------------------------------------------ launch helpers
struct Ctx {
  fal_handle* h;
  int rc = FAL_OK;
  bool ok() const { return rc == FAL_OK; }
  void check(int r, const char* what) {
    if (rc != FAL_OK || r == 0) return;
    rc = (r == 1) ? FAL_ERR_ARG : (r == 6) ? FAL_ERR_UNSUPPORTED : FAL_ERR_CUDA;
    if (h->err.empty() || h->err.find(what) == std::string::npos) h->err = std::string(what) + ": " + h->err;
  }
};

GemmSeg seg(const void* A, long lda, int amn, const void* B, long ldb, int bmn, int K) {
  GemmSeg s;
  s.A = {A, lda, amn};
  s.B = {B, ldb, bmn};
  s.K = K;
  return s;
}
EpiParams epi_out(void* out, long ldo, int mode) {
  EpiParams e;
  memset(&e, 0, sizeof(e));
  e.out = out; e.ldo = ldo; e.out_mode = mode;
  return e;
}
GemmCall call1(int M, int N, GemmSeg s0, const EpiParams& e) {
  GemmCall c;
  memset(&c, 0, sizeof(c));
  c.ngroups = 1;
  c.g[0].M = M; c.g[0].N = N; c.g[0].nseg = 1; c.g[0].seg[0] = s0; c.g[0].epi = e;
  return c;
}

// One launch running the groups of several calls (independent contractions),
// tiles in argument order.  Weight-gradient groups go first: their epilogues
// (fp32 stores, fused AdamW) then overlap the data-gradient main loops, and
// the wave tails of the separate launches disappear.
GemmCall group_calls(std::initializer_list<GemmCall> calls) {
  GemmCall out;
  memset(&out, 0, sizeof(out));
  for (const GemmCall& c : calls)
    for (int g = 0; g < c.ngroups && out.ngroups < kMaxGemmGroups; ++g) out.g[out.ngroups++] = c.g[g];
  return out;
}

float* Pp(fal_handle* h, size_t off) { return off == NPOS ? nullptr : h->P + off; }
float* Gp(fal_handle* h, size_t off) { return off == NPOS ? nullptr : h->G + off; }
// GEMM weight operand: bf16 copy on the bf16 path, fp32 master on the debug path.
const void* Wp(fal_handle* h, size_t off) {
  return h->bf ? (const void*)((const uint8_t*)h->Shb[h->sh_cur] + off * 2) : (const void*)(h->P + off);
}

// Epilogue of the weight-gradient GEMM of the matrix at offset w ([rows, ld]):
// the fp32 gradient, and under fal_train_step the AdamW update of the matrix.
EpiParams wgrad_out(fal_handle* h, size_t w, long ld) {
  EpiParams e = epi_out(Gp(h, w), ld, OUT_F32);
  if (h->fuse_opt) {
    const fal_config& c = h->cfg;
    e.op = EPI_ADAMW;
    e.opt_p = h->P + w; e.opt_m = h->Mo + w; e.opt_v = h->Vo + w;
    e.opt_sh = h->bf ? (void*)((uint8_t*)h->Shb[h->sh_cur ^ 1] + w * 2) : nullptr;
    e.opt_lr = c.lr; e.opt_b1 = c.beta1; e.opt_b2 = c.beta2; e.opt_eps = c.eps; e.opt_wd = c.weight_decay;
    e.opt_rbc1 = h->opt_rbc1; e.opt_rbc2 = h->opt_rbc2;
  }
  return e;
}

cudaEvent_t pool_event(fal_handle* h) {
  if (h->ev_next == h->ev_pool.size()) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    h->ev_pool.push_back(e);
  }
  return h->ev_pool[h->ev_next++];
}

// Brackets one launch with timing events when profiling is on.
struct ProfScope {
  fal_handle* h;
  cudaStream_t s;
  cudaEvent_t a = nullptr;
  int kind;
  double flops;
  const char* label;
  ProfScope(fal_handle* h_, cudaStream_t s_, int kind_, double flops_, const char* label_ = "")
      : h(h_), s(s_), kind(kind_), flops(flops_), label(label_) {
    if (h->prof > (kind == 3 ? 1 : 0) && (a = pool_event(h)) != nullptr) cudaEventRecord(a, s);
  }
  ~ProfScope() {
    if (!a) return;
    cudaEvent_t b = pool_event(h);
    if (!b) return;
    cudaEventRecord(b, s);
    h->recs.push_back({a, b, kind, flops, label, s == h->sm ? 0 : 1});
  }
};

double gemm_flops(const GemmCall& call) {
  double f = 0;
  for (int g = 0; g < call.ngroups; ++g)
    for (int k = 0; k < call.g[g].nseg; ++k) f += 2.0 * call.g[g].M * call.g[g].N * call.g[g].seg[k].K;
  return f;
}

void gemm(Ctx& c, const GemmCall& call, cudaStream_t s, const char* what) {
  if (!c.ok()) return;
  fal_handle* h = c.h;
  h->err.clear();
  ProfScope ps(h, s, 0, gemm_flops(call), what);
  int r = h->bf ? gemm_tc(call, h->dev_err, s, &h->err) : gemm_simt(call, 0, 0, s, &h->err);
  c.check(r, what);
}

double attn_fwd_flops(fal_handle* h) { return 2.0 * h->B * h->H * (double)h->T * h->T * h->hd; }

void colsum_(Ctx& c, cudaStream_t s, float* part, const void* src, int src_act, long ld, int d, const float* src2,
             int bmode, const float* x, const float* mean, const float* rstd, const float* bsrc, float* out1,
             float* out0, float* out0b, int accumulate) {
  if (!c.ok()) return;
  fal_handle* h = c.h;
  ColsumArgs a;
  memset(&a, 0, sizeof(a));
  a.rows = (int)h->BT; a.d = d; a.src = src; a.src_act = src_act; a.ld = ld; a.src2 = src2;
  a.bmode = bmode; a.x = x; a.mean = mean; a.rstd = rstd; a.bsrc = bsrc;
  a.partial = part; a.out1 = out1; a.out0 = out0; a.out0b = out0b; a.accumulate = accumulate;
  ProfScope ps(h, s, 3, 0.0, "column reduction");
  c.check(colsum(h->bf, a, s), "column reduction");
}

void ln_fwd_(Ctx& c, cudaStream_t s, const float* x, const float* gm, const float* bt, void* out, float* out_f32,
             float* mean, float* rstd, void* out2, const float* add_src, const float* add_g, const float* add_b) {
  if (!c.ok()) return;
  LnFwdArgs a;
  memset(&a, 0, sizeof(a));
  a.rows = (int)c.h->BT; a.d = c.h->d; a.x = x; a.gamma = gm; a.beta = bt; a.out = out; a.out_f32 = out_f32;
  a.mean = mean; a.rstd = rstd; a.out2 = out2; a.add_src = add_src; a.add_g = add_g; a.add_b = add_b;
  a.err = c.h->dev_err;
  ProfScope ps(c.h, s, 3, 0.0, "layernorm forward");
  c.check(ln_fwd(c.h->bf, a, s), "layernorm forward");
}

// Bias gradients that are column sums of a LayerNorm backward's output dx:
// the linear maps whose outputs add into the residual that the LN normalised.
struct BiasSum { float* b1 = nullptr; float* b2 = nullptr; };

// LayerNorm backward; with dgamma/dbeta also the affine parameters' gradients
// (column sums over the rows, computed in the same pass; part: scratch), and
// with bias targets the column sums of dx itself, stored there.
void ln_bwd_(Ctx& c, cudaStream_t s, const float* dy, const float* dy2, const float* x, const float* mean,
             const float* rstd, const float* gm, const float* dres, float* dx, void* dx_act, float* part = nullptr,
             float* dgamma = nullptr, float* dbeta = nullptr, BiasSum bias = BiasSum()) {
  if (!c.ok()) return;
  LnBwdArgs a;
  memset(&a, 0, sizeof(a));
  a.rows = (int)c.h->BT; a.d = c.h->d; a.dy = dy; a.dy2 = dy2; a.x = x; a.mean = mean; a.rstd = rstd; a.gamma = gm;
  a.dres = dres; a.dx = dx; a.dx_act = dx_act;
  a.err = c.h->dev_err;
  if (dgamma || dbeta || bias.b1 || bias.b2) { a.cs_part = part; a.cs_out1 = dgamma; a.cs_out0 = dbeta; }
  a.dxs_out = bias.b1; a.dxs_out2 = bias.b2;
  ProfScope ps(c.h, s, 3, 0.0, "layernorm backward");
  c.check(ln_bwd(c.h->bf, a, s), "layernorm backward");
}

void fork(fal_handle* h) {
  cudaEventRecord(h->ev_fork, h->sm);
  cudaStreamWaitEvent(h->ss, h->ev_fork, 0);
}
void join(fal_handle* h) {
  cudaEventRecord(h->ev_join, h->ss);
  cudaStreamWaitEvent(h->sm, h->ev_join, 0);
}

// ------------------------------------------------------------ forward
void qkv_and_attention(Ctx& c, int i, cudaStream_t s, cudaStream_t after_qkv = nullptr) {
  fal_handle* h = c.h;
  LayerA& A = h->la[i];
  const LayerP& p = h->lp[i];
  const int BT = (int)h->BT, d = h->d;
  EpiParams e = epi_out(A.qkv, h->DQ, OUT_ACT);
  e.bias = Pp(h, p.b_qkv);
  gemm(c, call1(BT, h->DQ, seg(A.u, d, 0, Wp(h, p.w_qkv), d, 0, d), e), s, "QKV projection");
  if (after_qkv) {
    // the other stream's work starts behind the projection, beside the attention
    cudaEventRecord(h->ev_mid, s);
    cudaStreamWaitEvent(after_qkv, h->ev_mid, 0);
  }
  if (!c.ok()) return;
  h->err.clear();
  ProfScope ps(h, s, 1, attn_fwd_flops(h), "attention forward");
  c.check(attn_fwd(h->bf, h->B, h->T, h->H, h->hd, A.qkv, A.ctx, A.lse, h->dev_err, s, &h->err, h->Hkv),
          "attention forward");
}

void up_gemm(Ctx& c, int i, cudaStream_t s) {
  fal_handle* h = c.h;
  LayerA& A = h->la[i];
  const LayerP& p = h->lp[i];
  EpiParams e = epi_out(A.h, h->F, OUT_ACT);
  e.op = EPI_GELU; e.out2 = A.g; e.ldo2 = h->F; e.bias = Pp(h, p.b_up);
  gemm(c, call1((int)h->BT, h->F, seg(mlp_in(h, i), h->d, 0, Wp(h, p.w_up), h->d, 0, h->d), e), s,
       "MLP up-projection");
}

// Whether splitting an M x N output of 256 x 256 tiles (one per pair of SMs)
// in two halves of K fills the last wave of the persistent grid clearly better.
bool split_k_pays(long M, long N) {
  const long units = num_sms() / 2, tiles = ((M + 255) / 256) * ((N + 255) / 256);
  auto fill = [&](long t) { return (double)t / (double)(((t + units - 1) / units) * units); };
  return fill(2 * tiles) > fill(tiles) + 0.05;
}

void layer_forward(Ctx& c, int i) {
  fal_handle* h = c.h;
  LayerA& A = h->la[i];
  const LayerP& p = h->lp[i];
  const int BT = (int)h->BT, d = h->d, F = h->F, var = h->cfg.variant;
  float* Xn = (i + 1 < h->L) ? h->la[i + 1].X : h->Xout;
  cudaStream_t s = h->sm;
  const int kind = block_kind(h, i);
  if (kind == BK_PAR) {
    if (var == FAL_FAL)  // m_i = LN1_i(X_i) + a1hat * gamma_F + beta_F  (Eq. 2), u_i = LN1_i(X_i)
      ln_fwd_(c, s, A.X, Pp(h, p.ln1_g), Pp(h, p.ln1_b), A.u, nullptr, A.ln1_mean, A.ln1_rstd, A.m, h->a1hat,
              Pp(h, h->lnF_g), Pp(h, h->lnF_b));
    else  // Parallel block: the MLP reads u_i = LN1_i(X_i) itself
      ln_fwd_(c, s, A.X, Pp(h, p.ln1_g), Pp(h, p.ln1_b), A.u, nullptr, A.ln1_mean, A.ln1_rstd, nullptr, nullptr,
              nullptr, nullptr);
    // The MHA branch and the MLP branch only share u/m: run them side by side.
    const bool two = h->cfg.schedule == FAL_SCHED_TWO_STREAM && h->ss != h->sm;
    if (two) {
      fork(h);
      qkv_and_attention(c, i, h->ss, s);
      up_gemm(c, i, s);
      join(h);
    } else {
      qkv_and_attention(c, i, s);
      up_gemm(c, i, s);
    }
    // X_{i+1} = X_i + [ctx | g] [W_o ; W_down]^T + b_o + b_down: one contraction over K = d + d_ff.
    GemmCall call;
    memset(&call, 0, sizeof(call));
    call.ngroups = 1;
    GemmGroupDesc& G = call.g[0];
    G.M = BT; G.N = d; G.nseg = 2;
    G.seg[0] = seg(A.ctx, d, 0, Wp(h, p.w_o), d, 0, d);
    G.seg[1] = seg(A.g, F, 0, Wp(h, p.w_down), F, 0, F);
    G.epi = epi_out(Xn, d, OUT_F32);
    G.epi.bias = Pp(h, p.b_o); G.epi.bias2 = Pp(h, p.b_down);
    G.epi.resid = A.X; G.epi.ldr = d;
    if (h->bf && d % 64 == 0 && F > d && split_k_pays(BT, d)) {
      // Two halves of K as two groups: twice the tiles of one N = d output, so
      // the last wave of the persistent grid is nearly full.  The first half
      // stores X_i + biases + its partial; the second adds its partial with TMA
      // reduce-adds only after the same tile of the first half has landed, so
      // the sum is formed in a fixed order (bitwise reproducible).
      const int k1 = ((d + F) / 2 + 63) / 64 * 64 - d;
      call.ngroups = 2;
      G.seg[1].K = k1;
      G.epi.ord_role = ORD_SIGNAL; G.epi.ord_flags = h->ord_flags; G.epi.ord_cap = h->ord_cap;
      h->ord_epoch = h->ord_epoch == INT_MAX ? 1 : h->ord_epoch + 1;
      G.epi.ord_epoch = h->ord_epoch;
      GemmGroupDesc& G1 = call.g[1];
      G1.M = BT; G1.N = d; G1.nseg = 1;
      G1.seg[0] = seg((const uint8_t*)A.g + (size_t)k1 * h->asz, F, 0, (const uint8_t*)Wp(h, p.w_down) + (size_t)k1 * 2,
                      F, 0, F - k1);
      G1.epi = epi_out(Xn, d, OUT_F32_ACCUM);
      G1.epi.ord_role = ORD_WAIT; G1.epi.ord_flags = h->ord_flags; G1.epi.ord_cap = h->ord_cap;
      G1.epi.ord_epoch = G.epi.ord_epoch;
    }
    gemm(c, call, s, "fused residual GEMM");
    return;
  }
  ln_fwd_(c, s, A.X, Pp(h, p.ln1_g), Pp(h, p.ln1_b), A.u, nullptr, A.ln1_mean, A.ln1_rstd, nullptr, nullptr, nullptr,
          nullptr);
  qkv_and_attention(c, i, s);
  if (kind == BK_FIRST || kind == BK_OWN) {
    // FAL block 1: a_1 = ctx W_o^T + b_o, a1hat = LN(a_1) without affine,
    // m_1 = LN1_1(X_1) + a1hat * gamma_F + beta_F, X_2 = X_1 + a_1 + MLP_1(m_1).
    // Ablation1 block i: the same with the block's own a_i and LN_{A,i}.
    const bool first = kind == BK_FIRST;
    float* a = first ? h->a1 : A.a;
    float* ahat = first ? h->a1hat : A.ahat;
    EpiParams e = epi_out(a, d, OUT_F32);
    e.bias = Pp(h, p.b_o);
    gemm(c, call1(BT, d, seg(A.ctx, d, 0, Wp(h, p.w_o), d, 0, d), e), s, "attention output projection");
    ln_fwd_(c, s, a, nullptr, nullptr, nullptr, ahat, first ? h->a1_mean : A.a_mean, first ? h->a1_rstd : A.a_rstd,
            nullptr, nullptr, nullptr, nullptr);
    ln_fwd_(c, s, A.X, Pp(h, p.ln1_g), Pp(h, p.ln1_b), nullptr, nullptr, nullptr, nullptr, A.m, ahat,
            Pp(h, first ? h->lnF_g : p.lnA_g), Pp(h, first ? h->lnF_b : p.lnA_b));
    up_gemm(c, i, s);
    EpiParams e2 = epi_out(Xn, d, OUT_F32);
    e2.bias = Pp(h, p.b_down); e2.resid = A.X; e2.ldr = d; e2.resid2 = a; e2.ldr2 = d;
    gemm(c, call1(BT, d, seg(A.g, F, 0, Wp(h, p.w_down), F, 0, F), e2), s, "MLP down-projection");
    return;
  }
  // GPT, FAL+ and Ablation2's block 1: Y = X + a; m = LN2(Y) (+ LN_{F,i}(a_k)
  // for FAL+ blocks after the reused block k)
  const bool keep_a = var == FAL_FALPLUS && i == h->reuse;
  EpiParams e = epi_out(A.Y, d, OUT_F32);
  e.bias = Pp(h, p.b_o); e.resid = A.X; e.ldr = d;
  if (keep_a) { e.pre_f32 = 1; e.out2 = h->a1; e.ldo2 = d; }
  gemm(c, call1(BT, d, seg(A.ctx, d, 0, Wp(h, p.w_o), d, 0, d), e), s, "attention output projection");
  if (keep_a)
    ln_fwd_(c, s, h->a1, nullptr, nullptr, nullptr, h->a1hat, h->a1_mean, h->a1_rstd, nullptr, nullptr, nullptr,
            nullptr);
  if (var == FAL_FALPLUS && i > h->reuse)
    ln_fwd_(c, s, A.Y, Pp(h, p.ln2_g), Pp(h, p.ln2_b), nullptr, nullptr, A.ln2_mean, A.ln2_rstd, A.m, h->a1hat,
            Pp(h, p.lnF_g), Pp(h, p.lnF_b));
  else
    ln_fwd_(c, s, A.Y, Pp(h, p.ln2_g), Pp(h, p.ln2_b), A.m, nullptr, A.ln2_mean, A.ln2_rstd, nullptr, nullptr,
            nullptr, nullptr);
  up_gemm(c, i, s);
  EpiParams e2 = epi_out(Xn, d, OUT_F32);
  e2.bias = Pp(h, p.b_down); e2.resid = A.Y; e2.ldr = d;
  gemm(c, call1(BT, d, seg(A.g, F, 0, Wp(h, p.w_down), F, 0, F), e2), s, "MLP down-projection");
}

int forward_impl(fal_handle* h, const int32_t* tokens, const int32_t* targets) {
  Ctx c{h};
  cudaStream_t s = h->sm;
  const size_t nb = (size_t)h->BT * sizeof(int32_t);
  if (cudaMemcpyAsync(h->tok, tokens, nb, cudaMemcpyDefault, s) != cudaSuccess ||
      cudaMemcpyAsync(h->tgt, targets, nb, cudaMemcpyDefault, s) != cudaSuccess)
    return fail(h, FAL_ERR_CUDA, "token copy failed");
  c.check(embed_fwd((int)h->BT, h->T, h->d, h->V, h->tok, Pp(h, h->wte), Pp(h, h->wpe), h->la[0].X, h->dev_err, s),
          "embedding");
  for (int i = 0; i < h->L && c.ok(); ++i) layer_forward(c, i);
  ln_fwd_(c, s, h->Xout, Pp(h, h->lnf_g), Pp(h, h->lnf_b), h->xf, nullptr, h->lnf_mean, h->lnf_rstd, nullptr, nullptr,
          nullptr, nullptr);
  if (h->hc) {
    // logits = xf wte^T reduced in the GEMM epilogue to per-slice (max, sum
    // exp) and the target logit; the loss and lse follow from those
    EpiParams e = epi_out(nullptr, 0, OUT_ACT);
    e.op = EPI_CE_STATS;
    e.ce_tgt = h->tgt; e.ce_stats = h->ce_stats; e.ce_tlogit = h->ce_tlogit; e.ce_ld = h->BT; e.ce_v0 = 0;
    gemm(c, call1((int)h->BT, h->V, seg(h->xf, h->d, 0, Wp(h, h->wte), h->d, 0, h->d), e), s,
         "LM head (loss statistics)");
    ProfScope ps_ce(h, s, 3, 0.0, "cross-entropy");
    if (c.ok())
      c.check(ce_combine((int)h->BT, h->ce_nsl, h->ce_stats, h->BT, h->ce_tlogit, h->tgt, h->V, h->ce_lse,
                         h->loss_rows, h->loss, h->dev_err, s),
              "cross-entropy");
    return c.rc;
  }
  // logits = xf wte^T (tied LM head), padded row pitch Vp
  gemm(c, call1((int)h->BT, h->V, seg(h->xf, h->d, 0, Wp(h, h->wte), h->d, 0, h->d), epi_out(h->logits, h->Vp, OUT_ACT)),
       s, "LM head");
  ProfScope ps_ce(h, s, 3, 0.0, "cross-entropy");
  if (c.ok())
    c.check(cross_entropy(h->bf, (int)h->BT, h->V, h->Vp, h->logits, h->tgt, h->dlogits, h->loss_rows, h->loss,
                          h->dev_err, s),
            "cross-entropy");
  return c.rc;
}

// ------------------------------------------------------------ backward
// Gradient GEMM helpers.  dgrad: dIn[BT, in] = dOut[BT, out] W[out, in]
// (B operand MN-major); wgrad: dW[out, in] = dOut^T In (both MN-major).
GemmSeg dgrad_seg(fal_handle* h, const void* dout, int out_dim, size_t w, int in_dim) {
  return seg(dout, out_dim, 0, Wp(h, w), in_dim, 1, out_dim);
}
GemmSeg wgrad_seg(fal_handle* h, const void* dout, int out_dim, const void* in, int in_dim) {
  return seg(dout, out_dim, 1, in, in_dim, 1, (int)h->BT);
}

void mlp_backward(Ctx& c, int i, const float* dXn, const void* dXn_act, cudaStream_t s, float* part) {
  // dh = (dXn W_down) * gelu'(h); dW_down; db_down; dm = dh W_up -> dU2; dW_up; db_up
  fal_handle* h = c.h;
  LayerA& A = h->la[i];
  const LayerP& p = h->lp[i];
  const int BT = (int)h->BT, d = h->d, F = h->F;
  EpiParams e = epi_out(h->dh, F, OUT_ACT);
  e.op = EPI_DGELU; e.aux = A.h; e.ldx = F;
  gemm(c, group_calls({call1(d, F, wgrad_seg(h, dXn_act, d, A.g, F), wgrad_out(h, p.w_down, F)),
                       call1(BT, F, dgrad_seg(h, dXn_act, d, p.w_down, F), e)}),
       s, "MLP down wgrad + dgrad");
  (void)dXn;  // db_down = column sums of dXn, summed by the LayerNorm backward that produced it
  gemm(c, group_calls({call1(F, d, wgrad_seg(h, h->dh, F, mlp_in(h, i), d), wgrad_out(h, p.w_up, d)),
                       call1(BT, d, dgrad_seg(h, h->dh, F, p.w_up, d), epi_out(h->dU2, d, OUT_F32))}),
       s, "MLP up wgrad + dgrad");
  colsum_(c, s, part, h->dh, 1, F, F, nullptr, 0, nullptr, nullptr, nullptr, nullptr, nullptr, Gp(h, p.b_up), nullptr, 0);
}

void attn_backward(Ctx& c, int i, const float* da, const void* da_act, cudaStream_t s, float* part, bool skip_wo,
                   bool d_ready = false) {
  // dctx = da W_o; dW_o; db_o; attention backward; du = dqkv W_qkv -> dU; dW_qkv; db_qkv
  fal_handle* h = c.h;
  LayerA& A = h->la[i];
  const LayerP& p = h->lp[i];
  const int BT = (int)h->BT, d = h->d;
  if (!skip_wo) {
    // dctx also yields the attention backward's D = rowsum(dctx * ctx) per head
    EpiParams edc = epi_out(h->dctx, d, OUT_ACT);
    if (h->bf) {
      edc.rd_src = A.ctx; edc.rd_ld = d; edc.rd_out = h->dvec; edc.rd_hd = h->hd; edc.rd_T = h->T; edc.rd_H = h->H;
      d_ready = true;
    }
    gemm(c, group_calls({call1(d, d, wgrad_seg(h, da_act, d, A.ctx, d), wgrad_out(h, p.w_o, d)),
                         call1(BT, d, dgrad_seg(h, da_act, d, p.w_o, d), edc)}),
         s, "attention out wgrad + dgrad");
    (void)da;  // db_o = column sums of da, summed by the LayerNorm backward that produced it
  }
  if (!c.ok()) return;
  h->err.clear();
  {
    ProfScope ps(h, s, 2, 2.0 * attn_fwd_flops(h), "attention backward");
    c.check(attn_bwd(h->bf, h->B, h->T, h->H, h->hd, A.qkv, A.ctx, A.lse, h->dctx, h->dqkv, h->dvec,
                     h->dev_err, s, &h->err, d_ready ? 1 : 0, h->Hkv),
            "attention backward");
  }
  gemm(c, group_calls({call1(h->DQ, d, wgrad_seg(h, h->dqkv, h->DQ, A.u, d), wgrad_out(h, p.w_qkv, d)),
                       call1(BT, d, dgrad_seg(h, h->dqkv, h->DQ, p.w_qkv, d), epi_out(h->dU, d, OUT_F32))}),
       s, "QKV wgrad + dgrad");
  colsum_(c, s, part, h->dqkv, 1, h->DQ, h->DQ, nullptr, 0, nullptr, nullptr, nullptr, nullptr, nullptr, Gp(h, p.b_qkv),
          nullptr, 0);
}

// attention term of MLP_i's input (first attention, or Ablation1's own):
// dA1hat += dU2 * gamma(i); dgamma(i), dbeta(i) from the normalised ahat
void first_attention_grad(Ctx& c, size_t g_off, size_t b_off, cudaStream_t s, float* part, int accumulate,
                          const float* ahat = nullptr) {
  fal_handle* h = c.h;
  if (!c.ok()) return;
  {
    ProfScope ps(h, s, 3, 0.0, "first-attention gradient");
    c.check(add_scaled_cols((int)h->BT, h->d, h->dU2, Pp(h, g_off), h->dA1hat, s), "first-attention gradient");
  }
  colsum_(c, s, part, h->dU2, 0, h->d, h->d, nullptr, 2, nullptr, nullptr, nullptr, ahat ? ahat : h->a1hat,
          Gp(h, g_off), Gp(h, b_off), nullptr, accumulate);
}

// The bias gradients of block j that are column sums of dX_{j+1} (the gradient
// of the block's output): b_down, and for blocks whose branches both add into
// the residual at once (Parallel-type), b_o too.  Summed by the LayerNorm
// backward that produces dX_{j+1}.
BiasSum down_biases(fal_handle* h, int j) {
  BiasSum b;
  if (j < 0) return b;
  const LayerP& p = h->lp[j];
  b.b1 = Gp(h, p.b_down);
  if (block_kind(h, j) == BK_PAR) b.b2 = Gp(h, p.b_o);
  return b;
}

void layer_backward(Ctx& c, int i) {
  fal_handle* h = c.h;
  LayerA& A = h->la[i];
  const LayerP& p = h->lp[i];
  const int BT = (int)h->BT, d = h->d, F = h->F, var = h->cfg.variant;
  cudaStream_t s = h->sm;
  // dX / dX_act hold the gradient w.r.t. X_{i+1} on entry and X_i on exit.
  const int kind = block_kind(h, i);
  if (kind == BK_PAR) {
    // One launch for the fused residual GEMM's gradients:
    // [dW_o | dW_down] = dX^T [ctx | g] and [dctx | dh] = dX [W_o | W_down] (dh with gelu').
    EpiParams edh = epi_out(h->dh, F, OUT_ACT);
    edh.op = EPI_DGELU; edh.aux = A.h; edh.ldx = F;
    // dctx also yields the attention backward's D = rowsum(dctx * ctx) per head
    EpiParams edc = epi_out(h->dctx, d, OUT_ACT);
    if (h->bf) {
      edc.rd_src = A.ctx; edc.rd_ld = d; edc.rd_out = h->dvec; edc.rd_hd = h->hd; edc.rd_T = h->T; edc.rd_H = h->H;
    }
    gemm(c, group_calls({call1(d, d, wgrad_seg(h, h->dX_act, d, A.ctx, d), wgrad_out(h, p.w_o, d)),
                         call1(d, F, wgrad_seg(h, h->dX_act, d, A.g, F), wgrad_out(h, p.w_down, F)),
                         call1(BT, d, dgrad_seg(h, h->dX_act, d, p.w_o, d), edc),
                         call1(BT, F, dgrad_seg(h, h->dX_act, d, p.w_down, F), edh)}),
         s, "fused residual wgrad + dgrad");
    // (db_o = db_down = column sums of dX, summed by the LayerNorm backward that produced dX)
    const bool two = h->cfg.schedule == FAL_SCHED_TWO_STREAM && h->ss != h->sm;
    cudaStream_t sa = two ? h->ss : s;
    if (two) fork(h);
    attn_backward(c, i, nullptr, nullptr, sa, two ? h->part1 : h->part0, true, h->bf != 0);
    gemm(c, group_calls({call1(F, d, wgrad_seg(h, h->dh, F, mlp_in(h, i), d), wgrad_out(h, p.w_up, d)),
                         call1(BT, d, dgrad_seg(h, h->dh, F, p.w_up, d), epi_out(h->dU2, d, OUT_F32))}),
         s, "MLP up wgrad + dgrad");
    colsum_(c, s, h->part0, h->dh, 1, F, F, nullptr, 0, nullptr, nullptr, nullptr, nullptr, nullptr, Gp(h, p.b_up),
            nullptr, 0);
    if (var == FAL_FAL) first_attention_grad(c, h->lnF_g, h->lnF_b, s, h->part0, 1);
    if (two) join(h);
    ln_bwd_(c, s, h->dU, h->dU2, A.X, A.ln1_mean, A.ln1_rstd, Pp(h, p.ln1_g), h->dX, h->dX, h->dX_act,
            h->part0, Gp(h, p.ln1_g), Gp(h, p.ln1_b), down_biases(h, i - 1));
    return;
  }
  if (kind == BK_FIRST || kind == BK_OWN) {  // FAL block 1, Ablation1 blocks
    const bool first = kind == BK_FIRST;
    mlp_backward(c, i, h->dX, h->dX_act, s, h->part0);
    if (first) {
      first_attention_grad(c, h->lnF_g, h->lnF_b, s, h->part0, 1);
    } else {
      cudaMemsetAsync(h->dA1hat, 0, (size_t)BT * d * 4, s);
      first_attention_grad(c, p.lnA_g, p.lnA_b, s, h->part0, 0, A.ahat);
    }
    // da = dX_{i+1} + (LN without affine)'(a) . dA1hat   (a feeds X_{i+1} and the MLP input)
    ln_bwd_(c, s, h->dA1hat, nullptr, first ? h->a1 : A.a, first ? h->a1_mean : A.a_mean,
            first ? h->a1_rstd : A.a_rstd, nullptr, h->dX, h->dA, h->dA_act, h->part0, nullptr, nullptr,
            BiasSum{Gp(h, p.b_o), nullptr});
    attn_backward(c, i, h->dA, h->dA_act, s, h->part0, false);
    ln_bwd_(c, s, h->dU, h->dU2, A.X, A.ln1_mean, A.ln1_rstd, Pp(h, p.ln1_g), h->dX, h->dX, h->dX_act,
            h->part0, Gp(h, p.ln1_g), Gp(h, p.ln1_b), down_biases(h, i - 1));
    return;
  }
  // GPT / FAL+
  mlp_backward(c, i, h->dX, h->dX_act, s, h->part0);
  // db_o = column sums of da: dY here, or dA for the block whose attention FAL+ reuses
  const bool reused = var == FAL_FALPLUS && i == h->reuse;
  ln_bwd_(c, s, h->dU2, nullptr, A.Y, A.ln2_mean, A.ln2_rstd, Pp(h, p.ln2_g), h->dX, h->dY, h->dY_act,
          h->part0, Gp(h, p.ln2_g), Gp(h, p.ln2_b), reused ? BiasSum() : BiasSum{Gp(h, p.b_o), nullptr});
  const float* da = h->dY;
  const void* da_act = h->dY_act;
  if (var == FAL_FALPLUS && i > h->reuse) first_attention_grad(c, p.lnF_g, p.lnF_b, s, h->part0, 0);
  if (var == FAL_FALPLUS && i == h->reuse) {
    ln_bwd_(c, s, h->dA1hat, nullptr, h->a1, h->a1_mean, h->a1_rstd, nullptr, h->dY, h->dA, h->dA_act, h->part0,
            nullptr, nullptr, BiasSum{Gp(h, p.b_o), nullptr});
    da = h->dA;
    da_act = h->dA_act;
  }
  attn_backward(c, i, da, da_act, s, h->part0, false);
  ln_bwd_(c, s, h->dU, nullptr, A.X, A.ln1_mean, A.ln1_rstd, Pp(h, p.ln1_g), h->dY, h->dX, h->dX_act,
          h->part0, Gp(h, p.ln1_g), Gp(h, p.ln1_b), down_biases(h, i - 1));
}

// Chunked LM head backward.  Chunk j covers vocabulary rows [j hc, j hc + nc)
// of wte: its logits are recomputed with the loss-gradient epilogue into
// chunk buffer j % 2, then dwte rows = chunk^T xf (stores) and dxf (+)= chunk
// wte rows.  The recompute of chunk j + 1 runs in the same launch as the
// gradients of chunk j, which read the other buffer.
void head_backward_chunked(Ctx& c, cudaStream_t s) {
  fal_handle* h = c.h;
  const int BT = (int)h->BT, d = h->d, V = h->V, C = h->hc;
  const int n = (V + C - 1) / C;
  auto width = [&](int j) { return V - j * C < C ? V - j * C : C; };
  auto recompute = [&](int j) {
    EpiParams e = epi_out(h->hbuf[j & 1], C, OUT_ACT);
    e.op = EPI_CE_GRAD;
    e.ce_lse = h->ce_lse; e.ce_tgt = h->tgt; e.ce_v0 = j * C; e.ce_scale = 1.f / (float)BT;
    return call1(BT, width(j), seg(h->xf, d, 0, Wp(h, h->wte + (size_t)j * C * d), d, 0, d), e);
  };
  auto grads = [&](int j) {
    const int nc = width(j);
    return group_calls(
        {call1(nc, d, seg(h->hbuf[j & 1], C, 1, h->xf, d, 1, BT), epi_out(Gp(h, h->wte + (size_t)j * C * d), d, OUT_F32)),
         call1(BT, d, seg(h->hbuf[j & 1], C, 0, Wp(h, h->wte + (size_t)j * C * d), d, 1, nc),
               epi_out(h->dU, d, j ? OUT_F32_ACCUM : OUT_F32))});
  };
  gemm(c, recompute(0), s, "LM head logits gradient (chunk)");
  for (int j = 0; j < n && c.ok(); ++j)
    gemm(c, j + 1 < n ? group_calls({grads(j), recompute(j + 1)}) : grads(j), s, "LM head wgrad + dgrad (chunk)");
}

int backward_impl(fal_handle* h) {
  Ctx c{h};
  cudaStream_t s = h->sm;
  const int BT = (int)h->BT, d = h->d;
  // LM head: dwte = dlogits^T xf and dxf = dlogits wte in one launch (stores;
  // the embedding adds later)
  if (h->hc) {
    head_backward_chunked(c, s);
  } else {
    gemm(c, group_calls({call1(h->V, d, seg(h->dlogits, h->Vp, 1, h->xf, d, 1, BT), epi_out(Gp(h, h->wte), d, OUT_F32)),
                         call1(BT, d, seg(h->dlogits, h->Vp, 0, Wp(h, h->wte), d, 1, h->V), epi_out(h->dU, d, OUT_F32))}),
         s, "LM head wgrad + dgrad");
  }
  ln_bwd_(c, s, h->dU, nullptr, h->Xout, h->lnf_mean, h->lnf_rstd, Pp(h, h->lnf_g), nullptr, h->dX, h->dX_act,
          h->part0, Gp(h, h->lnf_g), Gp(h, h->lnf_b), down_biases(h, h->L - 1));
  if (h->cfg.variant != FAL_GPT) cudaMemsetAsync(h->dA1hat, 0, (size_t)BT * d * 4, s);
  if (h->cfg.variant == FAL_FAL) {
    cudaMemsetAsync(Gp(h, h->lnF_g), 0, (size_t)d * 4, s);
    cudaMemsetAsync(Gp(h, h->lnF_b), 0, (size_t)d * 4, s);
  }
  for (int i = h->L - 1; i >= 0 && c.ok(); --i) layer_backward(c, i);
  if (c.ok())
    c.check(embed_bwd(h->B, h->T, d, h->V, h->tok, h->dX, Gp(h, h->wte), Gp(h, h->wpe), s), "embedding backward");
  return c.rc;
}

int read_dev_err(fal_handle* h) {
  int e = 0;
  if (cudaStreamSynchronize(h->ss) != cudaSuccess || cudaStreamSynchronize(h->sm) != cudaSuccess ||
      cudaMemcpy(&e, h->dev_err, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) {
    return fail(h, FAL_ERR_CUDA, std::string("CUDA error: ") + cudaGetErrorString(cudaGetLastError()));
  }
  if (e) {
    cudaMemset(h->dev_err, 0, sizeof(int));
    if (e == DEV_ERR_TOKEN) return fail(h, FAL_ERR_ARG, "token or target id outside [0, vocab)");
    return fail(h, FAL_ERR_TIMEOUT, "a bounded device wait expired inside a GEMM kernel");
  }
  return FAL_OK;
}

}  // namespace

// ================================================================ C ABI
extern "C" {

int fal_workspace_size(const fal_config* cfg, size_t* bytes) {
  std::string msg;
  if (!bytes) return FAL_ERR_ARG;
  int r = validate(cfg, &msg);
  if (r) return r;
  fal_handle tmp;
  init_dims(&tmp, cfg);
  build_table(&tmp);
  carve(&tmp, nullptr);
  *bytes = tmp.total_bytes;
  return FAL_OK;
}

int fal_create(const fal_config* cfg, void* workspace, size_t bytes, void* stream_main, void* stream_side,
               fal_handle** out) {
  if (!out) return FAL_ERR_ARG;
  *out = nullptr;
  std::string msg;
  int r = validate(cfg, &msg);
  if (r) return r;
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) % ALIGN)) return FAL_ERR_ARG;
  fal_handle* h = new fal_handle();
  init_dims(h, cfg);
  build_table(h);
  carve(h, nullptr);
  if (bytes < h->total_bytes) {
    delete h;
    return FAL_ERR_WORKSPACE;
  }
  carve(h, reinterpret_cast<uint8_t*>(workspace));
  h->sm = reinterpret_cast<cudaStream_t>(stream_main);
  h->ss = stream_side ? reinterpret_cast<cudaStream_t>(stream_side) : h->sm;
  if (cudaEventCreateWithFlags(&h->ev_fork, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_join, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_mid, cudaEventDisableTiming) != cudaSuccess) {
    delete h;
    return FAL_ERR_CUDA;
  }
  // zero parameters, gradients (their padding is never written), moments, error word
  cudaStream_t s = h->sm;
  cudaMemsetAsync(h->P, 0, h->n_params * 4, s);
  cudaMemsetAsync(h->G, 0, h->n_params * 4, s);
  cudaMemsetAsync(h->Mo, 0, h->n_params * 4, s);
  cudaMemsetAsync(h->Vo, 0, h->n_params * 4, s);
  for (void* b : h->Shb)
    if (b) cudaMemsetAsync(b, 0, h->n_params * 2, s);
  cudaMemsetAsync(h->dev_err, 0, 16, s);
  cudaMemsetAsync(h->ord_flags, 0, (size_t)h->ord_cap * sizeof(int), s);
  if (cudaStreamSynchronize(s) != cudaSuccess) {
    cudaEventDestroy(h->ev_fork);
    cudaEventDestroy(h->ev_join);
    if (h->ev_mid) cudaEventDestroy(h->ev_mid);
    delete h;
    return FAL_ERR_CUDA;
  }
  *out = h;
  return FAL_OK;
}

void fal_destroy(fal_handle* h) {
  if (!h) return;
  cudaStreamSynchronize(h->sm);
  if (h->ss != h->sm) cudaStreamSynchronize(h->ss);
  for (cudaEvent_t e : h->ev_pool) cudaEventDestroy(e);
  if (h->ev_fork) cudaEventDestroy(h->ev_fork);
  if (h->ev_join) cudaEventDestroy(h->ev_join);
  if (h->ev_mid) cudaEventDestroy(h->ev_mid);
  delete h;
}

int fal_get_grad_norm(fal_handle* h, float* norm_host) {
  if (!h || !norm_host) return FAL_ERR_ARG;
  if (!h->has_norm) return fail(h, FAL_ERR_STATE, "no step with gradient clipping yet");
  int r = read_dev_err(h);
  if (r) return r;
  if (cudaMemcpy(norm_host, h->gn_norm, sizeof(float), cudaMemcpyDeviceToHost) != cudaSuccess)
    return fail(h, FAL_ERR_CUDA, "norm copy failed");
  return FAL_OK;
}

int fal_sync(fal_handle* h) {
  if (!h) return FAL_ERR_ARG;
  return read_dev_err(h);
}

int fal_get_loss(fal_handle* h, float* loss_host) {
  if (!h || !loss_host) return FAL_ERR_ARG;
  if (!h->has_loss) return fail(h, FAL_ERR_STATE, "no forward pass yet");
  int r = read_dev_err(h);
  if (r) return r;
  if (cudaMemcpy(loss_host, h->loss, sizeof(float), cudaMemcpyDeviceToHost) != cudaSuccess)
    return fail(h, FAL_ERR_CUDA, "loss copy failed");
  return FAL_OK;
}

int fal_forward(fal_handle* h, const int32_t* tokens, const int32_t* targets, float* loss_host) {
  if (!h || !tokens || !targets) return h ? fail(h, FAL_ERR_ARG, "null tokens/targets") : FAL_ERR_ARG;
  int r = forward_impl(h, tokens, targets);
  if (r) return r;
  h->state = 1;
  h->has_loss = true;
  if (loss_host) {
    if (cudaMemcpyAsync(loss_host, h->loss, sizeof(float), cudaMemcpyDeviceToHost, h->sm) != cudaSuccess)
      return fail(h, FAL_ERR_CUDA, "loss copy failed");
    return read_dev_err(h);
  }
  return FAL_OK;
}

int fal_prefill(fal_handle* h, const int32_t* tokens, float* last_logits) {
  if (!h || !tokens) return h ? fail(h, FAL_ERR_ARG, "null tokens") : FAL_ERR_ARG;
  Ctx c{h};
  cudaStream_t s = h->sm;
  const int d = h->d;
  if (cudaMemcpyAsync(h->tok, tokens, (size_t)h->BT * sizeof(int32_t), cudaMemcpyDefault, s) != cudaSuccess)
    return fail(h, FAL_ERR_CUDA, "token copy failed");
  h->state = 0;  // the saved activations are overwritten: no backward after this
  c.check(embed_fwd((int)h->BT, h->T, d, h->V, h->tok, Pp(h, h->wte), Pp(h, h->wpe), h->la[0].X, h->dev_err, s),
          "embedding");
  for (int i = 0; i < h->L && c.ok(); ++i) layer_forward(c, i);
  ln_fwd_(c, s, h->Xout, Pp(h, h->lnf_g), Pp(h, h->lnf_b), h->xf, nullptr, h->lnf_mean, h->lnf_rstd, nullptr, nullptr,
          nullptr, nullptr);
  // LM head on the last position of every sequence: rows T-1, 2T-1, ... of xf
  // (row pitch T*d), fp32 logits [B, Vp] in the staging buffer when they fit,
  // else in the logits buffer or the first chunk buffer of the chunked head
  const size_t need = (size_t)h->B * h->Vp;
  void* alt = h->hc ? h->hbuf[0] : h->logits;
  const size_t avail = (size_t)h->BT * (h->hc ? (size_t)h->hc : (size_t)h->Vp) * h->asz / 4;
  float* out = need <= h->stage_floats ? h->stage : need <= avail ? reinterpret_cast<float*>(alt) : nullptr;
  if (!out) return fail(h, FAL_ERR_UNSUPPORTED, "prefill logits do not fit the workspace");
  const uint8_t* last = reinterpret_cast<const uint8_t*>(h->xf) + (size_t)(h->T - 1) * d * h->asz;
  gemm(c, call1(h->B, h->V, seg(last, (long)h->T * d, 0, Wp(h, h->wte), d, 0, d), epi_out(out, h->Vp, OUT_F32)), s,
       "LM head (last positions)");
  if (!c.ok()) return c.rc;
  if (last_logits) {
    if (cudaMemcpy2DAsync(last_logits, (size_t)h->V * 4, out, (size_t)h->Vp * 4, (size_t)h->V * 4, h->B,
                          cudaMemcpyDefault, s) != cudaSuccess)
      return fail(h, FAL_ERR_CUDA, "logits copy failed");
    return read_dev_err(h);
  }
  return FAL_OK;
}

int fal_backward(fal_handle* h) {
  if (!h) return FAL_ERR_ARG;
  if (h->state < 1) return fail(h, FAL_ERR_STATE, "fal_backward needs a preceding fal_forward");
  int r = backward_impl(h);
  if (r) return r;
  h->state = 2;
  return FAL_OK;
}

namespace {
// AdamW over the flat range [begin, end) of the parameter buffer; elements
// below decay_end get weight decay.
int adamw_range(fal_handle* h, size_t begin, size_t end, size_t decay_end) {
  const fal_config& c = h->cfg;
  const float bc1 = 1.f - (float)pow((double)c.beta1, (double)h->step_t);
  const float bc2 = 1.f - (float)pow((double)c.beta2, (double)h->step_t);
  void* sh = h->bf ? (void*)((uint8_t*)h->Shb[h->sh_cur ^ 1] + begin * 2) : nullptr;
  return adamw(end - begin, decay_end > begin ? decay_end - begin : 0, h->P + begin, h->G + begin, h->Mo + begin,
               h->Vo + begin, sh, c.lr, c.beta1, c.beta2, c.eps, c.weight_decay, bc1, bc2, h->sm,
               h->cfg.clip_norm > 0.f ? h->gn_scale : nullptr);
}

// Gradient clipping (App. A): the global norm of the whole flat gradient
// buffer (its padding is zero) and the factor AdamW applies to every gradient.
int clip_grads(fal_handle* h) {
  if (h->cfg.clip_norm <= 0.f) return 0;
  ProfScope ps(h, h->sm, 3, 0.0, "gradient norm");
  const int r = grad_norm_clip(h->n_params, h->G, h->cfg.clip_norm, h->gn_part, h->gn_norm, h->gn_scale, h->sm);
  if (r == 0) h->has_norm = true;
  return r;
}
}  // namespace

int fal_step(fal_handle* h) {
  if (!h) return FAL_ERR_ARG;
  if (h->state < 2) return fail(h, FAL_ERR_STATE, "fal_step needs a preceding fal_backward");
  h->step_t += 1;
  if (clip_grads(h)) return fail(h, FAL_ERR_CUDA, "gradient norm launch failed");
  if (adamw_range(h, 0, h->n_params, h->n_decay)) return fail(h, FAL_ERR_CUDA, "AdamW launch failed");
  h->sh_cur ^= 1;
  h->state = 0;
  return FAL_OK;
}

int fal_train_step(fal_handle* h, const int32_t* tokens, const int32_t* targets, float* loss_host) {
  int r = fal_forward(h, tokens, targets, nullptr);
  if (r) return r;
  // The block matrices (one contiguous range of the flat buffer, after wte and
  // wpe) are updated by their weight-gradient GEMMs during the backward; one
  // AdamW launch per remaining range follows.
  h->step_t += 1;
  {
    const fal_config& c = h->cfg;
    h->opt_rbc1 = 1.f / (1.f - (float)pow((double)c.beta1, (double)h->step_t));
    h->opt_rbc2 = 1.f / (1.f - (float)pow((double)c.beta2, (double)h->step_t));
  }
  // (bf16 path only: the fp32 debug path's GEMMs read the fp32 master weights,
  // which the fused update would overwrite under a concurrent reader.  With
  // gradient clipping the update needs the norm of every gradient first.)
  const bool fused = h->bf != 0 && !(h->cfg.clip_norm > 0.f);
  h->fuse_opt = fused;
  r = backward_impl(h);
  h->fuse_opt = false;
  if (r) return r;
  if (clip_grads(h)) return fail(h, FAL_ERR_CUDA, "gradient norm launch failed");
  const size_t blocks_begin = h->lp[0].w_qkv;
  const bool bad = fused ? (adamw_range(h, 0, blocks_begin, blocks_begin) ||
                            adamw_range(h, h->n_decay, h->n_params, h->n_decay))
                         : adamw_range(h, 0, h->n_params, h->n_decay);
  if (bad) return fail(h, FAL_ERR_CUDA, "AdamW launch failed");
  h->sh_cur ^= 1;
  h->state = 0;
  if (loss_host) {
    if (cudaMemcpyAsync(loss_host, h->loss, sizeof(float), cudaMemcpyDeviceToHost, h->sm) != cudaSuccess)
      return fail(h, FAL_ERR_CUDA, "loss copy failed");
    return read_dev_err(h);
  }
  return FAL_OK;
}

int fal_param_count(fal_handle* h, int* n_tensors, size_t* n_elems) {
  if (!h) return FAL_ERR_ARG;
  if (n_tensors) *n_tensors = (int)h->tensors.size();
  if (n_elems) *n_elems = h->n_params;
  return FAL_OK;
}

int fal_param_info(fal_handle* h, int idx, fal_tensor_info* info) {
  if (!h || !info || idx < 0 || idx >= (int)h->tensors.size()) return FAL_ERR_ARG;
  *info = h->tensors[idx];
  return FAL_OK;
}

int fal_set_params(fal_handle* h, const float* src, size_t n) {
  if (!h || !src) return FAL_ERR_ARG;
  if (n != h->n_params) return fail(h, FAL_ERR_ARG, "parameter count mismatch");
  cudaStream_t s = h->sm;
  if (cudaMemcpyAsync(h->P, src, n * 4, cudaMemcpyDefault, s) != cudaSuccess) return fail(h, FAL_ERR_CUDA, "copy failed");
  if (h->bf && f32_to_bf16(n, h->P, h->Shb[h->sh_cur], s)) return fail(h, FAL_ERR_CUDA, "bf16 refresh failed");
  cudaMemsetAsync(h->Mo, 0, n * 4, s);
  cudaMemsetAsync(h->Vo, 0, n * 4, s);
  h->step_t = 0;
  if (cudaStreamSynchronize(s) != cudaSuccess) return fail(h, FAL_ERR_CUDA, "copy failed");
  return FAL_OK;
}

int fal_get_params(fal_handle* h, float* dst, size_t n) {
  if (!h || !dst) return FAL_ERR_ARG;
  if (n != h->n_params) return fail(h, FAL_ERR_ARG, "parameter count mismatch");
  int r = read_dev_err(h);
  if (r) return r;
  if (cudaMemcpy(dst, h->P, n * 4, cudaMemcpyDefault) != cudaSuccess) return fail(h, FAL_ERR_CUDA, "copy failed");
  return FAL_OK;
}

int fal_get_grads(fal_handle* h, float* dst, size_t n) {
  if (!h || !dst) return FAL_ERR_ARG;
  if (n != h->n_params) return fail(h, FAL_ERR_ARG, "parameter count mismatch");
  int r = read_dev_err(h);
  if (r) return r;
  if (cudaMemcpy(dst, h->G, n * 4, cudaMemcpyDefault) != cudaSuccess) return fail(h, FAL_ERR_CUDA, "copy failed");
  return FAL_OK;
}

int fal_get_opt_state(fal_handle* h, float* m, float* v, size_t n, long long* step) {
  if (!h) return FAL_ERR_ARG;
  if (n != h->n_params) return fail(h, FAL_ERR_ARG, "parameter count mismatch");
  int r = read_dev_err(h);
  if (r) return r;
  if ((m && cudaMemcpy(m, h->Mo, n * 4, cudaMemcpyDefault) != cudaSuccess) ||
      (v && cudaMemcpy(v, h->Vo, n * 4, cudaMemcpyDefault) != cudaSuccess))
    return fail(h, FAL_ERR_CUDA, "copy failed");
  if (step) *step = h->step_t;
  return FAL_OK;
}

int fal_set_opt_state(fal_handle* h, const float* m, const float* v, size_t n, long long step) {
  if (!h) return FAL_ERR_ARG;
  if (n != h->n_params) return fail(h, FAL_ERR_ARG, "parameter count mismatch");
  if (step < 0) return fail(h, FAL_ERR_ARG, "negative step count");
  cudaStream_t s = h->sm;
  if ((m && cudaMemcpyAsync(h->Mo, m, n * 4, cudaMemcpyDefault, s) != cudaSuccess) ||
      (v && cudaMemcpyAsync(h->Vo, v, n * 4, cudaMemcpyDefault, s) != cudaSuccess) ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return fail(h, FAL_ERR_CUDA, "copy failed");
  h->step_t = (long)step;
  return FAL_OK;
}

int fal_get_tap(fal_handle* h, const char* name, int layer, float* dst, size_t n) {
  if (!h || !name || !dst) return FAL_ERR_ARG;
  const std::string nm = name;
  const long BT = h->BT;
  const int d = h->d, F = h->F;
  const bool lay = layer >= 0 && layer < h->L;
  const void* src = nullptr;
  int is_act = 1, cols = d;
  long ld = d;
  if (nm == "X") {
    if (layer == h->L) src = h->Xout;
    else if (lay) src = h->la[layer].X;
    is_act = 0;
  } else if (nm == "Y") { if (lay) src = h->la[layer].Y; is_act = 0; }
  else if (nm == "u") { if (lay) src = h->la[layer].u; }
  else if (nm == "m") { if (lay) src = mlp_in(h, layer); }
  else if (nm == "ctx") { if (lay) src = h->la[layer].ctx; }
  else if (nm == "qkv") { if (lay) src = h->la[layer].qkv; cols = h->DQ; ld = h->DQ; }
  else if (nm == "h") { if (lay) src = h->la[layer].h; cols = F; ld = F; }
  else if (nm == "g") { if (lay) src = h->la[layer].g; cols = F; ld = F; }
  else if (nm == "a1") { src = h->a1; is_act = 0; }
  else if (nm == "xf") { src = h->xf; }
  else if (nm == "logits") {
    if (h->hc) return fail(h, FAL_ERR_ARG, "the logits are never stored whole with head_chunk > 0");
    src = h->logits; cols = h->V; ld = h->Vp;
  }
  if (!src) return fail(h, FAL_ERR_ARG, "unknown tap or layer (or not present for this variant)");
  if (n != (size_t)BT * cols) return fail(h, FAL_ERR_ARG, "tap size mismatch");
  int r = read_dev_err(h);
  if (r) return r;
  if (!is_act) {
    if (cudaMemcpy(dst, src, n * 4, cudaMemcpyDefault) != cudaSuccess) return fail(h, FAL_ERR_CUDA, "copy failed");
    return FAL_OK;
  }
  const long rows_per = (long)(h->stage_floats / cols) > 0 ? (long)(h->stage_floats / cols) : 1;
  for (long r0 = 0; r0 < BT; r0 += rows_per) {
    const long nr = (BT - r0) < rows_per ? (BT - r0) : rows_per;
    const uint8_t* s = reinterpret_cast<const uint8_t*>(src) + (size_t)r0 * ld * h->asz;
    if (act_to_f32_2d(h->bf, (int)nr, cols, ld, s, h->stage, h->sm)) return fail(h, FAL_ERR_CUDA, "tap convert");
    if (cudaMemcpyAsync(dst + (size_t)r0 * cols, h->stage, (size_t)nr * cols * 4, cudaMemcpyDefault, h->sm) != cudaSuccess)
      return fail(h, FAL_ERR_CUDA, "tap copy");
    if (cudaStreamSynchronize(h->sm) != cudaSuccess) return fail(h, FAL_ERR_CUDA, "tap copy");
  }
  return FAL_OK;
}

int fal_profile_enable(fal_handle* h, int enable) {
  if (!h) return FAL_ERR_ARG;
  h->prof = enable < 0 ? 0 : (enable > 2 ? 2 : enable);
  return FAL_OK;
}

int fal_profile_timeline(fal_handle* h, fal_launch_record* out, int cap, int* n) {
  if (!h || !n || cap < 0 || (cap > 0 && !out)) return FAL_ERR_ARG;
  *n = 0;
  if (cudaStreamSynchronize(h->sm) != cudaSuccess || cudaStreamSynchronize(h->ss) != cudaSuccess)
    return fail(h, FAL_ERR_CUDA, "synchronize failed");
  if (h->recs.empty()) return FAL_OK;
  const cudaEvent_t t0 = h->recs.front().a;
  for (const auto& r : h->recs) {
    if (*n >= cap) break;
    fal_launch_record& o = out[*n];
    memset(&o, 0, sizeof(o));
    float a = 0.f, b = 0.f;
    if (cudaEventElapsedTime(&a, t0, r.a) != cudaSuccess || cudaEventElapsedTime(&b, t0, r.b) != cudaSuccess) continue;
    o.start_ms = a; o.end_ms = b; o.kind = r.kind; o.stream = r.stream; o.flops = r.flops;
    snprintf(o.label, sizeof(o.label), "%s", r.label ? r.label : "");
    ++*n;
  }
  return FAL_OK;
}

int fal_profile_read(fal_handle* h, fal_profile* out) {
  if (!h || !out) return FAL_ERR_ARG;
  memset(out, 0, sizeof(*out));
  if (cudaStreamSynchronize(h->sm) != cudaSuccess || cudaStreamSynchronize(h->ss) != cudaSuccess)
    return fail(h, FAL_ERR_CUDA, "synchronize failed");
  for (const auto& r : h->recs) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, r.a, r.b) != cudaSuccess) continue;
    if (r.kind == 0) { out->gemm_ms += ms; out->gemm_flops += r.flops; out->gemm_launches++; }
    else if (r.kind == 1 || r.kind == 2) { out->attn_ms += ms; out->attn_flops += r.flops; out->attn_launches++; }
  }
  h->recs.clear();
  h->ev_next = 0;
  return FAL_OK;
}

long long fal_launch_count(void) { return launches_total(); }

int fal_debug_layernorm_stall(int rows, long long wait_ns) {
  ln_debug_stall(rows < 0 ? -1 : rows, wait_ns > 0 ? wait_ns : 0);
  return FAL_OK;
}

const char* fal_last_error(const fal_handle* h) {
  if (!h) return "null handle";
  return h->err.c_str();
}

const char* fal_status_string(int status) {
  switch (status) {
    case FAL_OK: return "ok";
    case FAL_ERR_ARG: return "invalid argument";
    case FAL_ERR_STATE: return "invalid call order";
    case FAL_ERR_WORKSPACE: return "workspace too small";
    case FAL_ERR_CUDA: return "CUDA error";
    case FAL_ERR_TIMEOUT: return "device wait timed out";
    case FAL_ERR_UNSUPPORTED: return "unsupported configuration";
    default: return "unknown status";
  }
}

}  // extern "C"
