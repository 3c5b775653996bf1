// GEMM epilogue shared by the SIMT and the tcgen05 GEMM kernels.
#pragma once

#include "common.cuh"
#include "internal.h"

namespace fal {

// GELU in the epilogue: the bf16 path rounds its result to bf16 at once, so it
// uses the hardware tanh approximation; the fp32 debug path keeps tanhf.
template <typename act_t> __device__ __forceinline__ float epi_gelu(float x) { return gelu_f(x); }
template <> __device__ __forceinline__ float epi_gelu<bf16>(float x) { return gelu_fast(x); }
template <typename act_t> __device__ __forceinline__ float epi_gelu_grad(float x) { return gelu_grad_f(x); }
template <> __device__ __forceinline__ float epi_gelu_grad<bf16>(float x) { return gelu_grad_fast(x); }

// ---- compile-time specialised epilogue arithmetic
// Which inputs an epilogue reads, as bits of a compile-time KIND.
// EK_ADAMW (a weight gradient with the optimizer update fused) and the two
// cross-entropy epilogues of the LM head read nothing else and are never part
// of EK_ANY.
enum EpiKind {
  EK_BIAS = 1, EK_BIAS2 = 2, EK_DGELU = 4, EK_PRE = 8, EK_RESID = 16, EK_RESID2 = 32, EK_GELU = 64,
  EK_ANY = 127,  // every input present-or-null, tested at run time
  EK_ADAMW = 128, EK_CEGRAD = 256, EK_CESTATS = 512
};

__host__ __device__ inline int epi_kind(const EpiParams& e) {
  if (e.op == EPI_ADAMW) return EK_ADAMW;
  if (e.op == EPI_CE_GRAD) return EK_CEGRAD;
  if (e.op == EPI_CE_STATS) return EK_CESTATS;
  return (e.bias ? EK_BIAS : 0) | (e.bias2 ? EK_BIAS2 : 0) | (e.op == EPI_DGELU ? EK_DGELU : 0) |
         (e.pre_f32 ? EK_PRE : 0) | (e.resid ? EK_RESID : 0) | (e.resid2 ? EK_RESID2 : 0) |
         (e.op == EPI_GELU ? EK_GELU : 0);
}

// AdamW applied to the parameter elements (row, c..c+n) of an EPI_ADAMW
// epilogue, given their gradient g (the value just stored to `out`).
template <int NE>
__device__ __forceinline__ void epi_adamw(const EpiParams& e, int row, int c, const float* g) {
  const long o = (long)row * e.ldo + c;
  if (NE == 4) {
    float4 p = load4(e.opt_p + o), m = load4(e.opt_m + o), v = load4(e.opt_v + o);
    adamw_elem(p.x, m.x, v.x, g[0], e.opt_lr, e.opt_b1, e.opt_b2, e.opt_eps, e.opt_wd, e.opt_rbc1, e.opt_rbc2);
    adamw_elem(p.y, m.y, v.y, g[1], e.opt_lr, e.opt_b1, e.opt_b2, e.opt_eps, e.opt_wd, e.opt_rbc1, e.opt_rbc2);
    adamw_elem(p.z, m.z, v.z, g[2], e.opt_lr, e.opt_b1, e.opt_b2, e.opt_eps, e.opt_wd, e.opt_rbc1, e.opt_rbc2);
    adamw_elem(p.w, m.w, v.w, g[3], e.opt_lr, e.opt_b1, e.opt_b2, e.opt_eps, e.opt_wd, e.opt_rbc1, e.opt_rbc2);
    store4(e.opt_p + o, p); store4(e.opt_m + o, m); store4(e.opt_v + o, v);
    if (e.opt_sh) store4(reinterpret_cast<bf16*>(e.opt_sh) + o, p);
  } else {
    for (int j = 0; j < NE; ++j) {
      float p = e.opt_p[o + j], m = e.opt_m[o + j], v = e.opt_v[o + j];
      adamw_elem(p, m, v, g[j], e.opt_lr, e.opt_b1, e.opt_b2, e.opt_eps, e.opt_wd, e.opt_rbc1, e.opt_rbc2);
      e.opt_p[o + j] = p; e.opt_m[o + j] = m; e.opt_v[o + j] = v;
      if (e.opt_sh) reinterpret_cast<bf16*>(e.opt_sh)[o + j] = __float2bfloat16_rn(p);
    }
  }
}

// The pointers and strides an epilogue reads, held by value so that they stay
// in registers (no address is ever taken).
struct EpiIn {
  const float* bias; const float* bias2;
  const float* resid; const float* resid2;
  const void* aux; float* pre;
  long ldr, ldr2, ldx, ldpre;
};

__device__ __forceinline__ EpiIn epi_in(const EpiParams& e) {
  EpiIn q;
  q.bias = e.bias; q.bias2 = e.bias2; q.resid = e.resid; q.resid2 = e.resid2; q.aux = e.aux;
  q.pre = e.pre_f32 ? reinterpret_cast<float*>(e.out2) : nullptr;
  q.ldr = e.ldr; q.ldr2 = e.ldr2; q.ldx = e.ldx; q.ldpre = e.ldo2;
  return q;
}

// Value for `out` at row `row`, columns [c, c+4), from the accumulator v.
// Reads are bounds-guarded; EK_PRE stores the pre-residual fp32 copy.
template <typename act_t, int KIND>
__device__ __forceinline__ float4 epi_value4(const EpiIn q, int M, int N, int row, int c, float4 v) {
  if (row >= M || c >= N) return make_float4(0.f, 0.f, 0.f, 0.f);
  float x[4] = {v.x, v.y, v.z, v.w};
  if (c + 4 <= N) {
    if ((KIND & EK_BIAS) && (KIND != EK_ANY || q.bias)) {
      const float4 b = load4(q.bias + c); x[0] += b.x; x[1] += b.y; x[2] += b.z; x[3] += b.w;
    }
    if ((KIND & EK_BIAS2) && (KIND != EK_ANY || q.bias2)) {
      const float4 b = load4(q.bias2 + c); x[0] += b.x; x[1] += b.y; x[2] += b.z; x[3] += b.w;
    }
    if ((KIND & EK_DGELU) && (KIND != EK_ANY || q.aux)) {
      const float4 h = load4(reinterpret_cast<const act_t*>(q.aux) + (long)row * q.ldx + c);
      x[0] *= epi_gelu_grad<act_t>(h.x); x[1] *= epi_gelu_grad<act_t>(h.y);
      x[2] *= epi_gelu_grad<act_t>(h.z); x[3] *= epi_gelu_grad<act_t>(h.w);
    }
    if ((KIND & EK_PRE) && (KIND != EK_ANY || q.pre)) store4(q.pre + (long)row * q.ldpre + c, make_float4(x[0], x[1], x[2], x[3]));
    if ((KIND & EK_RESID) && (KIND != EK_ANY || q.resid)) {
      const float4 r = load4(q.resid + (long)row * q.ldr + c); x[0] += r.x; x[1] += r.y; x[2] += r.z; x[3] += r.w;
    }
    if ((KIND & EK_RESID2) && (KIND != EK_ANY || q.resid2)) {
      const float4 r = load4(q.resid2 + (long)row * q.ldr2 + c); x[0] += r.x; x[1] += r.y; x[2] += r.z; x[3] += r.w;
    }
  } else {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int cc = c + j;
      if (cc >= N) { x[j] = 0.f; continue; }
      if ((KIND & EK_BIAS) && (KIND != EK_ANY || q.bias)) x[j] += q.bias[cc];
      if ((KIND & EK_BIAS2) && (KIND != EK_ANY || q.bias2)) x[j] += q.bias2[cc];
      if ((KIND & EK_DGELU) && (KIND != EK_ANY || q.aux))
        x[j] *= epi_gelu_grad<act_t>(to_f(reinterpret_cast<const act_t*>(q.aux)[(long)row * q.ldx + cc]));
      if ((KIND & EK_PRE) && (KIND != EK_ANY || q.pre)) q.pre[(long)row * q.ldpre + cc] = x[j];
      if ((KIND & EK_RESID) && (KIND != EK_ANY || q.resid)) x[j] += q.resid[(long)row * q.ldr + cc];
      if ((KIND & EK_RESID2) && (KIND != EK_ANY || q.resid2)) x[j] += q.resid2[(long)row * q.ldr2 + cc];
    }
  }
  return make_float4(x[0], x[1], x[2], x[3]);
}

// Epilogue arithmetic for the 4 columns [c, c+4) of one row without the final
// stores: on return x[] holds the value for `out` (the GELU output, when the
// epilogue has one, is gelu(x)).  Every global read is bounds-guarded
// (row < M, column < N); the optional fp32 pre-residual copy (pre_f32) is
// stored here.
template <typename act_t>
__device__ __forceinline__ void epi_math4(const EpiParams& e, int M, int N, int row, int c, float* x) {
  if (row >= M || c >= N) {
    x[0] = x[1] = x[2] = x[3] = 0.f;
    return;
  }
  if (c + 4 <= N) {
    if (e.bias) { float4 b = load4(e.bias + c); x[0] += b.x; x[1] += b.y; x[2] += b.z; x[3] += b.w; }
    if (e.bias2) { float4 b = load4(e.bias2 + c); x[0] += b.x; x[1] += b.y; x[2] += b.z; x[3] += b.w; }
    if (e.op == EPI_DGELU) {
      float4 h = load4(reinterpret_cast<const act_t*>(e.aux) + (long)row * e.ldx + c);
      x[0] *= epi_gelu_grad<act_t>(h.x); x[1] *= epi_gelu_grad<act_t>(h.y);
      x[2] *= epi_gelu_grad<act_t>(h.z); x[3] *= epi_gelu_grad<act_t>(h.w);
    }
    if (e.pre_f32) store4(reinterpret_cast<float*>(e.out2) + (long)row * e.ldo2 + c, make_float4(x[0], x[1], x[2], x[3]));
    if (e.resid) { float4 r = load4(e.resid + (long)row * e.ldr + c); x[0] += r.x; x[1] += r.y; x[2] += r.z; x[3] += r.w; }
    if (e.resid2) { float4 r = load4(e.resid2 + (long)row * e.ldr2 + c); x[0] += r.x; x[1] += r.y; x[2] += r.z; x[3] += r.w; }
  } else {
    for (int j = 0; j < 4; ++j) {
      const int cc = c + j;
      if (cc >= N) { x[j] = 0.f; continue; }
      if (e.bias) x[j] += e.bias[cc];
      if (e.bias2) x[j] += e.bias2[cc];
      if (e.op == EPI_DGELU) x[j] *= epi_gelu_grad<act_t>(to_f(reinterpret_cast<const act_t*>(e.aux)[(long)row * e.ldx + cc]));
      if (e.pre_f32) reinterpret_cast<float*>(e.out2)[(long)row * e.ldo2 + cc] = x[j];
      if (e.resid) x[j] += e.resid[(long)row * e.ldr + cc];
      if (e.resid2) x[j] += e.resid2[(long)row * e.ldr2 + cc];
    }
  }
}

// Gradient of the mean cross-entropy for one logit x of row `row`, column c of
// the chunk: (softmax - one-hot) / rows, with the row's log-sum-exp lse and
// target column t (vocabulary index minus the chunk's first one).
__device__ __forceinline__ float ce_grad1(float x, float lse, int t, int c, float scale) {
  return (__expf(x - lse) - (c == t ? 1.f : 0.f)) * scale;
}

// Applies the epilogue to NV consecutive accumulator columns [col0, col0+NV)
// of one output row.  Handles the ragged N edge per element.
template <typename act_t, int NV>
__device__ __forceinline__ void epi_row(const EpiParams& e, int M, int N, int row, int col0,
                                        float* v) {
  if (row >= M) return;
  const bool full = (col0 + NV <= N);
  if (e.op == EPI_CE_GRAD) {
    const float lse = e.ce_lse[row];
    const int t = e.ce_tgt[row] - e.ce_v0;
    act_t* o = reinterpret_cast<act_t*>(e.out) + (long)row * e.ldo;
    for (int j = 0; j < NV && col0 + j < N; ++j) o[col0 + j] = from_f<act_t>(ce_grad1(v[j], lse, t, col0 + j, e.ce_scale));
    return;
  }
#pragma unroll
  for (int j0 = 0; j0 < NV; j0 += 4) {
    const int c = col0 + j0;
    if (c >= N) break;
    float x[4] = {v[j0], v[j0 + 1], v[j0 + 2], v[j0 + 3]};
    const bool vec = full || (c + 4 <= N);
    if (vec) {
      if (e.bias) { float4 b = load4(e.bias + c); x[0] += b.x; x[1] += b.y; x[2] += b.z; x[3] += b.w; }
      if (e.bias2) { float4 b = load4(e.bias2 + c); x[0] += b.x; x[1] += b.y; x[2] += b.z; x[3] += b.w; }
      if (e.op == EPI_DGELU) {
        float4 h = load4(reinterpret_cast<const act_t*>(e.aux) + (long)row * e.ldx + c);
        x[0] *= epi_gelu_grad<act_t>(h.x); x[1] *= epi_gelu_grad<act_t>(h.y); x[2] *= epi_gelu_grad<act_t>(h.z); x[3] *= epi_gelu_grad<act_t>(h.w);
      }
      if (e.pre_f32) store4(reinterpret_cast<float*>(e.out2) + (long)row * e.ldo2 + c, make_float4(x[0], x[1], x[2], x[3]));
      if (e.resid) { float4 r = load4(e.resid + (long)row * e.ldr + c); x[0] += r.x; x[1] += r.y; x[2] += r.z; x[3] += r.w; }
      if (e.resid2) { float4 r = load4(e.resid2 + (long)row * e.ldr2 + c); x[0] += r.x; x[1] += r.y; x[2] += r.z; x[3] += r.w; }
      float4 o = make_float4(x[0], x[1], x[2], x[3]);
      if (e.op == EPI_GELU) {
        store4(reinterpret_cast<act_t*>(e.out) + (long)row * e.ldo + c, o);
        store4(reinterpret_cast<act_t*>(e.out2) + (long)row * e.ldo2 + c,
               make_float4(epi_gelu<act_t>(x[0]), epi_gelu<act_t>(x[1]), epi_gelu<act_t>(x[2]), epi_gelu<act_t>(x[3])));
      } else if (e.out_mode == OUT_ACT) {
        store4(reinterpret_cast<act_t*>(e.out) + (long)row * e.ldo + c, o);
      } else {
        float* p = reinterpret_cast<float*>(e.out) + (long)row * e.ldo + c;
        if (e.out_mode == OUT_F32_ACCUM) { float4 q = load4(p); o.x += q.x; o.y += q.y; o.z += q.z; o.w += q.w; }
        store4(p, o);
        if (e.op == EPI_ADAMW) epi_adamw<4>(e, row, c, &o.x);
      }
    } else {
      for (int j = 0; j < 4 && c + j < N; ++j) {
        const int cc = c + j;
        float y = x[j];
        if (e.bias) y += e.bias[cc];
        if (e.bias2) y += e.bias2[cc];
        if (e.op == EPI_DGELU) y *= epi_gelu_grad<act_t>(to_f(reinterpret_cast<const act_t*>(e.aux)[(long)row * e.ldx + cc]));
        if (e.pre_f32) reinterpret_cast<float*>(e.out2)[(long)row * e.ldo2 + cc] = y;
        if (e.resid) y += e.resid[(long)row * e.ldr + cc];
        if (e.resid2) y += e.resid2[(long)row * e.ldr2 + cc];
        if (e.op == EPI_GELU) {
          reinterpret_cast<act_t*>(e.out)[(long)row * e.ldo + cc] = from_f<act_t>(y);
          reinterpret_cast<act_t*>(e.out2)[(long)row * e.ldo2 + cc] = from_f<act_t>(epi_gelu<act_t>(y));
        } else if (e.out_mode == OUT_ACT) {
          reinterpret_cast<act_t*>(e.out)[(long)row * e.ldo + cc] = from_f<act_t>(y);
        } else {
          float* p = reinterpret_cast<float*>(e.out) + (long)row * e.ldo + cc;
          *p = (e.out_mode == OUT_F32_ACCUM) ? *p + y : y;
          if (e.op == EPI_ADAMW) epi_adamw<1>(e, row, cc, &y);
        }
      }
    }
  }
}

}  // namespace fal
