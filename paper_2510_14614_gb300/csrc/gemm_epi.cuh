// GEMM epilogue shared by the SIMT and the tcgen05 GEMM kernels.
#pragma once

#include "common.cuh"
#include "internal.h"

namespace fal {

// Applies the epilogue to NV consecutive accumulator columns [col0, col0+NV)
// of one output row.  Handles the ragged N edge per element.
template <typename act_t, int NV>
__device__ __forceinline__ void epi_row(const EpiParams& e, int M, int N, int row, int col0,
                                        float* v) {
  if (row >= M) return;
  const bool full = (col0 + NV <= N);
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
        x[0] *= gelu_grad_f(h.x); x[1] *= gelu_grad_f(h.y); x[2] *= gelu_grad_f(h.z); x[3] *= gelu_grad_f(h.w);
      }
      if (e.pre_f32) store4(reinterpret_cast<float*>(e.out2) + (long)row * e.ldo2 + c, make_float4(x[0], x[1], x[2], x[3]));
      if (e.resid) { float4 r = load4(e.resid + (long)row * e.ldr + c); x[0] += r.x; x[1] += r.y; x[2] += r.z; x[3] += r.w; }
      if (e.resid2) { float4 r = load4(e.resid2 + (long)row * e.ldr2 + c); x[0] += r.x; x[1] += r.y; x[2] += r.z; x[3] += r.w; }
      float4 o = make_float4(x[0], x[1], x[2], x[3]);
      if (e.op == EPI_GELU) {
        store4(reinterpret_cast<act_t*>(e.out) + (long)row * e.ldo + c, o);
        store4(reinterpret_cast<act_t*>(e.out2) + (long)row * e.ldo2 + c,
               make_float4(gelu_f(x[0]), gelu_f(x[1]), gelu_f(x[2]), gelu_f(x[3])));
      } else if (e.out_mode == OUT_ACT) {
        store4(reinterpret_cast<act_t*>(e.out) + (long)row * e.ldo + c, o);
      } else {
        float* p = reinterpret_cast<float*>(e.out) + (long)row * e.ldo + c;
        if (e.out_mode == OUT_F32_ACCUM) { float4 q = load4(p); o.x += q.x; o.y += q.y; o.z += q.z; o.w += q.w; }
        store4(p, o);
      }
    } else {
      for (int j = 0; j < 4 && c + j < N; ++j) {
        const int cc = c + j;
        float y = x[j];
        if (e.bias) y += e.bias[cc];
        if (e.bias2) y += e.bias2[cc];
        if (e.op == EPI_DGELU) y *= gelu_grad_f(to_f(reinterpret_cast<const act_t*>(e.aux)[(long)row * e.ldx + cc]));
        if (e.pre_f32) reinterpret_cast<float*>(e.out2)[(long)row * e.ldo2 + cc] = y;
        if (e.resid) y += e.resid[(long)row * e.ldr + cc];
        if (e.resid2) y += e.resid2[(long)row * e.ldr2 + cc];
        if (e.op == EPI_GELU) {
          reinterpret_cast<act_t*>(e.out)[(long)row * e.ldo + cc] = from_f<act_t>(y);
          reinterpret_cast<act_t*>(e.out2)[(long)row * e.ldo2 + cc] = from_f<act_t>(gelu_f(y));
        } else if (e.out_mode == OUT_ACT) {
          reinterpret_cast<act_t*>(e.out)[(long)row * e.ldo + cc] = from_f<act_t>(y);
        } else {
          float* p = reinterpret_cast<float*>(e.out) + (long)row * e.ldo + cc;
          *p = (e.out_mode == OUT_F32_ACCUM) ? *p + y : y;
        }
      }
    }
  }
}

}  // namespace fal
