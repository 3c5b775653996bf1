// Bandwidth-bound kernels of the path: embedding gather/scatter, LayerNorm
// forward/backward (one warp per row, 128-bit vector access, warp-shuffle
// reductions), column reductions for LN/bias gradients, the cross-entropy
// head, and AdamW over the flat parameter buffer.
#include <cstring>

#include "common.cuh"
#include "internal.h"

namespace fal {

namespace {

constexpr float LN_EPS = 1e-5f;

// ------------------------------------------------------------ embedding
__global__ void embed_fwd_kernel(int rows, int T, int d, int V, const int32_t* __restrict__ tok,
                                 const float* __restrict__ wte, const float* __restrict__ wpe, float* __restrict__ X,
                                 int* err) {
  const int r = blockIdx.x;
  if (r >= rows) return;
  int id = tok[r];
  const bool bad = id < 0 || id >= V;
  if (bad) {
    if (threadIdx.x == 0) set_dev_err(err, DEV_ERR_TOKEN);
  }
  const int t = r % T;
  for (int c = threadIdx.x * 4; c < d; c += blockDim.x * 4) {
    float4 e = bad ? make_float4(0.f, 0.f, 0.f, 0.f) : load4(wte + (long)id * d + c);
    float4 p = load4(wpe + (long)t * d + c);
    store4(X + (long)r * d + c, make_float4(e.x + p.x, e.y + p.y, e.z + p.z, e.w + p.w));
  }
}

__global__ void embed_bwd_tok_kernel(int rows, int d, const int32_t* __restrict__ tok, const float* __restrict__ dX,
                                     float* __restrict__ dwte, int V) {
  const int r = blockIdx.x;
  const int id = tok[r];
  if (id < 0 || id >= V) return;
  for (int c = threadIdx.x; c < d; c += blockDim.x) atomicAdd(dwte + (long)id * d + c, dX[(long)r * d + c]);
}

__global__ void embed_bwd_pos_kernel(int B, int T, int d, const float* __restrict__ dX, float* __restrict__ dwpe) {
  const long n = (long)T * d;
  for (long i = blockIdx.x * (long)blockDim.x + threadIdx.x; i < n; i += (long)gridDim.x * blockDim.x) {
    float s = 0.f;
    for (int b = 0; b < B; ++b) s += dX[(long)b * n + i];
    dwpe[i] = s;
  }
}

// ------------------------------------------------------------ LayerNorm
// NV float4 per lane covers up to NV*128 columns.
template <typename act_t, int NV>
__global__ void __launch_bounds__(256) ln_fwd_kernel(LnFwdArgs a) {
  const int warps = blockDim.x / 32;
  const int row = blockIdx.x * warps + threadIdx.x / 32, lane = threadIdx.x % 32;
  if (row >= a.rows) return;
  const int d = a.d;
  const float* x = a.x + (long)row * d;
  float4 v[NV];
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    const int c = (i * 32 + lane) * 4;
    v[i] = (c < d) ? load4(x + c) : make_float4(0.f, 0.f, 0.f, 0.f);
    s += v[i].x + v[i].y + v[i].z + v[i].w;
  }
  const float mean = warp_sum(s) / d;
  float q = 0.f;
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    const int c = (i * 32 + lane) * 4;
    if (c < d) {
      const float dx = v[i].x - mean, dy = v[i].y - mean, dz = v[i].z - mean, dw = v[i].w - mean;
      q += dx * dx + dy * dy + dz * dz + dw * dw;
    }
  }
  const float rstd = rsqrtf(warp_sum(q) / d + LN_EPS);
  if (lane == 0) {
    if (a.mean) a.mean[row] = mean;
    if (a.rstd) a.rstd[row] = rstd;
  }
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    const int c = (i * 32 + lane) * 4;
    if (c >= d) continue;
    float4 y = make_float4((v[i].x - mean) * rstd, (v[i].y - mean) * rstd, (v[i].z - mean) * rstd, (v[i].w - mean) * rstd);
    if (a.gamma) {
      const float4 g = load4(a.gamma + c), b = load4(a.beta + c);
      y = make_float4(y.x * g.x + b.x, y.y * g.y + b.y, y.z * g.z + b.z, y.w * g.w + b.w);
    }
    if (a.out) store4(reinterpret_cast<act_t*>(a.out) + (long)row * d + c, y);
    if (a.out_f32) store4(a.out_f32 + (long)row * d + c, y);
    if (a.out2) {
      float4 z = load4(a.add_src + (long)row * d + c);
      if (a.add_g) { const float4 g = load4(a.add_g + c); z = make_float4(z.x * g.x, z.y * g.y, z.z * g.z, z.w * g.w); }
      if (a.add_b) { const float4 b = load4(a.add_b + c); z = make_float4(z.x + b.x, z.y + b.y, z.z + b.z, z.w + b.w); }
      store4(reinterpret_cast<act_t*>(a.out2) + (long)row * d + c, make_float4(y.x + z.x, y.y + z.y, y.z + z.z, y.w + z.w));
    }
  }
}

// dx = rstd * (gdy - mean(gdy) - xhat * mean(gdy * xhat)) + dres, gdy = (dy + dy2) * gamma
template <typename act_t, int NV>
__global__ void __launch_bounds__(256) ln_bwd_kernel(LnBwdArgs a) {
  const int warps = blockDim.x / 32;
  const int row = blockIdx.x * warps + threadIdx.x / 32, lane = threadIdx.x % 32;
  if (row >= a.rows) return;
  const int d = a.d;
  const long off = (long)row * d;
  const float mean = a.mean[row], rstd = a.rstd[row];
  float4 xh[NV], gd[NV];
  float s1 = 0.f, s2 = 0.f;
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    const int c = (i * 32 + lane) * 4;
    if (c < d) {
      float4 x = load4(a.x + off + c);
      xh[i] = make_float4((x.x - mean) * rstd, (x.y - mean) * rstd, (x.z - mean) * rstd, (x.w - mean) * rstd);
      float4 g = load4(a.dy + off + c);
      if (a.dy2) { float4 g2 = load4(a.dy2 + off + c); g = make_float4(g.x + g2.x, g.y + g2.y, g.z + g2.z, g.w + g2.w); }
      if (a.gamma) { float4 w = load4(a.gamma + c); g = make_float4(g.x * w.x, g.y * w.y, g.z * w.z, g.w * w.w); }
      gd[i] = g;
      s1 += g.x + g.y + g.z + g.w;
      s2 += g.x * xh[i].x + g.y * xh[i].y + g.z * xh[i].z + g.w * xh[i].w;
    } else {
      xh[i] = gd[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
  const float m1 = warp_sum(s1) / d, m2 = warp_sum(s2) / d;
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    const int c = (i * 32 + lane) * 4;
    if (c >= d) continue;
    float4 r = make_float4(rstd * (gd[i].x - m1 - xh[i].x * m2), rstd * (gd[i].y - m1 - xh[i].y * m2),
                           rstd * (gd[i].z - m1 - xh[i].z * m2), rstd * (gd[i].w - m1 - xh[i].w * m2));
    if (a.dres) { float4 q = load4(a.dres + off + c); r = make_float4(r.x + q.x, r.y + q.y, r.z + q.z, r.w + q.w); }
    store4(a.dx + off + c, r);
    if (a.dx_act) store4(reinterpret_cast<act_t*>(a.dx_act) + off + c, r);
  }
}

// ------------------------------------------------------------ column sums
constexpr int CS_THREADS = 256;
constexpr int CS_CHUNKS = 64;  // row chunks of the scalar fallback

// V consecutive values of row r from a [rows, ld] source of type T (fp32 or the
// activation type), as floats.
template <typename T, int V>
__device__ __forceinline__ void load_row_vec(const T* p, float* v) {
  if constexpr (V == 1) {
    v[0] = to_f(p[0]);
  } else if constexpr (sizeof(T) == 4) {
#pragma unroll
    for (int j = 0; j < V; j += 4) {
      const float4 q = load4(reinterpret_cast<const float*>(p) + j);
      v[j] = q.x; v[j + 1] = q.y; v[j + 2] = q.z; v[j + 3] = q.w;
    }
  } else {
    // 8 bf16 per 16-byte load
#pragma unroll
    for (int j = 0; j < V; j += 8) {
      const uint4 q = *reinterpret_cast<const uint4*>(p + j);
      const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[k]));
        v[j + 2 * k] = f.x;
        v[j + 2 * k + 1] = f.y;
      }
    }
  }
}

// Per-chunk column sums: thread owns V consecutive columns, the CTA's y index
// picks a range of rows; s0 = sum a, s1 = sum a*b (a = src (+ src2), b per bmode).
// Rows are taken four at a time with every load issued before any is used.
template <typename src_t, int V>
__global__ void __launch_bounds__(CS_THREADS) colsum_kernel(ColsumArgs a) {
  const int c = (blockIdx.x * CS_THREADS + threadIdx.x) * V;
  const int chunk = blockIdx.y, nch = gridDim.y;
  const int per = (a.rows + nch - 1) / nch;
  const int r0 = chunk * per, r1 = min(a.rows, r0 + per);
  if (c >= a.d) return;
  const src_t* src = reinterpret_cast<const src_t*>(a.src);
  float s0[V], s1[V];
#pragma unroll
  for (int j = 0; j < V; ++j) s0[j] = s1[j] = 0.f;
  auto rows4 = [&](int r, int n) {
    float v[4][V], w[4][V], mu[4], rs[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      if (i >= n) continue;
      load_row_vec<src_t, V>(src + (long)(r + i) * a.ld + c, v[i]);
      if (a.src2) {
        float t[V];
        load_row_vec<float, V>(a.src2 + (long)(r + i) * a.ld + c, t);
#pragma unroll
        for (int j = 0; j < V; ++j) v[i][j] += t[j];
      }
      if (a.bmode == 1) {
        load_row_vec<float, V>(a.x + (long)(r + i) * a.d + c, w[i]);
        mu[i] = a.mean[r + i];
        rs[i] = a.rstd[r + i];
      } else if (a.bmode == 2) {
        load_row_vec<float, V>(a.bsrc + (long)(r + i) * a.d + c, w[i]);
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      if (i >= n) continue;
#pragma unroll
      for (int j = 0; j < V; ++j) {
        s0[j] += v[i][j];
        if (a.bmode == 1) s1[j] += v[i][j] * (w[i][j] - mu[i]) * rs[i];
        else if (a.bmode == 2) s1[j] += v[i][j] * w[i][j];
      }
    }
  };
  int r = r0;
  for (; r + 4 <= r1; r += 4) rows4(r, 4);
  if (r < r1) rows4(r, r1 - r);
#pragma unroll
  for (int j = 0; j < V; ++j) {
    a.partial[((long)chunk * 2 + 0) * a.d + c + j] = s0[j];
    a.partial[((long)chunk * 2 + 1) * a.d + c + j] = s1[j];
  }
}

// Plain column sums (no second source, no product term) over rows of 16-byte
// segments: eight rows are requested before any is added, with the raw bytes
// held in registers, so that ~1000 threads per SM keep ~128 KB in flight.
template <typename src_t>
__global__ void __launch_bounds__(CS_THREADS) colsum_plain_kernel(const src_t* __restrict__ src, long ld, int d,
                                                                  int rows, float* __restrict__ partial) {
  constexpr int V = 16 / (int)sizeof(src_t);
  const int c = (blockIdx.x * CS_THREADS + threadIdx.x) * V;
  const int chunk = blockIdx.y, nch = gridDim.y;
  const int per = (rows + nch - 1) / nch;
  const int r0 = chunk * per, r1 = min(rows, r0 + per);
  if (c >= d) return;
  float acc[V];
#pragma unroll
  for (int j = 0; j < V; ++j) acc[j] = 0.f;
  for (int r = r0; r < r1; r += 8) {
    uint4 q[8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
      q[i] = (r + i < r1) ? *reinterpret_cast<const uint4*>(src + (long)(r + i) * ld + c) : make_uint4(0, 0, 0, 0);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const uint32_t w[4] = {q[i].x, q[i].y, q[i].z, q[i].w};
      if constexpr (sizeof(src_t) == 4) {
#pragma unroll
        for (int k = 0; k < 4; ++k) acc[k] += __uint_as_float(w[k]);
      } else {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[k]));
          acc[2 * k] += f.x;
          acc[2 * k + 1] += f.y;
        }
      }
    }
  }
#pragma unroll
  for (int j = 0; j < V; ++j) {
    partial[((long)chunk * 2 + 0) * d + c + j] = acc[j];
    partial[((long)chunk * 2 + 1) * d + c + j] = 0.f;
  }
}

// Sums nchunk partials [nchunk][NS][d]: slot 0 -> out0 (and out0b), slot 1 ->
// out1, slot 2 -> out2 (and out2b).  One CTA per 32 columns: its 8 warps take
// every 8th chunk (one coalesced 128-byte row segment per warp and slot), then
// combine through shared memory in a fixed order.
constexpr int CF_WARPS = 8;
template <int NS>
__global__ void __launch_bounds__(CF_WARPS * 32) colsum_finish_kernel(const float* __restrict__ partial, int nchunk,
                                                                      int d, float* out1, float* out0, float* out0b,
                                                                      float* out2, float* out2b, int accumulate) {
  __shared__ float red[NS][CF_WARPS][32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int c = blockIdx.x * 32 + lane;
  float sv[NS];
#pragma unroll
  for (int q = 0; q < NS; ++q) sv[q] = 0.f;
  if (c < d) {
    int k = warp;
    for (; k + 3 * CF_WARPS < nchunk; k += 4 * CF_WARPS) {
      float a[4][NS];
#pragma unroll
      for (int j = 0; j < 4; ++j)
#pragma unroll
        for (int q = 0; q < NS; ++q) a[j][q] = partial[((long)(k + j * CF_WARPS) * NS + q) * d + c];
#pragma unroll
      for (int j = 0; j < 4; ++j)
#pragma unroll
        for (int q = 0; q < NS; ++q) sv[q] += a[j][q];
    }
    for (; k < nchunk; k += CF_WARPS)
#pragma unroll
      for (int q = 0; q < NS; ++q) sv[q] += partial[((long)k * NS + q) * d + c];
  }
#pragma unroll
  for (int q = 0; q < NS; ++q) red[q][warp][lane] = sv[q];
  __syncthreads();
  if (warp != 0 || c >= d) return;
#pragma unroll
  for (int q = 0; q < NS; ++q) {
    sv[q] = 0.f;
#pragma unroll
    for (int w = 0; w < CF_WARPS; ++w) sv[q] += red[q][w][lane];
  }
  float* outs[5] = {out0, out0b, out1, NS > 2 ? out2 : nullptr, NS > 2 ? out2b : nullptr};
  const int slot[5] = {0, 0, 1, NS > 2 ? 2 : 0, NS > 2 ? 2 : 0};
#pragma unroll
  for (int o = 0; o < 5; ++o) {
    if (!outs[o]) continue;
    outs[o][c] = accumulate ? outs[o][c] + sv[slot[o]] : sv[slot[o]];
  }
}

// ------------------------------------------------------------ cross-entropy
// One CTA per row: pass 1 online max/sum-exp, pass 2 dlogits = (softmax - onehot)/rows.
template <typename act_t>
__global__ void __launch_bounds__(256) ce_kernel(int rows, int V, long ld, const act_t* __restrict__ logits,
                                                 const int32_t* __restrict__ tgt, act_t* __restrict__ dlogits,
                                                 float* __restrict__ loss_rows, int* err) {
  const int r = blockIdx.x;
  const act_t* x = logits + (long)r * ld;
  act_t* dx = dlogits + (long)r * ld;
  float m = -INFINITY, s = 0.f;
  const int V4 = V & ~3;
  for (int c = threadIdx.x * 4; c < V4; c += blockDim.x * 4) {
    const float4 v = load4(x + c);
    const float mx = fmaxf(fmaxf(v.x, v.y), fmaxf(v.z, v.w));
    if (mx > m) { s *= __expf(m - mx); m = mx; }
    s += __expf(v.x - m) + __expf(v.y - m) + __expf(v.z - m) + __expf(v.w - m);
  }
  for (int c = V4 + threadIdx.x; c < V; c += blockDim.x) {
    const float v = to_f(x[c]);
    if (v > m) { s *= __expf(m - v); m = v; }
    s += __expf(v - m);
  }
  __shared__ float sm[32], ss[32];
  // warp combine
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o), s2 = __shfl_xor_sync(0xffffffffu, s, o);
    const float mn = fmaxf(m, m2);
    s = (m == -INFINITY ? 0.f : s * __expf(m - mn)) + (m2 == -INFINITY ? 0.f : s2 * __expf(m2 - mn));
    m = mn;
  }
  const int w = threadIdx.x / 32, lane = threadIdx.x % 32, nw = blockDim.x / 32;
  if (lane == 0) { sm[w] = m; ss[w] = s; }
  __syncthreads();
  if (w == 0) {
    m = lane < nw ? sm[lane] : -INFINITY;
    s = lane < nw ? ss[lane] : 0.f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m, o), s2 = __shfl_xor_sync(0xffffffffu, s, o);
      const float mn = fmaxf(m, m2);
      s = (m == -INFINITY ? 0.f : s * __expf(m - mn)) + (m2 == -INFINITY ? 0.f : s2 * __expf(m2 - mn));
      m = mn;
    }
    if (lane == 0) { sm[0] = m; ss[0] = s; }
  }
  __syncthreads();
  m = sm[0];
  const float inv = 1.f / ss[0];
  int t = tgt[r];
  if (t < 0 || t >= V) {
    if (threadIdx.x == 0) set_dev_err(err, DEV_ERR_TOKEN);
    t = -1;
  }
  if (threadIdx.x == 0) loss_rows[r] = (m + logf(ss[0])) - (t >= 0 ? to_f(x[t]) : 0.f);
  const float scale = 1.f / rows;
  for (int c = threadIdx.x * 4; c < V4; c += blockDim.x * 4) {
    const float4 v = load4(x + c);
    float4 p = make_float4(__expf(v.x - m) * inv, __expf(v.y - m) * inv, __expf(v.z - m) * inv, __expf(v.w - m) * inv);
    if (t >= c && t < c + 4) {
      if (t == c) p.x -= 1.f; else if (t == c + 1) p.y -= 1.f; else if (t == c + 2) p.z -= 1.f; else p.w -= 1.f;
    }
    store4(dx + c, make_float4(p.x * scale, p.y * scale, p.z * scale, p.w * scale));
  }
  for (int c = V4 + threadIdx.x; c < V; c += blockDim.x) {
    float p = __expf(to_f(x[c]) - m) * inv;
    if (c == t) p -= 1.f;
    dx[c] = from_f<act_t>(p * scale);
  }
  for (int c = V + threadIdx.x; c < ld; c += blockDim.x) dx[c] = from_f<act_t>(0.f);
}

// Loss of the chunked LM head, one thread per row: the per-slice (max, sum of
// exp(x - max)) pairs of the logits GEMM's epilogue merge into
// lse = M + log(sum_j s_j exp(m_j - M)), and loss_row = lse - (target logit).
// The statistics are slice-major, so a warp reads 32 consecutive rows.
__global__ void __launch_bounds__(128) ce_combine_kernel(int rows, int nsl, const float2* __restrict__ st, long ld,
                                                         const float* __restrict__ tl, const int32_t* __restrict__ tgt,
                                                         int V, float* __restrict__ lse, float* __restrict__ loss_rows,
                                                         int* err) {
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= rows) return;
  float m = -INFINITY, s = 0.f;
#pragma unroll 4
  for (int j = 0; j < nsl; ++j) {
    const float2 v = st[(long)j * ld + r];
    const float mn = fmaxf(m, v.x);
    s = s * __expf(m - mn) + v.y * __expf(v.x - mn);
    m = mn;
  }
  const float l = m + logf(s);
  lse[r] = l;
  const int t = tgt[r];
  float x = 0.f;
  if (t < 0 || t >= V) set_dev_err(err, DEV_ERR_TOKEN);
  else x = tl[r];
  loss_rows[r] = l - x;
}

__global__ void mean_kernel(int n, const float* __restrict__ x, float* __restrict__ out) {
  __shared__ float sh[32];
  float s = 0.f;
  for (int i = threadIdx.x; i < n; i += blockDim.x) s += x[i];
  s = warp_sum(s);
  if (threadIdx.x % 32 == 0) sh[threadIdx.x / 32] = s;
  __syncthreads();
  if (threadIdx.x < 32) {
    s = threadIdx.x < blockDim.x / 32 ? sh[threadIdx.x] : 0.f;
    s = warp_sum(s);
    if (threadIdx.x == 0) *out = s / n;
  }
}

// ------------------------------------------------------------ misc
__global__ void add_scaled_cols_kernel(long n, int d, const float* __restrict__ src, const float* __restrict__ colvec,
                                       float* __restrict__ dst) {
  for (long i = blockIdx.x * (long)blockDim.x + threadIdx.x; i < n / 4; i += (long)gridDim.x * blockDim.x) {
    const long e = i * 4;
    const int c = e % d;
    const float4 s = load4(src + e), g = load4(colvec + c);
    float4 o = load4(dst + e);
    o.x += s.x * g.x; o.y += s.y * g.y; o.z += s.z * g.z; o.w += s.w * g.w;
    store4(dst + e, o);
  }
}

// p <- p - lr * (mhat / (sqrt(vhat) + eps) + wd * p) for i < n_decay, no decay after;
// shadow (bf16 copy of p) refreshed in the same pass.
__global__ void adamw_kernel(size_t n, size_t n_decay, float* __restrict__ p, const float* __restrict__ g,
                             float* __restrict__ m, float* __restrict__ v, bf16* __restrict__ shadow, float lr,
                             float b1, float b2, float eps, float wd, float rbc1, float rbc2,
                             const float* __restrict__ gscale) {
  const size_t n4 = n / 4;
  const float gs = gscale ? *gscale : 1.f;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n4; i += (size_t)gridDim.x * blockDim.x) {
    const size_t e = i * 4;
    float4 pp = load4(p + e), gg = load4(g + e), mm = load4(m + e), vv = load4(v + e);
    gg.x *= gs; gg.y *= gs; gg.z *= gs; gg.w *= gs;
    float* pa = &pp.x; float* ga = &gg.x; float* ma = &mm.x; float* va = &vv.x;
#pragma unroll
    for (int j = 0; j < 4; ++j)
      adamw_elem(pa[j], ma[j], va[j], ga[j], lr, b1, b2, eps, (e + j < n_decay) ? wd : 0.f, rbc1, rbc2);
    store4(p + e, pp); store4(m + e, mm); store4(v + e, vv);
    if (shadow) store4(shadow + e, pp);
  }
}

// Sum of squares of g over this block's contiguous slice (16-byte loads, fp32
// per thread, fp64 across threads): one partial per block, in block order.
constexpr int GN_BLOCKS = 1024, GN_THREADS = 256;
__global__ void __launch_bounds__(GN_THREADS) grad_sumsq_kernel(size_t n4, const float* __restrict__ g,
                                                                 double* __restrict__ partial) {
  const size_t per = (n4 + gridDim.x - 1) / gridDim.x;
  const size_t b0 = blockIdx.x * per, b1 = b0 + per < n4 ? b0 + per : n4;
  float acc = 0.f;
  for (size_t i = b0 + threadIdx.x; i < b1; i += blockDim.x) {
    const float4 v = load4(g + 4 * i);
    acc = fmaf(v.x, v.x, fmaf(v.y, v.y, fmaf(v.z, v.z, fmaf(v.w, v.w, acc))));
  }
  double s = acc;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  __shared__ double sh[GN_THREADS / 32];
  if (threadIdx.x % 32 == 0) sh[threadIdx.x / 32] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int w = 0; w < GN_THREADS / 32; ++w) t += sh[w];
    partial[blockIdx.x] = t;
  }
}

// norm = sqrt(sum of the partials in block order); scale = max_norm / norm when
// the norm exceeds max_norm, else 1.
__global__ void grad_clip_finish_kernel(int nb, const double* __restrict__ partial, float max_norm,
                                        float* __restrict__ norm_out, float* __restrict__ scale_out) {
  __shared__ double sh[32];
  double s = 0.0;
  const int per = (nb + 31) / 32;
  if (threadIdx.x < 32)
    for (int b = threadIdx.x * per; b < (threadIdx.x + 1) * per && b < nb; ++b) s += partial[b];
  if (threadIdx.x < 32) sh[threadIdx.x] = s;
  __syncwarp();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int w = 0; w < 32; ++w) t += sh[w];
    const double norm = sqrt(t);
    *norm_out = (float)norm;
    *scale_out = norm > (double)max_norm ? (float)((double)max_norm / norm) : 1.f;
  }
}

__global__ void f32_to_bf16_kernel(size_t n, const float* __restrict__ s, bf16* __restrict__ d) {
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x)
    d[i] = __float2bfloat16_rn(s[i]);
}

template <typename act_t>
__global__ void act_to_f32_2d_kernel(int rows, int cols, long ld, const act_t* __restrict__ s, float* __restrict__ d) {
  const long n = (long)rows * cols;
  for (long i = blockIdx.x * (long)blockDim.x + threadIdx.x; i < n; i += (long)gridDim.x * blockDim.x) {
    const long r = i / cols, c = i % cols;
    d[i] = to_f(s[r * ld + c]);
  }
}

int grid_for(long n, int block) {
  long g = (n + block - 1) / block;
  if (g > 8192) g = 8192;
  if (g < 1) g = 1;
  return (int)g;
}

template <typename act_t>
int ln_fwd_t(const LnFwdArgs& a, cudaStream_t s) {
  const int nv = (a.d + 127) / 128;
  const int blocks = (a.rows + 7) / 8;
  if (nv <= 1) ln_fwd_kernel<act_t, 1><<<blocks, 256, 0, s>>>(a);
  else if (nv <= 2) ln_fwd_kernel<act_t, 2><<<blocks, 256, 0, s>>>(a);
  else if (nv <= 4) ln_fwd_kernel<act_t, 4><<<blocks, 256, 0, s>>>(a);
  else if (nv <= 8) ln_fwd_kernel<act_t, 8><<<blocks, 256, 0, s>>>(a);
  else if (nv <= 16) ln_fwd_kernel<act_t, 16><<<blocks, 256, 0, s>>>(a);
  else return 6;
  return 0;
}
template <typename act_t>
int ln_bwd_t(const LnBwdArgs& a, cudaStream_t s) {
  const int nv = (a.d + 127) / 128;
  const int blocks = (a.rows + 7) / 8;
  if (nv <= 1) ln_bwd_kernel<act_t, 1><<<blocks, 256, 0, s>>>(a);
  else if (nv <= 2) ln_bwd_kernel<act_t, 2><<<blocks, 256, 0, s>>>(a);
  else if (nv <= 4) ln_bwd_kernel<act_t, 4><<<blocks, 256, 0, s>>>(a);
  else if (nv <= 8) ln_bwd_kernel<act_t, 8><<<blocks, 256, 0, s>>>(a);
  else if (nv <= 16) ln_bwd_kernel<act_t, 16><<<blocks, 256, 0, s>>>(a);
  else return 6;
  return 0;
}

int last_err() { return cudaGetLastError() == cudaSuccess ? 0 : 4; }

}  // namespace

int ln_fwd(int act_bf16, const LnFwdArgs& a, cudaStream_t s) {
  if (a.rows <= 0) return 0;
  if (a.d % 4) return 1;
  if (ln_fwd_bulk(act_bf16, a, s) == 0) {
    count_launches(1);
    return last_err();
  }
  int r = act_bf16 ? ln_fwd_t<bf16>(a, s) : ln_fwd_t<float>(a, s);
  count_launches(1);
  return r ? r : last_err();
}

int ln_bwd(int act_bf16, const LnBwdArgs& a, cudaStream_t s) {
  if (a.rows <= 0) return 0;
  if (a.d % 4) return 1;
  if (ln_bwd_bulk(act_bf16, a, s) == 0) {
    count_launches(a.cs_part ? 2 : 1);
    return last_err();
  }
  int r = act_bf16 ? ln_bwd_t<bf16>(a, s) : ln_bwd_t<float>(a, s);
  count_launches(1);
  if (r) return r;
  if (a.cs_part && (a.cs_out1 || a.cs_out0)) {
    // column sums of the affine parameters' gradients by the separate reduction
    ColsumArgs c;
    memset(&c, 0, sizeof(c));
    c.rows = a.rows; c.d = a.d; c.src = a.dy; c.src_act = 0; c.ld = a.d; c.src2 = a.dy2;
    c.bmode = 1; c.x = a.x; c.mean = a.mean; c.rstd = a.rstd;
    c.partial = a.cs_part; c.out1 = a.cs_out1; c.out0 = a.cs_out0; c.accumulate = a.cs_accumulate;
    if ((r = colsum(act_bf16, c, s)) != 0) return r;
  }
  if (a.cs_part && (a.dxs_out || a.dxs_out2)) {
    // and of dx itself
    ColsumArgs c;
    memset(&c, 0, sizeof(c));
    c.rows = a.rows; c.d = a.d; c.src = a.dx; c.src_act = 0; c.ld = a.d;
    c.partial = a.cs_part; c.out0 = a.dxs_out; c.out0b = a.dxs_out2; c.accumulate = a.cs_accumulate;
    if ((r = colsum(act_bf16, c, s)) != 0) return r;
  }
  return last_err();
}

int colsum_finish(const float* partial, int nchunk, int d, float* out1, float* out0, float* out0b, int accumulate,
                  cudaStream_t s, int nslot, float* out2, float* out2b) {
  if (d <= 0) return 0;
  if (nslot == 3)
    colsum_finish_kernel<3><<<(d + 31) / 32, CF_WARPS * 32, 0, s>>>(partial, nchunk, d, out1, out0, out0b, out2, out2b,
                                                                     accumulate);
  else
    colsum_finish_kernel<2><<<(d + 31) / 32, CF_WARPS * 32, 0, s>>>(partial, nchunk, d, out1, out0, out0b, nullptr,
                                                                     nullptr, accumulate);
  return last_err();
}

size_t colsum_partial_floats(int d) { return (size_t)kMaxColsumChunks * 3 * d; }

int colsum(int act_bf16, const ColsumArgs& a, cudaStream_t s) {
  if (a.d <= 0) return 0;
  // 16-byte row segments per thread when the layout allows (V = 8 bf16 or 4 fp32
  // columns), else one column per thread; enough row chunks for ~3 CTAs per SM.
  const bool src_bf16 = a.src_act && act_bf16;
  const int vec = src_bf16 ? 8 : 4;
  const bool aligned = (a.d % vec) == 0 && (a.ld % vec) == 0 && (!a.src2 || vec == 4 || (a.d % 4) == 0) &&
                       (reinterpret_cast<uintptr_t>(a.src) & 15) == 0 &&
                       (!a.src2 || (reinterpret_cast<uintptr_t>(a.src2) & 15) == 0) &&
                       (!a.x || (reinterpret_cast<uintptr_t>(a.x) & 15) == 0) &&
                       (!a.bsrc || (reinterpret_cast<uintptr_t>(a.bsrc) & 15) == 0);
  const int V = aligned ? vec : 1;
  const int col_blocks = (a.d / V + CS_THREADS - 1) / CS_THREADS;
  int nch = aligned ? (3 * num_sms() + col_blocks - 1) / col_blocks : CS_CHUNKS;
  if (nch > kMaxColsumChunks) nch = kMaxColsumChunks;
  if (nch > a.rows) nch = a.rows > 0 ? a.rows : 1;
  dim3 grid(col_blocks, nch);
  if (aligned && a.bmode == 0 && !a.src2) {
    if (src_bf16) colsum_plain_kernel<bf16><<<grid, CS_THREADS, 0, s>>>(reinterpret_cast<const bf16*>(a.src), a.ld, a.d,
                                                                       a.rows, a.partial);
    else colsum_plain_kernel<float><<<grid, CS_THREADS, 0, s>>>(reinterpret_cast<const float*>(a.src), a.ld, a.d,
                                                               a.rows, a.partial);
  } else if (!aligned) {
    if (a.src_act && act_bf16) colsum_kernel<bf16, 1><<<grid, CS_THREADS, 0, s>>>(a);
    else colsum_kernel<float, 1><<<grid, CS_THREADS, 0, s>>>(a);
  } else if (src_bf16) {
    colsum_kernel<bf16, 8><<<grid, CS_THREADS, 0, s>>>(a);
  } else {
    colsum_kernel<float, 4><<<grid, CS_THREADS, 0, s>>>(a);
  }
  colsum_finish_kernel<2><<<(a.d + 31) / 32, CF_WARPS * 32, 0, s>>>(a.partial, nch, a.d, a.out1, a.out0, a.out0b,
                                                                     nullptr, nullptr, a.accumulate);
  count_launches(2);
  return last_err();
}

int embed_fwd(int rows, int T, int d, int V, const int32_t* tok, const float* wte, const float* wpe, float* X, int* err,
              cudaStream_t s) {
  if (rows <= 0) return 0;
  if (d % 4) return 1;
  embed_fwd_kernel<<<rows, 128, 0, s>>>(rows, T, d, V, tok, wte, wpe, X, err);
  count_launches(1);
  return last_err();
}

int embed_bwd(int B, int T, int d, int V, const int32_t* tok, const float* dX, float* dwte, float* dwpe,
              cudaStream_t s) {
  const int rows = B * T;
  if (rows <= 0) return 0;
  embed_bwd_pos_kernel<<<grid_for((long)T * d, 256), 256, 0, s>>>(B, T, d, dX, dwpe);
  embed_bwd_tok_kernel<<<rows, 256, 0, s>>>(rows, d, tok, dX, dwte, V);
  count_launches(2);
  return last_err();
}

int ce_combine(int rows, int nslices, const float2* stats, long ld, const float* tlogit, const int32_t* tgt, int V,
               float* lse, float* loss_rows, float* loss, int* err, cudaStream_t s) {
  if (rows <= 0) return 0;
  ce_combine_kernel<<<(rows + 127) / 128, 128, 0, s>>>(rows, nslices, stats, ld, tlogit, tgt, V, lse, loss_rows, err);
  mean_kernel<<<1, 1024, 0, s>>>(rows, loss_rows, loss);
  count_launches(2);
  return last_err();
}

int cross_entropy(int act_bf16, int rows, int V, long ld, const void* logits, const int32_t* tgt, void* dlogits,
                  float* loss_rows, float* loss, int* err, cudaStream_t s) {
  if (rows <= 0) return 0;
  if (act_bf16)
    ce_kernel<bf16><<<rows, 256, 0, s>>>(rows, V, ld, reinterpret_cast<const bf16*>(logits), tgt,
                                         reinterpret_cast<bf16*>(dlogits), loss_rows, err);
  else
    ce_kernel<float><<<rows, 256, 0, s>>>(rows, V, ld, reinterpret_cast<const float*>(logits), tgt,
                                          reinterpret_cast<float*>(dlogits), loss_rows, err);
  mean_kernel<<<1, 1024, 0, s>>>(rows, loss_rows, loss);
  count_launches(2);
  return last_err();
}

int add_scaled_cols(int rows, int d, const float* src, const float* colvec, float* dst, cudaStream_t s) {
  const long n = (long)rows * d;
  if (n <= 0) return 0;
  if (d % 4) return 1;
  add_scaled_cols_kernel<<<grid_for(n / 4, 256), 256, 0, s>>>(n, d, src, colvec, dst);
  count_launches(1);
  return last_err();
}

int adamw(size_t n, size_t n_decay, float* p, const float* g, float* m, float* v, void* shadow, float lr, float beta1,
          float beta2, float eps, float wd, float bc1, float bc2, cudaStream_t s, const float* gscale) {
  if (n == 0) return 0;
  if (n % 4) return 1;
  const int blocks = num_sms() * 8;
  adamw_kernel<<<blocks, 256, 0, s>>>(n, n_decay, p, g, m, v, reinterpret_cast<bf16*>(shadow), lr, beta1, beta2, eps, wd,
                                      1.f / bc1, 1.f / bc2, gscale);
  count_launches(1);
  return last_err();
}

int grad_norm_partials() { return 2 * GN_BLOCKS; }  // GN_BLOCKS doubles

int grad_norm_clip(size_t n, const float* g, float max_norm, float* partial, float* norm_out, float* scale_out,
                   cudaStream_t s) {
  if (n % 4) return 1;
  double* part = reinterpret_cast<double*>(partial);
  grad_sumsq_kernel<<<GN_BLOCKS, GN_THREADS, 0, s>>>(n / 4, g, part);
  grad_clip_finish_kernel<<<1, 32, 0, s>>>(GN_BLOCKS, part, max_norm, norm_out, scale_out);
  count_launches(2);
  return last_err();
}

int f32_to_bf16(size_t n, const float* src, void* dst, cudaStream_t s) {
  if (n == 0) return 0;
  f32_to_bf16_kernel<<<grid_for((long)n, 256), 256, 0, s>>>(n, src, reinterpret_cast<bf16*>(dst));
  count_launches(1);
  return last_err();
}

int act_to_f32_2d(int act_bf16, int rows, int cols, long ld, const void* src, float* dst, cudaStream_t s) {
  const long n = (long)rows * cols;
  if (n <= 0) return 0;
  if (act_bf16) act_to_f32_2d_kernel<bf16><<<grid_for(n, 256), 256, 0, s>>>(rows, cols, ld, reinterpret_cast<const bf16*>(src), dst);
  else act_to_f32_2d_kernel<float><<<grid_for(n, 256), 256, 0, s>>>(rows, cols, ld, reinterpret_cast<const float*>(src), dst);
  count_launches(1);
  return last_err();
}

int act_to_f32(int act_bf16, size_t n, const void* src, float* dst, cudaStream_t s) {
  return act_to_f32_2d(act_bf16, 1, (int)n, (long)n, src, dst, s);
}

}  // namespace fal
