// Causal multi-head attention, forward and backward (the MHA_i of every block).
//
// bf16 path: the tcgen05 kernels live in attention_tc.cu; this file holds the
// backward's pre-pass (D = rowsum(dO * O), zeroed dQ accumulator) and post-pass
// (dQ accumulator -> bf16), the fp32 debug kernels (one thread per query row,
// plain fp32 arithmetic) and the allocation-free backward entry point.
//
// Scores: S = Q K^T / sqrt(hd), key j visible to query t iff j <= t.  The
// saved log-sum-exp is in log2 units of S*log2(e).
#include "common.cuh"
#include "internal.h"

namespace fal {

namespace {

constexpr float LOG2E = 1.4426950408889634f;

// ------------------------------------------------------------ backward (bf16)
// D[b,h,t] = sum_c dO[t,c] * O[t,c].
__global__ void attn_bwd_pre_kernel(const bf16* __restrict__ ctx, const bf16* __restrict__ dctx,
                                    float* __restrict__ dvec, int T, int H, int hd) {
  const int warps = blockDim.x / 32;
  const int w = blockIdx.x * warps + threadIdx.x / 32, lane = threadIdx.x % 32;
  const int d = H * hd;
  const long rows = (long)gridDim.y;  // unused guard
  (void)rows;
  const int bt = blockIdx.y;           // token row
  if (w >= H) return;
  const int h = w;
  const bf16* o = ctx + (long)bt * d + h * hd;
  const bf16* g = dctx + (long)bt * d + h * hd;
  float acc = 0.f;
  for (int c = lane; c < hd; c += 32) acc += __bfloat162float(o[c]) * __bfloat162float(g[c]);
  acc = warp_sum(acc);
  if (lane == 0) {
    const int b = bt / T, t = bt % T;
    dvec[((long)b * H + h) * T + t] = acc;
  }
}

// ------------------------------------------------------------ fp32 debug path
__global__ void attn_fwd_naive(const float* __restrict__ qkv, float* __restrict__ ctx, float* __restrict__ lse, int B,
                               int T, int H, int hd, float scale) {
  const long idx = blockIdx.x * (long)blockDim.x + threadIdx.x;
  if (idx >= (long)B * H * T) return;
  const int t = idx % T, h = (idx / T) % H, b = idx / ((long)T * H);
  const int d = H * hd;
  const long ld = 3L * d;
  const float* q = qkv + ((long)b * T + t) * ld + h * hd;
  float o[128];
  for (int c = 0; c < hd; ++c) o[c] = 0.f;
  float m = -INFINITY, l = 0.f;
  for (int j = 0; j <= t; ++j) {
    const float* k = qkv + ((long)b * T + j) * ld + d + h * hd;
    const float* v = qkv + ((long)b * T + j) * ld + 2 * d + h * hd;
    float s = 0.f;
    for (int c = 0; c < hd; ++c) s = fmaf(q[c], k[c], s);
    s *= scale;
    const float mn = fmaxf(m, s);
    const float corr = (m == -INFINITY) ? 0.f : expf(m - mn);
    const float p = expf(s - mn);
    l = l * corr + p;
    for (int c = 0; c < hd; ++c) o[c] = o[c] * corr + p * v[c];
    m = mn;
  }
  float* out = ctx + ((long)b * T + t) * d + h * hd;
  for (int c = 0; c < hd; ++c) out[c] = o[c] / l;
  lse[((long)b * H + h) * T + t] = (m + logf(l)) * LOG2E;
}

// Per query row: dq directly; dk, dv by fp32 atomics into dqkv (zeroed first).
__global__ void attn_bwd_naive(const float* __restrict__ qkv, const float* __restrict__ ctx,
                               const float* __restrict__ lse, const float* __restrict__ dctx, float* __restrict__ dqkv,
                               int B, int T, int H, int hd, float scale) {
  const long idx = blockIdx.x * (long)blockDim.x + threadIdx.x;
  if (idx >= (long)B * H * T) return;
  const int t = idx % T, h = (idx / T) % H, b = idx / ((long)T * H);
  const int d = H * hd;
  const long ld = 3L * d;
  const float* q = qkv + ((long)b * T + t) * ld + h * hd;
  const float* o = ctx + ((long)b * T + t) * d + h * hd;
  const float* go = dctx + ((long)b * T + t) * d + h * hd;
  const float L = lse[((long)b * H + h) * T + t] / LOG2E;
  float D = 0.f;
  for (int c = 0; c < hd; ++c) D = fmaf(go[c], o[c], D);
  float dq[128];
  for (int c = 0; c < hd; ++c) dq[c] = 0.f;
  for (int j = 0; j <= t; ++j) {
    const float* k = qkv + ((long)b * T + j) * ld + d + h * hd;
    const float* v = qkv + ((long)b * T + j) * ld + 2 * d + h * hd;
    float s = 0.f, dp = 0.f;
    for (int c = 0; c < hd; ++c) { s = fmaf(q[c], k[c], s); dp = fmaf(go[c], v[c], dp); }
    const float p = expf(s * scale - L);
    const float ds = p * (dp - D);
    float* dk = dqkv + ((long)b * T + j) * ld + d + h * hd;
    float* dv = dqkv + ((long)b * T + j) * ld + 2 * d + h * hd;
    for (int c = 0; c < hd; ++c) {
      dq[c] = fmaf(ds, k[c], dq[c]);
      atomicAdd(dk + c, ds * q[c] * scale);
      atomicAdd(dv + c, p * go[c]);
    }
  }
  float* dqp = dqkv + ((long)b * T + t) * ld + h * hd;
  for (int c = 0; c < hd; ++c) dqp[c] = dq[c] * scale;
}

__global__ void zero_kv_grad(float* dqkv, long rows, int d) {
  const long n = rows * 2L * d;
  for (long i = blockIdx.x * (long)blockDim.x + threadIdx.x; i < n; i += (long)gridDim.x * blockDim.x) {
    const long r = i / (2L * d), c = i % (2L * d);
    dqkv[r * 3L * d + d + c] = 0.f;
  }
}

int check_launch(const char* what, std::string* msg) {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    if (msg) *msg = std::string(what) + ": " + cudaGetErrorString(e);
    return 4;
  }
  return 0;
}

}  // namespace

int attn_fwd(int act_bf16, int B, int T, int H, int hd, const void* qkv, void* ctx, float* lse, int* dev_err,
             cudaStream_t s, std::string* msg) {
  if (B <= 0 || T <= 0) return 0;
  if (act_bf16) {
    return attn_fwd_tc(B, T, H, hd, qkv, ctx, lse, dev_err, s, msg);
  } else {
    if (hd > 128) { if (msg) *msg = "fp32 attention needs head_dim <= 128"; return 6; }
    const long n = (long)B * H * T;
    attn_fwd_naive<<<(unsigned)((n + 127) / 128), 128, 0, s>>>(reinterpret_cast<const float*>(qkv),
                                                               reinterpret_cast<float*>(ctx), lse, B, T, H, hd,
                                                               1.f / sqrtf((float)hd));
  }
  count_launches(1);
  return check_launch("attention forward", msg);
}

int attn_bwd(int act_bf16, int B, int T, int H, int hd, const void* qkv, const void* ctx, const float* lse,
             const void* dctx, void* dqkv, float* dvec, int* dev_err, cudaStream_t s, std::string* msg,
             int d_ready) {
  if (B <= 0 || T <= 0) return 0;
  const long rows = (long)B * T;
  const int d = H * hd;
  if (act_bf16) {
    if (hd != 64 && hd != 128) { if (msg) *msg = "bf16 attention needs head_dim 64 or 128"; return 6; }
    const int wpb = 4;
    dim3 pg((H + wpb - 1) / wpb, (unsigned)rows);
    if (!d_ready) {
      attn_bwd_pre_kernel<<<pg, wpb * 32, 0, s>>>(reinterpret_cast<const bf16*>(ctx),
                                                 reinterpret_cast<const bf16*>(dctx), dvec, T, H, hd);
      count_launches(1);
    }
    const int r = attn_bwd2_tc(B, T, H, hd, qkv, dctx, lse, dvec, dqkv, dev_err, s, msg);
    if (r) return r;
    (void)d;
  } else {
    if (hd > 128) { if (msg) *msg = "fp32 attention needs head_dim <= 128"; return 6; }
    zero_kv_grad<<<256, 256, 0, s>>>(reinterpret_cast<float*>(dqkv), rows, d);
    const long n = (long)B * H * T;
    attn_bwd_naive<<<(unsigned)((n + 127) / 128), 128, 0, s>>>(
        reinterpret_cast<const float*>(qkv), reinterpret_cast<const float*>(ctx), lse,
        reinterpret_cast<const float*>(dctx), reinterpret_cast<float*>(dqkv), B, T, H, hd, 1.f / sqrtf((float)hd));
    count_launches(2);
  }
  return check_launch("attention backward", msg);
}

}  // namespace fal

// ------------------------------------------------------------ allocation-free entry point
// Scratch for fal_kernel_attention_bwd_noalloc: a fixed file-scope device array
// (dQ accumulator followed by the D = rowsum(dO * O) vector).  Host code only
// ever sees a stand-in for this symbol, so its device address is looked up
// once per device with cudaGetSymbolAddress while that device is current.
#include <mutex>

#include "../../include/fal.h"
#include "../../include/fal_kernels.h"

namespace {

constexpr size_t kNoAllocFloats = FAL_NOALLOC_ATTN_SCRATCH_FLOATS;
static __device__ __align__(256) float g_noalloc_attn_scratch[kNoAllocFloats];

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
float* g_noalloc_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device (looked up once).
int noalloc_scratch(float** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return FAL_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return FAL_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_attn_scratch) != cudaSuccess || !p) return FAL_ERR_CUDA;
    g_noalloc_ptr[dev] = static_cast<float*>(p);
  }
  *out = g_noalloc_ptr[dev];
  return FAL_OK;
}

}  // namespace

extern "C" int fal_kernel_attention_bwd_noalloc(int B, int T, int H, int hd, const void* qkv, const void* ctx,
                                                const float* lse, const void* dctx, void* dqkv, void* stream) {
  if (B < 0 || T < 0 || H <= 0 || hd <= 0 || !qkv || !ctx || !lse || !dctx || !dqkv) return FAL_ERR_ARG;
  const size_t need = (size_t)B * H * T;
  if (need > kNoAllocFloats) return FAL_ERR_WORKSPACE;
  float* scratch = nullptr;
  const int rc = noalloc_scratch(&scratch);
  if (rc != FAL_OK) return rc;
  std::string msg;
  // attn_bwd's first kernel writes every D entry before it is read, so nothing
  // left in the shared array by an earlier call leaks into this one.
  const int r = fal::attn_bwd(1, B, T, H, hd, qkv, ctx, lse, dctx, dqkv, scratch, nullptr,
                              reinterpret_cast<cudaStream_t>(stream), &msg);
  return r == 0 ? FAL_OK : r == 1 ? FAL_ERR_ARG : r == 6 ? FAL_ERR_UNSUPPORTED : FAL_ERR_CUDA;
}
