// Causal multi-head attention, forward and backward (the MHA_i of every block).
//
// bf16 path: the tcgen05 kernels live in attention_tc.cu (forward) and
// attention_bwd_tc.cu (backward); this file holds the backward's pre-pass
// D = rowsum(dO * O) for the kernel-level entry points (the model takes D from
// the epilogue of the GEMM that produces dO), the fp32 debug kernels (one thread
// per query row, plain fp32 arithmetic) and the allocation-free backward entry
// point.
//
// Scores: S = Q K^T / sqrt(hd), key j visible to query t iff j <= t.  The
// saved log-sum-exp is in log2 units of S*log2(e).
#include "common.cuh"
#include "internal.h"

namespace fal {

namespace {

constexpr float LOG2E = 1.4426950408889634f;

// ------------------------------------------------------------ backward (bf16)
// D[b,h,t] = sum_c dO[t,c] * O[t,c]: one warp per (token row, head), in a
// grid-stride loop over all B*T*H of them (any B*T, no grid-dimension limit).
__global__ void attn_bwd_pre_kernel(const bf16* __restrict__ ctx, const bf16* __restrict__ dctx,
                                    float* __restrict__ dvec, long rows, int T, int H, int hd) {
  const int lane = threadIdx.x % 32;
  const long nwarps = (long)gridDim.x * (blockDim.x / 32);
  const long d = (long)H * hd;
  for (long w = blockIdx.x * (long)(blockDim.x / 32) + threadIdx.x / 32; w < rows * H; w += nwarps) {
    const long bt = w / H;
    const int h = (int)(w - bt * H);
    const bf16* o = ctx + bt * d + (long)h * hd;
    const bf16* g = dctx + bt * d + (long)h * hd;
    float acc = 0.f;
    for (int c = lane; c < hd; c += 32) acc += __bfloat162float(o[c]) * __bfloat162float(g[c]);
    acc = warp_sum(acc);
    if (lane == 0) {
      const long b = bt / T, t = bt % T;
      dvec[(b * H + h) * T + t] = acc;
    }
  }
}

// ------------------------------------------------------------ fp32 debug path
// Head h reads the key / value head g = h / (H / Hkv) (grouped-query attention).
__global__ void attn_fwd_naive(const float* __restrict__ qkv, float* __restrict__ ctx, float* __restrict__ lse, int B,
                               int T, int H, int Hkv, int hd, float scale) {
  const long idx = blockIdx.x * (long)blockDim.x + threadIdx.x;
  if (idx >= (long)B * H * T) return;
  const int t = idx % T, h = (idx / T) % H, b = idx / ((long)T * H);
  const int d = H * hd, g = h / (H / Hkv);
  const long ld = (long)(H + 2 * Hkv) * hd;
  const int kc = d + g * hd, vc = d + (Hkv + g) * hd;
  const float* q = qkv + ((long)b * T + t) * ld + h * hd;
  float o[128];
  for (int c = 0; c < hd; ++c) o[c] = 0.f;
  float m = -INFINITY, l = 0.f;
  for (int j = 0; j <= t; ++j) {
    const float* k = qkv + ((long)b * T + j) * ld + kc;
    const float* v = qkv + ((long)b * T + j) * ld + vc;
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

// Per query row: dq directly; dk, dv by fp32 atomics into dqkv (zeroed first),
// which also sums them over the query heads of a key / value head's group.
__global__ void attn_bwd_naive(const float* __restrict__ qkv, const float* __restrict__ ctx,
                               const float* __restrict__ lse, const float* __restrict__ dctx, float* __restrict__ dqkv,
                               int B, int T, int H, int Hkv, int hd, float scale) {
  const long idx = blockIdx.x * (long)blockDim.x + threadIdx.x;
  if (idx >= (long)B * H * T) return;
  const int t = idx % T, h = (idx / T) % H, b = idx / ((long)T * H);
  const int d = H * hd, g = h / (H / Hkv);
  const long ld = (long)(H + 2 * Hkv) * hd;
  const int kc = d + g * hd, vc = d + (Hkv + g) * hd;
  const float* q = qkv + ((long)b * T + t) * ld + h * hd;
  const float* o = ctx + ((long)b * T + t) * d + h * hd;
  const float* go = dctx + ((long)b * T + t) * d + h * hd;
  const float L = lse[((long)b * H + h) * T + t] / LOG2E;
  float D = 0.f;
  for (int c = 0; c < hd; ++c) D = fmaf(go[c], o[c], D);
  float dq[128];
  for (int c = 0; c < hd; ++c) dq[c] = 0.f;
  for (int j = 0; j <= t; ++j) {
    const float* k = qkv + ((long)b * T + j) * ld + kc;
    const float* v = qkv + ((long)b * T + j) * ld + vc;
    float s = 0.f, dp = 0.f;
    for (int c = 0; c < hd; ++c) { s = fmaf(q[c], k[c], s); dp = fmaf(go[c], v[c], dp); }
    const float p = expf(s * scale - L);
    const float ds = p * (dp - D);
    float* dk = dqkv + ((long)b * T + j) * ld + kc;
    float* dv = dqkv + ((long)b * T + j) * ld + vc;
    for (int c = 0; c < hd; ++c) {
      dq[c] = fmaf(ds, k[c], dq[c]);
      atomicAdd(dk + c, ds * q[c] * scale);
      atomicAdd(dv + c, p * go[c]);
    }
  }
  float* dqp = dqkv + ((long)b * T + t) * ld + h * hd;
  for (int c = 0; c < hd; ++c) dqp[c] = dq[c] * scale;
}

// Zeroes the key / value columns [d, d + dkv) of rows of width d + dkv.
__global__ void zero_kv_grad(float* dqkv, long rows, int d, int dkv) {
  const long n = rows * dkv;
  for (long i = blockIdx.x * (long)blockDim.x + threadIdx.x; i < n; i += (long)gridDim.x * blockDim.x) {
    const long r = i / dkv, c = i % dkv;
    dqkv[r * (long)(d + dkv) + d + c] = 0.f;
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
             cudaStream_t s, std::string* msg, int Hkv) {
  if (B <= 0 || T <= 0) return 0;
  if (Hkv <= 0) Hkv = H;
  if (H % Hkv) { if (msg) *msg = "heads must be a multiple of the key/value heads"; return 1; }
  if (act_bf16) {
    return attn_fwd_tc(B, T, H, Hkv, hd, qkv, ctx, lse, dev_err, s, msg);
  } else {
    if (hd > 128) { if (msg) *msg = "fp32 attention needs head_dim <= 128"; return 6; }
    const long n = (long)B * H * T;
    attn_fwd_naive<<<(unsigned)((n + 127) / 128), 128, 0, s>>>(reinterpret_cast<const float*>(qkv),
                                                               reinterpret_cast<float*>(ctx), lse, B, T, H, Hkv, hd,
                                                               1.f / sqrtf((float)hd));
  }
  count_launches(1);
  return check_launch("attention forward", msg);
}

int attn_bwd(int act_bf16, int B, int T, int H, int hd, const void* qkv, const void* ctx, const float* lse,
             const void* dctx, void* dqkv, float* dvec, int* dev_err, cudaStream_t s, std::string* msg,
             int d_ready, int Hkv) {
  if (B <= 0 || T <= 0) return 0;
  if (Hkv <= 0) Hkv = H;
  if (H % Hkv) { if (msg) *msg = "heads must be a multiple of the key/value heads"; return 1; }
  const long rows = (long)B * T;
  const int d = H * hd;
  if (act_bf16) {
    if (hd != 64 && hd != 128) { if (msg) *msg = "bf16 attention needs head_dim 64 or 128"; return 6; }
    if (!d_ready) {
      const int wpb = 8;
      const long warps = rows * H;
      const long want = (warps + wpb - 1) / wpb, cap = 16L * num_sms();
      attn_bwd_pre_kernel<<<(unsigned)(want < cap ? want : cap), wpb * 32, 0, s>>>(
          reinterpret_cast<const bf16*>(ctx), reinterpret_cast<const bf16*>(dctx), dvec, rows, T, H, hd);
      count_launches(1);
    }
    int* counter = reinterpret_cast<int*>(dvec + (rows * H + 63) / 64 * 64);
    const int r = attn_bwd_tc(B, T, H, Hkv, hd, qkv, dctx, lse, dvec, counter, dqkv, dev_err, s, msg);
    if (r) return r;
    (void)d;
  } else {
    if (hd > 128) { if (msg) *msg = "fp32 attention needs head_dim <= 128"; return 6; }
    zero_kv_grad<<<256, 256, 0, s>>>(reinterpret_cast<float*>(dqkv), rows, d, 2 * Hkv * hd);
    const long n = (long)B * H * T;
    attn_bwd_naive<<<(unsigned)((n + 127) / 128), 128, 0, s>>>(
        reinterpret_cast<const float*>(qkv), reinterpret_cast<const float*>(ctx), lse,
        reinterpret_cast<const float*>(dctx), reinterpret_cast<float*>(dqkv), B, T, H, Hkv, hd,
        1.f / sqrtf((float)hd));
    count_launches(2);
  }
  return check_launch("attention backward", msg);
}

}  // namespace fal

// ------------------------------------------------------------ allocation-free entry point
// Scratch for fal_kernel_attention_bwd_noalloc: a fixed file-scope device array
// that receives the D = rowsum(dO * O) vector, [B, H, T] fp32, followed by the
// backward kernel's work counter.  Host code only
// ever sees a stand-in for this symbol, so its device address is looked up
// with cudaGetSymbolAddress while the caller's device is current.
#include <cuda.h>
#include <mutex>

#include "../../include/fal.h"
#include "../../include/fal_kernels.h"

namespace {

constexpr size_t kNoAllocFloats = FAL_NOALLOC_ATTN_SCRATCH_FLOATS;
static __device__ __align__(256) float g_noalloc_attn_scratch[kNoAllocFloats];

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
// Address of the array per device, and the CUDA context it was looked up in:
// after a device reset (or under another context) the module is loaded anew
// and the array may sit elsewhere.
float* g_noalloc_ptr[kMaxDevices] = {};
CUcontext g_noalloc_ctx[kMaxDevices] = {};

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
CtxGetCurrentFn ctx_get_current() {
  static CtxGetCurrentFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<CtxGetCurrentFn>(p);
  });
  return fn;
}

// Device address of the scratch array in the current context.  Outside stream
// capture the address is looked up on every call (cheap once the module is
// loaded), so a cached value never outlives a device reset; while `s` is being
// captured no runtime lookup is made and the address cached for this device
// and context by an earlier call is used.
int noalloc_scratch(cudaStream_t s, float** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return FAL_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return FAL_ERR_UNSUPPORTED;
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &cap) != cudaSuccess) return FAL_ERR_CUDA;
  // The runtime makes the device's primary context current on first use; the
  // call above has done that, so the driver now reports the context in use.
  CUcontext ctx = nullptr;
  CtxGetCurrentFn get = ctx_get_current();
  if (!get || get(&ctx) != CUDA_SUCCESS) return FAL_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (cap != cudaStreamCaptureStatusNone) {
    if (!g_noalloc_ptr[dev] || g_noalloc_ctx[dev] != ctx) return FAL_ERR_STATE;
    *out = g_noalloc_ptr[dev];
    return FAL_OK;
  }
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_noalloc_attn_scratch) != cudaSuccess || !p) return FAL_ERR_CUDA;
  g_noalloc_ptr[dev] = static_cast<float*>(p);
  g_noalloc_ctx[dev] = ctx;
  *out = g_noalloc_ptr[dev];
  return FAL_OK;
}

}  // namespace

extern "C" int fal_kernel_attention_bwd_noalloc(int B, int T, int H, int hd, const void* qkv, const void* ctx,
                                                const float* lse, const void* dctx, void* dqkv, void* stream) {
  if (B < 0 || T < 0 || H <= 0 || hd <= 0 || !qkv || !ctx || !lse || !dctx || !dqkv) return FAL_ERR_ARG;
  const size_t need = fal::attn_bwd_scratch_floats(B, T, H);
  if (need > kNoAllocFloats) return FAL_ERR_WORKSPACE;
  float* scratch = nullptr;
  const int rc = noalloc_scratch(reinterpret_cast<cudaStream_t>(stream), &scratch);
  if (rc != FAL_OK) return rc;
  std::string msg;
  // attn_bwd's first kernel writes every D entry before it is read, and the
  // work counter behind D is cleared before the backward kernel starts, so
  // nothing left in the shared array by an earlier call leaks into this one.
  const int r = fal::attn_bwd(1, B, T, H, hd, qkv, ctx, lse, dctx, dqkv, scratch, nullptr,
                              reinterpret_cast<cudaStream_t>(stream), &msg);
  return r == 0 ? FAL_OK : r == 1 ? FAL_ERR_ARG : r == 6 ? FAL_ERR_UNSUPPORTED : FAL_ERR_CUDA;
}
