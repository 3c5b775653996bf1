// Causal multi-head attention, forward and backward (the MHA_i of every block).
//
// bf16 path: the forward runs on tcgen05 (attention_tc.cu).  The backward here
// is flash-attention style (scores recomputed, never written to HBM) on
// warp-level bf16 MMA with fp32 accumulation: one CTA per (64-key block, head),
// 4 warps of 16 keys, query tiles of 64 streamed through shared memory with
// cp.async; dK/dV accumulate in registers, dQ in an fp32 scratch buffer with
// vector atomics.
// fp32 debug path: one thread per query row, plain fp32 arithmetic.
//
// Scores: S = Q K^T / sqrt(hd), key j visible to query t iff j <= t.  The
// saved log-sum-exp is in log2 units of S*log2(e).
#include "common.cuh"
#include "internal.h"

namespace fal {

namespace {

constexpr float LOG2E = 1.4426950408889634f;

// ------------------------------------------------------------ PTX helpers
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
  const int n = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(n) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3) : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3) : "r"(addr));
}
// D(16x8) += A(16x16, row) * B(16x8, col), bf16 inputs, fp32 accumulators.
__device__ __forceinline__ void mma_bf16(float* d, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Tile [64 rows][HD] bf16 in shared memory, 16-byte chunks XOR-swizzled by row
// so that ldmatrix row reads hit distinct banks.
template <int HD>
__device__ __forceinline__ uint32_t tile_off(int row, int col) {  // col multiple of 8
  return (uint32_t)((row * HD + (((col >> 3) ^ (row & 7)) << 3)) * 2);
}

// Loads rows [r0, r0+64) of one head's slice (column offset coff) of a
// row-major [B*T, ld] bf16 matrix for batch b; rows >= T are zero-filled.
template <int HD, int NT>
__device__ __forceinline__ void load_tile(uint32_t sbase, const bf16* g, long ld, int b, int T, int r0, int coff) {
  constexpr int CH = HD / 8;
  for (int i = threadIdx.x; i < 64 * CH; i += NT) {
    const int r = i / CH, c = (i % CH) * 8;
    const int t = r0 + r;
    const bool valid = t < T;
    const bf16* src = g + ((long)b * T + (valid ? t : 0)) * ld + coff + c;
    cp_async16(sbase + tile_off<HD>(r, c), src, valid);
  }
}

// ------------------------------------------------------------ backward (bf16)
// D[b,h,t] = sum_c dO[t,c] * O[t,c]; also clears the dQ accumulator.
__global__ void attn_bwd_pre_kernel(const bf16* __restrict__ ctx, const bf16* __restrict__ dctx,
                                    float* __restrict__ dvec, float* __restrict__ dq_acc, int T, int H, int hd) {
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
  float* dq = dq_acc + (long)bt * d + h * hd;
  for (int c = lane; c < hd; c += 32) dq[c] = 0.f;
  if (lane == 0) {
    const int b = bt / T, t = bt % T;
    dvec[((long)b * H + h) * T + t] = acc;
  }
}

__global__ void attn_bwd_post_kernel(const float* __restrict__ dq_acc, bf16* __restrict__ dqkv, long rows, int d) {
  const long n = rows * d / 4;
  for (long i = blockIdx.x * (long)blockDim.x + threadIdx.x; i < n; i += (long)gridDim.x * blockDim.x) {
    const long e = i * 4;
    const long r = e / d, c = e % d;
    store4(dqkv + r * 3L * d + c, load4(dq_acc + e));
  }
}

template <int HD>
__global__ void __launch_bounds__(128) attn_bwd_kernel(const bf16* __restrict__ qkv, const bf16* __restrict__ dctx,
                                                       const float* __restrict__ lse, const float* __restrict__ dvec,
                                                       float* __restrict__ dq_acc, bf16* __restrict__ dqkv, int T, int H,
                                                       float scale, float scale_log2) {
  extern __shared__ __align__(128) uint8_t smem[];
  const uint32_t sK = smem_addr(smem);
  const uint32_t sV = sK + 64 * HD * 2;
  const uint32_t sQ = sV + 64 * HD * 2;
  const uint32_t sdO = sQ + 64 * HD * 2;
  const uint32_t sdS = sdO + 64 * HD * 2;  // [64 q][64 keys] bf16
  bf16* dS_ptr = reinterpret_cast<bf16*>(smem + 4 * 64 * HD * 2);
  float* s_lse = reinterpret_cast<float*>(smem + 4 * 64 * HD * 2 + 64 * 64 * 2);
  float* s_d = s_lse + 64;

  const int nkb = (T + 63) / 64;
  const int kb = nkb - 1 - blockIdx.x;  // shortest work last... (longest first: kb small has most q blocks)
  const int kblk = blockIdx.x;          // process kv block index directly for load balance below
  (void)kb;
  const int bh = blockIdx.y, b = bh / H, h = bh % H;
  const int d = H * HD;
  const long ld = 3L * d;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int g = lane / 4, t4 = lane % 4;
  const int key0 = kblk * 64;

  load_tile<HD, 128>(sK, qkv, ld, b, T, key0, d + h * HD);
  load_tile<HD, 128>(sV, qkv, ld, b, T, key0, 2 * d + h * HD);
  cp_async_commit();

  float dk[HD / 8][4], dv[HD / 8][4];
#pragma unroll
  for (int i = 0; i < HD / 8; ++i)
#pragma unroll
    for (int e = 0; e < 4; ++e) dk[i][e] = dv[i][e] = 0.f;

  const int nqb = (T + 63) / 64;
  for (int qb = kblk; qb < nqb; ++qb) {
    const int q0 = qb * 64;
    load_tile<HD, 128>(sQ, qkv, ld, b, T, q0, h * HD);
    load_tile<HD, 128>(sdO, dctx, d, b, T, q0, h * HD);
    cp_async_commit();
    if (threadIdx.x < 64) {
      const int t = q0 + threadIdx.x;
      s_lse[threadIdx.x] = (t < T) ? lse[(long)bh * T + t] : 0.f;
      s_d[threadIdx.x] = (t < T) ? dvec[(long)bh * T + t] : 0.f;
    }
    cp_async_wait<0>();
    __syncthreads();

    // S^T (16 keys of this warp x 64 queries) = K_w Q^T
    float st[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) st[i][0] = st[i][1] = st[i][2] = st[i][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
      uint32_t a[4];
      {
        const int r = warp * 16 + (lane % 8) + 8 * ((lane / 8) % 2);
        const int c = kk * 16 + 8 * (lane / 16);
        ldsm_x4(sK + tile_off<HD>(r, c), a[0], a[1], a[2], a[3]);
      }
#pragma unroll
      for (int nb = 0; nb < 8; nb += 2) {
        uint32_t b0, b1, b2, b3;
        const int r = nb * 8 + (lane % 8) + 8 * (lane / 16);
        const int c = kk * 16 + 8 * ((lane / 8) % 2);
        ldsm_x4(sQ + tile_off<HD>(r, c), b0, b1, b2, b3);
        mma_bf16(st[nb], a, b0, b1);
        mma_bf16(st[nb + 1], a, b2, b3);
      }
    }
    // P^T = exp2(S^T * scale_log2 - lse[q]) with causal mask (q >= key)
#pragma unroll
    for (int nb = 0; nb < 8; ++nb) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = key0 + warp * 16 + g + (e >> 1) * 8;
        const int ql = nb * 8 + 2 * t4 + (e & 1);
        const int q = q0 + ql;
        float pv = exp2f(st[nb][e] * scale_log2 - s_lse[ql]);
        if (q < key || q >= T || key >= T) pv = 0.f;
        st[nb][e] = pv;
      }
    }
    // dV_w += P^T dO
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      uint32_t a[4];
      a[0] = pack_bf16(st[2 * kk][0], st[2 * kk][1]);
      a[1] = pack_bf16(st[2 * kk][2], st[2 * kk][3]);
      a[2] = pack_bf16(st[2 * kk + 1][0], st[2 * kk + 1][1]);
      a[3] = pack_bf16(st[2 * kk + 1][2], st[2 * kk + 1][3]);
#pragma unroll
      for (int nd = 0; nd < HD / 8; nd += 2) {
        uint32_t b0, b1, b2, b3;
        const int r = kk * 16 + (lane % 8) + 8 * ((lane / 8) % 2);
        const int c = nd * 8 + 8 * (lane / 16);
        ldsm_x4_t(sdO + tile_off<HD>(r, c), b0, b1, b2, b3);
        mma_bf16(dv[nd], a, b0, b1);
        mma_bf16(dv[nd + 1], a, b2, b3);
      }
    }
    // dP^T = V_w dO^T
    float dpt[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) dpt[i][0] = dpt[i][1] = dpt[i][2] = dpt[i][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
      uint32_t a[4];
      {
        const int r = warp * 16 + (lane % 8) + 8 * ((lane / 8) % 2);
        const int c = kk * 16 + 8 * (lane / 16);
        ldsm_x4(sV + tile_off<HD>(r, c), a[0], a[1], a[2], a[3]);
      }
#pragma unroll
      for (int nb = 0; nb < 8; nb += 2) {
        uint32_t b0, b1, b2, b3;
        const int r = nb * 8 + (lane % 8) + 8 * (lane / 16);
        const int c = kk * 16 + 8 * ((lane / 8) % 2);
        ldsm_x4(sdO + tile_off<HD>(r, c), b0, b1, b2, b3);
        mma_bf16(dpt[nb], a, b0, b1);
        mma_bf16(dpt[nb + 1], a, b2, b3);
      }
    }
    // dS^T = P^T * (dP^T - D[q]); stash dS (q-major) in shared memory for dQ
#pragma unroll
    for (int nb = 0; nb < 8; ++nb) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int ql = nb * 8 + 2 * t4 + (e & 1);
        const float ds = st[nb][e] * (dpt[nb][e] - s_d[ql]);
        dpt[nb][e] = ds;
        const int kl = warp * 16 + g + (e >> 1) * 8;
        // element (row ql, col kl) of the [64][64] q-major tile, same swizzle as tile_off<64>
        const uint32_t off = tile_off<64>(ql, kl & ~7) / 2 + (kl & 7);
        dS_ptr[off] = __float2bfloat16_rn(ds);
      }
    }
    // dK_w += dS^T Q
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      uint32_t a[4];
      a[0] = pack_bf16(dpt[2 * kk][0], dpt[2 * kk][1]);
      a[1] = pack_bf16(dpt[2 * kk][2], dpt[2 * kk][3]);
      a[2] = pack_bf16(dpt[2 * kk + 1][0], dpt[2 * kk + 1][1]);
      a[3] = pack_bf16(dpt[2 * kk + 1][2], dpt[2 * kk + 1][3]);
#pragma unroll
      for (int nd = 0; nd < HD / 8; nd += 2) {
        uint32_t b0, b1, b2, b3;
        const int r = kk * 16 + (lane % 8) + 8 * ((lane / 8) % 2);
        const int c = nd * 8 + 8 * (lane / 16);
        ldsm_x4_t(sQ + tile_off<HD>(r, c), b0, b1, b2, b3);
        mma_bf16(dk[nd], a, b0, b1);
        mma_bf16(dk[nd + 1], a, b2, b3);
      }
    }
    __syncthreads();
    // dQ (rows 16*warp.. of this q block) += dS K, accumulated in fp32 scratch
    {
      float dq[HD / 8][4];
#pragma unroll
      for (int i = 0; i < HD / 8; ++i) dq[i][0] = dq[i][1] = dq[i][2] = dq[i][3] = 0.f;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        uint32_t a[4];
        const int r = warp * 16 + (lane % 8) + 8 * ((lane / 8) % 2);
        const int c = kk * 16 + 8 * (lane / 16);
        ldsm_x4(sdS + tile_off<64>(r, c), a[0], a[1], a[2], a[3]);
#pragma unroll
        for (int nd = 0; nd < HD / 8; nd += 2) {
          uint32_t b0, b1, b2, b3;
          const int rr = kk * 16 + (lane % 8) + 8 * ((lane / 8) % 2);
          const int cc = nd * 8 + 8 * (lane / 16);
          ldsm_x4_t(sK + tile_off<HD>(rr, cc), b0, b1, b2, b3);
          mma_bf16(dq[nd], a, b0, b1);
          mma_bf16(dq[nd + 1], a, b2, b3);
        }
      }
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const int q = q0 + warp * 16 + g + r * 8;
        if (q >= T) continue;
        float* dst = dq_acc + ((long)b * T + q) * d + h * HD;
#pragma unroll
        for (int nd = 0; nd < HD / 8; ++nd) {
          atomicAdd(reinterpret_cast<float2*>(dst + nd * 8 + 2 * t4),
                    make_float2(dq[nd][2 * r] * scale, dq[nd][2 * r + 1] * scale));
        }
      }
    }
    __syncthreads();
  }
  // write dK (scaled) and dV for this warp's 16 keys
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int key = key0 + warp * 16 + g + r * 8;
    if (key >= T) continue;
    bf16* dkp = dqkv + ((long)b * T + key) * ld + d + h * HD;
    bf16* dvp = dqkv + ((long)b * T + key) * ld + 2 * d + h * HD;
#pragma unroll
    for (int nd = 0; nd < HD / 8; ++nd) {
      *reinterpret_cast<uint32_t*>(dkp + nd * 8 + 2 * t4) = pack_bf16(dk[nd][2 * r] * scale, dk[nd][2 * r + 1] * scale);
      *reinterpret_cast<uint32_t*>(dvp + nd * 8 + 2 * t4) = pack_bf16(dv[nd][2 * r], dv[nd][2 * r + 1]);
    }
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

template <int HD>
int launch_bwd(int B, int T, int H, const void* qkv, const void* dctx, const float* lse, const float* dvec,
               float* dq_acc, void* dqkv, cudaStream_t s) {
  const int smem = 4 * 64 * HD * 2 + 64 * 64 * 2 + 2 * 64 * 4;
  static bool set = false;
  if (!set) {
    cudaFuncSetAttribute(attn_bwd_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    set = true;
  }
  dim3 grid((T + 63) / 64, B * H);
  attn_bwd_kernel<HD><<<grid, 128, smem, s>>>(reinterpret_cast<const bf16*>(qkv), reinterpret_cast<const bf16*>(dctx),
                                             lse, dvec, dq_acc, reinterpret_cast<bf16*>(dqkv), T, H,
                                             1.f / sqrtf((float)HD), LOG2E / sqrtf((float)HD));
  return 0;
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
             const void* dctx, void* dqkv, float* dq_acc, float* dvec, cudaStream_t s, std::string* msg) {
  if (B <= 0 || T <= 0) return 0;
  const long rows = (long)B * T;
  const int d = H * hd;
  if (act_bf16) {
    if (hd != 64 && hd != 128) { if (msg) *msg = "bf16 attention needs head_dim 64 or 128"; return 6; }
    const int wpb = 4;
    dim3 pg((H + wpb - 1) / wpb, (unsigned)rows);
    attn_bwd_pre_kernel<<<pg, wpb * 32, 0, s>>>(reinterpret_cast<const bf16*>(ctx), reinterpret_cast<const bf16*>(dctx),
                                               dvec, dq_acc, T, H, hd);
    if (hd == 64) launch_bwd<64>(B, T, H, qkv, dctx, lse, dvec, dq_acc, dqkv, s);
    else launch_bwd<128>(B, T, H, qkv, dctx, lse, dvec, dq_acc, dqkv, s);
    const long n4 = rows * d / 4;
    const int blocks = (int)((n4 + 255) / 256 < 4096 ? (n4 + 255) / 256 : 4096);
    attn_bwd_post_kernel<<<blocks, 256, 0, s>>>(dq_acc, reinterpret_cast<bf16*>(dqkv), rows, d);
    count_launches(3);
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
  const size_t dq_floats = (size_t)B * T * H * hd;
  const size_t need = dq_floats + (size_t)B * H * T;
  if (need > kNoAllocFloats) return FAL_ERR_WORKSPACE;
  float* scratch = nullptr;
  const int rc = noalloc_scratch(&scratch);
  if (rc != FAL_OK) return rc;
  std::string msg;
  // attn_bwd's first kernel zeroes the dQ accumulator and writes every D entry,
  // so nothing left in the shared array by an earlier call leaks into this one.
  const int r = fal::attn_bwd(1, B, T, H, hd, qkv, ctx, lse, dctx, dqkv, scratch, scratch + dq_floats,
                              reinterpret_cast<cudaStream_t>(stream), &msg);
  return r == 0 ? FAL_OK : r == 1 ? FAL_ERR_ARG : r == 6 ? FAL_ERR_UNSUPPORTED : FAL_ERR_CUDA;
}
