// Causal multi-head attention forward on tcgen05 (bf16 operands, fp32
// accumulation in TMEM): ctx = softmax(Q K^T / sqrt(hd) + causal) V for one
// (batch, head, 128-query tile) per CTA.
//
//   warp 0      TMA producer: the Q tile once, then K and V tiles of 128 keys
//               (two stages each) straight out of the packed qkv rows.
//   warp 1      MMA issuer: S_j = Q K_j^T into one of two TMEM score buffers
//               (128 x 128 fp32), then O += P_j V_j into the TMEM output
//               accumulator (128 x hd fp32).  S_{j+1} is issued before O += P_j
//               V_j so that the scores of the next tile are ready when the
//               softmax finishes the current one.
//   warps 2..5  softmax, one thread per query row: reads its score row from
//               TMEM, scales and masks it, keeps a running maximum m and sum l,
//               writes P = 2^(s - m) in bf16 into a swizzled shared-memory tile
//               (the A operand of the PV MMA).  The maximum used for the
//               exponent is only raised when the row maximum grows by more than
//               2^8 (P then stays below 256); only then is the row of O in TMEM
//               rescaled.  Finally O / l is stored in bf16 and the log-sum-exp
//               m + log2(l) (log2 units of S*log2(e)) is saved for the backward.
// Every mbarrier wait is bounded; on expiry the kernel records DEV_ERR_TIMEOUT
// and returns.
#include <cstring>

#include "common.cuh"
#include "internal.h"
#include "tc_ptx.cuh"

namespace fal {

namespace {

using namespace ptx;

constexpr int AT_BM = 128, AT_BN = 128;
constexpr int AT_THREADS = 192;
constexpr float AT_RESCALE_LOG2 = 8.f;  // raise the exponent's maximum only beyond 2^8 growth

struct AttnParams {
  CUtensorMap qkv;  // [B*T rows, 3*H*hd cols] bf16, box 64 x 128, 128-byte swizzle
  bf16* ctx;
  float* lse;
  int T, H, nq;
  float scale_log2;
  int* err;
};

template <int HD>
struct AttnSmem {
  static constexpr int KCH = HD / 64;                 // 64-column chunks of a head
  static constexpr int CHUNK = AT_BM * 64 * 2;        // one [128 rows][64] bf16 chunk = 16 KB
  static constexpr int Q_OFF = 0;
  static constexpr int K_OFF = Q_OFF + KCH * CHUNK;   // 2 stages
  static constexpr int V_OFF = K_OFF + 2 * KCH * CHUNK;
  static constexpr int P_OFF = V_OFF + 2 * KCH * CHUNK;  // 2 buffers of [128 q][128 keys]
  static constexpr int P_BYTES = AT_BM * AT_BN * 2;
  static constexpr int BAR_OFF = P_OFF + 2 * P_BYTES;
  static constexpr int TOTAL = BAR_OFF + 256 + 1024;  // + barriers + alignment slack
};

template <int HD>
__global__ void __launch_bounds__(AT_THREADS, 1) attn_fwd_tc_kernel(const __grid_constant__ AttnParams p) {
  using L = AttnSmem<HD>;
  constexpr int KCH = L::KCH;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* sbase = smem_raw + (base - raw);
  const uint32_t bar = base + L::BAR_OFF;
  // barriers
  const uint32_t qfull = bar;
  auto kfull = [&](int s) { return bar + 8u * (1 + s); };
  auto kempty = [&](int s) { return bar + 8u * (3 + s); };
  auto vfull = [&](int s) { return bar + 8u * (5 + s); };
  auto vempty = [&](int s) { return bar + 8u * (7 + s); };
  auto sfull = [&](int s) { return bar + 8u * (9 + s); };
  auto sfree = [&](int s) { return bar + 8u * (11 + s); };
  auto pfull = [&](int s) { return bar + 8u * (13 + s); };
  auto pempty = [&](int s) { return bar + 8u * (15 + s); };
  const uint32_t odone = bar + 8u * 17;
  const uint32_t drain = bar + 8u * 18;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sbase + L::BAR_OFF + 8 * 19);
  volatile uint32_t* abort_flag = reinterpret_cast<volatile uint32_t*>(sbase + L::BAR_OFF + 8 * 19 + 4);

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int qt = p.nq - 1 - (int)blockIdx.x;  // heaviest query tiles first
  const int bh = blockIdx.y, b = bh / p.H, h = bh % p.H;
  const int d = p.H * HD;
  const int row_base = b * p.T;  // first qkv row of this sequence
  const int nkv = qt + 1;         // causal: key tiles 0..qt

  if (threadIdx.x == 0) {
    mbar_init(qfull, 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(kfull(s), 1); mbar_init(kempty(s), 1); mbar_init(vfull(s), 1); mbar_init(vempty(s), 1);
      mbar_init(sfull(s), 1); mbar_init(sfree(s), 4); mbar_init(pfull(s), 4); mbar_init(pempty(s), 1);
    }
    mbar_init(odone, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;  // S buffers at columns 0 and 128, O at column 256

  if (warp == 0) {
    // ------------------------------------------------ producer
    bool ok = true;
    if (lane == 0) {
      mbar_arrive_expect_tx(qfull, KCH * L::CHUNK);
      for (int c = 0; c < KCH; ++c)
        tma_load_2d(base + L::Q_OFF + c * L::CHUNK, &p.qkv, h * HD + 64 * c, row_base + qt * AT_BM, qfull);
    }
    for (int j = 0; j < nkv && ok; ++j) {
      const int s = j & 1;
      const uint32_t par = ((j >> 1) & 1) ^ 1u;
      if (!mbar_wait(kempty(s), par, abort_flag)) { ok = false; break; }
      if (lane == 0) {
        mbar_arrive_expect_tx(kfull(s), KCH * L::CHUNK);
        for (int c = 0; c < KCH; ++c)
          tma_load_2d(base + L::K_OFF + (s * KCH + c) * L::CHUNK, &p.qkv, d + h * HD + 64 * c, row_base + j * AT_BN,
                      kfull(s));
      }
      __syncwarp();
      if (!mbar_wait(vempty(s), par, abort_flag)) { ok = false; break; }
      if (lane == 0) {
        mbar_arrive_expect_tx(vfull(s), KCH * L::CHUNK);
        for (int c = 0; c < KCH; ++c)
          tma_load_2d(base + L::V_OFF + (s * KCH + c) * L::CHUNK, &p.qkv, 2 * d + h * HD + 64 * c,
                      row_base + j * AT_BN, vfull(s));
      }
      __syncwarp();
    }
    if (!ok && lane == 0) set_dev_err(p.err, DEV_ERR_TIMEOUT);
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    const uint32_t id_qk = make_idesc_bf16(0, 0, AT_BM, AT_BN);
    const uint32_t id_pv = make_idesc_bf16(0, 1, AT_BM, HD);
    bool ok = mbar_wait(qfull, 0, abort_flag);
    bool issued = false;
    auto issue_s = [&](int j) -> bool {
      const int s = j & 1;
      const uint32_t par = (j >> 1) & 1;
      if (!mbar_wait(kfull(s), par, abort_flag)) return false;
      if (!mbar_wait(sfree(s), par ^ 1u, abort_flag)) return false;
      tc_fence_after();
      if (lane == 0) {
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
          const uint32_t qa = base + L::Q_OFF + (kk >> 2) * L::CHUNK + (kk & 3) * 32;
          const uint32_t kb = base + L::K_OFF + (s * KCH + (kk >> 2)) * L::CHUNK + (kk & 3) * 32;
          tc_mma(tmem + s * AT_BN, smem_desc(qa, 16, 1024), smem_desc(kb, 16, 1024), id_qk, kk > 0);
        }
        tc_commit(sfull(s));
        tc_commit(kempty(s));
      }
      __syncwarp();
      issued = true;
      return true;
    };
    auto issue_pv = [&](int j) -> bool {
      const int s = j & 1;
      const uint32_t par = (j >> 1) & 1;
      if (!mbar_wait(pfull(s), par, abort_flag)) return false;
      if (!mbar_wait(vfull(s), par, abort_flag)) return false;
      tc_fence_after();
      if (lane == 0) {
#pragma unroll
        for (int kk = 0; kk < AT_BN / 16; ++kk) {
          const uint32_t pa = base + L::P_OFF + s * L::P_BYTES + (kk >> 2) * L::CHUNK + (kk & 3) * 32;
          const uint32_t vb = base + L::V_OFF + s * KCH * L::CHUNK + kk * 2048;
          tc_mma(tmem + 256, smem_desc(pa, 16, 1024), smem_desc(vb, L::CHUNK, 1024), id_pv, (j > 0 || kk > 0));
        }
        tc_commit(vempty(s));
        tc_commit(pempty(s));
        tc_commit(odone);
      }
      __syncwarp();
      return true;
    };
    if (ok) ok = issue_s(0);
    for (int j = 0; j < nkv && ok; ++j) {
      if (j + 1 < nkv && !issue_s(j + 1)) { ok = false; break; }
      if (!issue_pv(j)) { ok = false; break; }
    }
    if (!ok) {
      if (lane == 0) set_dev_err(p.err, DEV_ERR_TIMEOUT);
      if (issued) {
        if (lane == 0) tc_commit(drain);
        __syncwarp();
        const uint64_t t0 = global_timer_ns();
        while (!mbar_try_wait(drain, 0) && global_timer_ns() - t0 < kWaitNs) {}
      }
    }
  } else {
    // ------------------------------------------------ softmax (one thread per query row)
    const int q4 = warp & 3;
    const int r = q4 * 32 + lane;         // row inside the 128-query tile = TMEM lane
    const int qpos = qt * AT_BM + r;      // query position in the sequence
    const uint32_t lane_addr = tmem + ((uint32_t)(q4 * 32) << 16);
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < nkv; ++j) {
      const int s = j & 1;
      const uint32_t par = (j >> 1) & 1;
      if (!mbar_wait(sfull(s), par, abort_flag)) { ok = false; break; }
      tc_fence_after();
      float sv[AT_BN];
#pragma unroll
      for (int c = 0; c < AT_BN / 32; ++c) {
        uint32_t rr[32];
        TMEM_LD32(lane_addr + s * AT_BN + c * 32, rr);
        tmem_wait_ld();
#pragma unroll
        for (int i = 0; i < 32; ++i) sv[c * 32 + i] = __uint_as_float(rr[i]) * p.scale_log2;
      }
      // the score buffer can be refilled once every row has been read
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(sfree(s));
      const int key0 = j * AT_BN;
      if (j == qt || key0 + AT_BN > p.T) {
#pragma unroll
        for (int i = 0; i < AT_BN; ++i)
          if (key0 + i > qpos || key0 + i >= p.T) sv[i] = -INFINITY;
      }
      float mt = -INFINITY;
#pragma unroll
      for (int i = 0; i < AT_BN; ++i) mt = fmaxf(mt, sv[i]);
      if (mt > m + AT_RESCALE_LOG2) {
        const float corr = (m == -INFINITY) ? 0.f : ex2_approx(m - mt);
        l *= corr;
        if (j > 0) {
          // O += P_{j-1} V_{j-1} must be complete before this row of O is rescaled
          if (!mbar_wait(odone, (j - 1) & 1, abort_flag)) { ok = false; break; }
          tc_fence_after();
#pragma unroll
          for (int c = 0; c < HD / 32; ++c) {
            uint32_t rr[32];
            TMEM_LD32(lane_addr + 256 + c * 32, rr);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i) rr[i] = __float_as_uint(__uint_as_float(rr[i]) * corr);
            TMEM_ST32(lane_addr + 256 + c * 32, rr);
          }
          tmem_wait_st();
        }
        m = mt;
      }
      // P_j = 2^(s - m) into the swizzled [128 q][128 keys] tile (two 64-key chunks)
      if (!mbar_wait(pempty(s), par ^ 1u, abort_flag)) { ok = false; break; }
      uint8_t* pt = sbase + L::P_OFF + s * L::P_BYTES;
      float rs = 0.f;
#pragma unroll
      for (int g = 0; g < AT_BN / 8; ++g) {
        float e[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          e[i] = ex2_approx(sv[g * 8 + i] - m);
          rs += e[i];
        }
        uint4 pk;
        __nv_bfloat162 t0 = __floats2bfloat162_rn(e[0], e[1]), t1 = __floats2bfloat162_rn(e[2], e[3]);
        __nv_bfloat162 t2 = __floats2bfloat162_rn(e[4], e[5]), t3 = __floats2bfloat162_rn(e[6], e[7]);
        pk.x = *reinterpret_cast<uint32_t*>(&t0); pk.y = *reinterpret_cast<uint32_t*>(&t1);
        pk.z = *reinterpret_cast<uint32_t*>(&t2); pk.w = *reinterpret_cast<uint32_t*>(&t3);
        const int chunk = g >> 3, gi = g & 7;
        *reinterpret_cast<uint4*>(pt + chunk * L::CHUNK + r * 128 + ((gi ^ (r & 7)) << 4)) = pk;
      }
      l += rs;
      fence_proxy_async_smem();  // generic-proxy P writes become visible to the MMA
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(pfull(s));
    }
    if (ok) ok = mbar_wait(odone, (nkv - 1) & 1, abort_flag);
    if (ok) {
      tc_fence_after();
      const float inv = 1.f / l;
      bf16* out = p.ctx + ((long)row_base + qpos) * d + h * HD;
#pragma unroll
      for (int c = 0; c < HD / 32; ++c) {
        uint32_t rr[32];
        TMEM_LD32(lane_addr + 256 + c * 32, rr);
        tmem_wait_ld();
        if (qpos < p.T) {
#pragma unroll
          for (int i = 0; i < 32; i += 8) {
            uint4 pk;
            __nv_bfloat162 t0 = __floats2bfloat162_rn(__uint_as_float(rr[i]) * inv, __uint_as_float(rr[i + 1]) * inv);
            __nv_bfloat162 t1 = __floats2bfloat162_rn(__uint_as_float(rr[i + 2]) * inv, __uint_as_float(rr[i + 3]) * inv);
            __nv_bfloat162 t2 = __floats2bfloat162_rn(__uint_as_float(rr[i + 4]) * inv, __uint_as_float(rr[i + 5]) * inv);
            __nv_bfloat162 t3 = __floats2bfloat162_rn(__uint_as_float(rr[i + 6]) * inv, __uint_as_float(rr[i + 7]) * inv);
            pk.x = *reinterpret_cast<uint32_t*>(&t0); pk.y = *reinterpret_cast<uint32_t*>(&t1);
            pk.z = *reinterpret_cast<uint32_t*>(&t2); pk.w = *reinterpret_cast<uint32_t*>(&t3);
            *reinterpret_cast<uint4*>(out + c * 32 + i) = pk;
          }
        }
      }
      if (qpos < p.T) p.lse[(long)bh * p.T + qpos] = m + __log2f(l);
    } else if (lane == 0) {
      set_dev_err(p.err, DEV_ERR_TIMEOUT);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

template <int HD>
int launch_fwd_tc(int B, int T, int H, const void* qkv, void* ctx, float* lse, int* err, cudaStream_t s,
                  std::string* msg) {
  using L = AttnSmem<HD>;
  static bool set = false;
  if (!set) {
    if (cudaFuncSetAttribute(attn_fwd_tc_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, L::TOTAL) !=
        cudaSuccess) {
      if (msg) *msg = "attention smem attribute failed";
      return 4;
    }
    set = true;
  }
  AttnParams p;
  memset(&p, 0, sizeof(p));
  const long d = (long)H * HD;
  if (!tma_map_2d(&p.qkv, qkv, 0, 3 * d, (unsigned long long)B * T, 3 * d, 64, AT_BM, 1, msg)) return 1;
  p.ctx = reinterpret_cast<bf16*>(ctx);
  p.lse = lse;
  p.T = T;
  p.H = H;
  p.nq = (T + AT_BM - 1) / AT_BM;
  p.scale_log2 = 1.4426950408889634f / sqrtf((float)HD);
  p.err = err;
  dim3 grid(p.nq, B * H);
  attn_fwd_tc_kernel<HD><<<grid, AT_THREADS, L::TOTAL, s>>>(p);
  count_launches(1);
  return 0;
}

}  // namespace

int attn_fwd_tc(int B, int T, int H, int hd, const void* qkv, void* ctx, float* lse, int* dev_err, cudaStream_t s,
                std::string* msg) {
  if (B <= 0 || T <= 0) return 0;
  int r;
  if (hd == 64) r = launch_fwd_tc<64>(B, T, H, qkv, ctx, lse, dev_err, s, msg);
  else if (hd == 128) r = launch_fwd_tc<128>(B, T, H, qkv, ctx, lse, dev_err, s, msg);
  else { if (msg) *msg = "tcgen05 attention needs head_dim 64 or 128"; return 6; }
  if (r) return r;
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) { if (msg) *msg = std::string("attention forward launch: ") + cudaGetErrorString(e); return 4; }
  return 0;
}

}  // namespace fal
