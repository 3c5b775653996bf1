// Causal multi-head attention forward on tcgen05 (bf16 operands, fp32
// accumulation in TMEM): ctx = softmax(Q K^T / sqrt(hd) + causal) V, one CTA
// per (batch, head, 256-query block) holding two 128-query tiles A and B.
//
//   warp 0      TMA producer: both Q tiles once, then K and V tiles of 128 keys
//               (two stages each) straight out of the packed qkv rows; every
//               K / V tile serves both query tiles.
//   warp 1      MMA issuer: S_x = Q_x K_j^T (128 x 128 fp32 in TMEM), then
//               O_x += P_x V_j with P_x read from TMEM.  Per key tile the
//               order is PV_A(j), S_A(j+1), PV_B(j), S_B(j+1), so each tile's
//               scores for the next key tile are computed while the other
//               tile's softmax runs.
//   warps 2..5  softmax of tile A, warps 6..9 of tile B, one thread per query
//               row: reads its score row from TMEM, masks it, keeps a running
//               maximum m and sum l and writes P = 2^(s*scale - m) in bf16 pairs
//               over the score columns it read.  The maximum used for the
//               exponent is only raised when the row maximum grows by more than
//               2^8 (P then stays below 256); only then is the row of O in TMEM
//               rescaled.  Finally O / l is stored in bf16 and the log-sum-exp
//               m + log2(l) (log2 units of S*log2(e)) is saved for the backward.
// Every mbarrier wait is bounded; on expiry the kernel records DEV_ERR_TIMEOUT
// and returns.
#include <cstring>

#include "common.cuh"
#include "internal.h"
#include "attn_ptx.cuh"

namespace fal {

namespace {

using namespace ptx;

constexpr int AT_BM = 128, AT_BN = 128;
constexpr float AT_RESCALE_LOG2 = 8.f;  // raise the exponent's maximum only beyond 2^8 growth

struct AttnParams {
  CUtensorMap qkv;  // [B*T rows, (H + 2 Hkv)*hd cols] bf16, box 64 x 128, 128-byte swizzle
  bf16* ctx;
  float* lse;
  int T, H, Hkv, nq;  // Hkv key/value heads, each serving H / Hkv query heads (Hkv = H: MHA)
  float scale_log2;
  int* err;
};

// ---------------------------------------------------------------- two query tiles per CTA
// One CTA per (256-query block, head): query tiles A (rows 256t..256t+127)
// and B (the next 128 rows) share every K and V tile.  TMEM columns: S_A at 0,
// S_B at 128, O_A at 256, O_B at 256 + HD.  Each softmax writes P in bf16 over
// the score columns it came from, and O += P V reads P from TMEM as the A
// operand.  Warps 2..5 run tile A's softmax and warps 6..9 tile B's, so each
// tile's softmax overlaps the other tile's products and the two softmax
// warpgroups hide each other's latencies.
constexpr int AT2_THREADS = 320;

template <int HD>
struct Attn2Smem {
  static constexpr int KCH = HD / 64;
  static constexpr int CHUNK = 128 * 64 * 2;       // one [128 rows][64] bf16 chunk = 16 KB
  static constexpr int QA_OFF = 0;
  static constexpr int QB_OFF = KCH * CHUNK;
  static constexpr int K_OFF = 2 * KCH * CHUNK;    // 2 stages
  static constexpr int V_OFF = K_OFF + 2 * KCH * CHUNK;
  static constexpr int BAR_OFF = V_OFF + 2 * KCH * CHUNK;
  static constexpr int TOTAL = BAR_OFF + 256 + 1024;
};

template <int HD>
__global__ void __launch_bounds__(AT2_THREADS, 1) attn_fwd2_kernel(const __grid_constant__ AttnParams p) {
  using L = Attn2Smem<HD>;
  constexpr int KCH = L::KCH;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* sbase = smem_raw + (base - raw);
  const uint32_t bar = base + L::BAR_OFF;
  const uint32_t qfull = bar;
  auto kfull = [&](int s) { return bar + 8u * (1 + s); };
  auto kempty = [&](int s) { return bar + 8u * (3 + s); };
  auto vfull = [&](int s) { return bar + 8u * (5 + s); };
  auto vempty = [&](int s) { return bar + 8u * (7 + s); };
  auto sfull = [&](int x) { return bar + 8u * (9 + x); };
  auto pfull = [&](int x) { return bar + 8u * (11 + x); };
  auto odone = [&](int x) { return bar + 8u * (13 + x); };
  const uint32_t drain = bar + 8u * 15;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sbase + L::BAR_OFF + 8 * 16);
  volatile uint32_t* abort_flag = reinterpret_cast<volatile uint32_t*>(sbase + L::BAR_OFF + 8 * 16 + 4);

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int t2 = p.nq - 1 - (int)blockIdx.x;  // heaviest 256-query blocks first
  const int bh = blockIdx.y, b = bh / p.H, h = bh % p.H;
  const int d = p.H * HD;
  const int g = h / (p.H / p.Hkv);                     // key / value head of this query head
  const int kcol = d + g * HD, vcol = d + (p.Hkv + g) * HD;
  const int row_base = b * p.T;
  const int nkb_all = (p.T + AT_BN - 1) / AT_BN;
  // causal: tile A sees key blocks 0..2t2, tile B 0..2t2+1 (none if it starts past T)
  const int nA = min(2 * t2 + 1, nkb_all);
  const int nB = (256 * t2 + 128 < p.T) ? min(2 * t2 + 2, nkb_all) : 0;
  const int nkb = max(nA, nB);

  if (threadIdx.x == 0) {
    mbar_init(qfull, 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(kfull(s), 1); mbar_init(kempty(s), 1); mbar_init(vfull(s), 1); mbar_init(vempty(s), 1);
      mbar_init(sfull(s), 1); mbar_init(pfull(s), 4); mbar_init(odone(s), 1);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------ producer
    bool ok = true;
    if (lane == 0) {
      mbar_arrive_expect_tx(qfull, 2 * KCH * L::CHUNK);
      for (int c = 0; c < KCH; ++c) {
        tma_load_2d(base + L::QA_OFF + c * L::CHUNK, &p.qkv, h * HD + 64 * c, row_base + 256 * t2, qfull);
        tma_load_2d(base + L::QB_OFF + c * L::CHUNK, &p.qkv, h * HD + 64 * c, row_base + 256 * t2 + 128, qfull);
      }
    }
    for (int j = 0; j < nkb && ok; ++j) {
      const int s = j & 1;
      const uint32_t par = ((j >> 1) & 1) ^ 1u;
      if (!mbar_wait(kempty(s), par, abort_flag)) { ok = false; break; }
      if (lane == 0) {
        mbar_arrive_expect_tx(kfull(s), KCH * L::CHUNK);
        for (int c = 0; c < KCH; ++c)
          tma_load_2d(base + L::K_OFF + (s * KCH + c) * L::CHUNK, &p.qkv, kcol + 64 * c, row_base + j * AT_BN,
                      kfull(s));
      }
      __syncwarp();
      if (!mbar_wait(vempty(s), par, abort_flag)) { ok = false; break; }
      if (lane == 0) {
        mbar_arrive_expect_tx(vfull(s), KCH * L::CHUNK);
        for (int c = 0; c < KCH; ++c)
          tma_load_2d(base + L::V_OFF + (s * KCH + c) * L::CHUNK, &p.qkv, vcol + 64 * c,
                      row_base + j * AT_BN, vfull(s));
      }
      __syncwarp();
    }
    if (!ok && lane == 0) set_dev_err(p.err, DEV_ERR_TIMEOUT);
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    const uint32_t id_qk = make_idesc_bf16(0, 0, AT_BM, AT_BN);
    const uint32_t id_pv = make_idesc_bf16(0, 1, AT_BM, HD);
    const uint32_t dhi = desc_hi(1024);
    bool ok = mbar_wait(qfull, 0, abort_flag);
    bool issued = false;
    // S_x = Q_x K_j^T into columns 128 x
    auto issue_s = [&](int x, int j) -> bool {
      const int s = j & 1;
      if (!mbar_wait(kfull(s), (j >> 1) & 1, abort_flag)) return false;
      tc_fence_after();
      if (lane == 0) {
        // descriptor low words stepped by immediates along K (one shared high word)
        const uint32_t lo_q = desc_lo(base + (x ? L::QB_OFF : L::QA_OFF), 16);
        const uint32_t lo_k = desc_lo(base + L::K_OFF + s * KCH * L::CHUNK, 16);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
          const uint32_t o = (kk >> 2) * (L::CHUNK >> 4) + (kk & 3) * 2;
          tc_mma_w(tmem + x * AT_BN, lo_q + o, lo_k + o, dhi, id_qk, kk > 0);
        }
        tc_commit(sfull(x));
      }
      __syncwarp();
      issued = true;
      return true;
    };
    // O_x += P_x V_j with P_x read from TMEM (bf16 pairs over the S_x columns)
    auto issue_pv = [&](int x, int j) -> bool {
      const int s = j & 1;
      if (!mbar_wait(pfull(x), j & 1, abort_flag)) return false;
      if (!mbar_wait(vfull(s), (j >> 1) & 1, abort_flag)) return false;
      tc_fence_after();
      if (lane == 0) {
        const uint32_t lo_v = desc_lo(base + L::V_OFF + s * KCH * L::CHUNK, L::CHUNK);  // MN-major
#pragma unroll
        for (int kk = 0; kk < AT_BN / 16; ++kk)
          tc_mma_ts_w(tmem + 256 + x * HD, tmem + x * AT_BN + kk * 8, lo_v + kk * 128, dhi, id_pv, (j > 0 || kk > 0));
        tc_commit(odone(x));
      }
      __syncwarp();
      return true;
    };
    if (ok && nA > 0) ok = issue_s(0, 0);
    if (ok && nB > 0) ok = issue_s(1, 0);
    if (ok && lane == 0) tc_commit(kempty(0));
    __syncwarp();
    for (int j = 0; j < nkb && ok; ++j) {
      // tile A: its products for block j, then its scores for block j+1 (which
      // overwrite P_A: issued after the product that reads it)
      if (j < nA) {
        if (!issue_pv(0, j)) { ok = false; break; }
        if (j + 1 < nA && !issue_s(0, j + 1)) { ok = false; break; }
      }
      if (j < nB && !issue_pv(1, j)) { ok = false; break; }
      if (lane == 0) tc_commit(vempty(j & 1));
      __syncwarp();
      if (j + 1 < nB && !issue_s(1, j + 1)) { ok = false; break; }
      if (j + 1 < nkb) {
        if (lane == 0) tc_commit(kempty((j + 1) & 1));
        __syncwarp();
      }
    }
    if (!ok) {
      if (lane == 0) set_dev_err(p.err, DEV_ERR_TIMEOUT);
      if (issued) {
        if (lane == 0) tc_commit(drain);
        __syncwarp();
        const uint64_t t0 = global_timer_ns();
        while (!mbar_try_wait(drain, 0) && global_timer_ns() - t0 < kWaitNs) {}
      }
      *abort_flag = 1;
    }
  } else {
    // ------------------------------------------------ softmax (one thread per query row of tile x)
    const int x = (warp - 2) >> 2;
    const int q4 = warp & 3;
    const int r = q4 * 32 + lane;                 // TMEM lane = row inside the tile
    const int qpos = 256 * t2 + 128 * x + r;      // query position in the sequence
    const int nx = x ? nB : nA;
    const uint32_t lane_addr = tmem + ((uint32_t)(q4 * 32) << 16);
    const uint32_t s_col = x * AT_BN, o_col = 256 + x * HD;
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < nx; ++j) {
      if (!mbar_wait(sfull(x), j & 1, abort_flag)) { ok = false; break; }
      tc_fence_after();
      // raw scores; the scale is applied inside the exponent (it is positive, so
      // the maximum of the raw scores gives the scaled maximum)
      float sv[AT_BN];
#pragma unroll
      for (int c = 0; c < AT_BN / 32; ++c) TMEM_LD32(lane_addr + s_col + c * 32, (reinterpret_cast<uint32_t*>(sv) + c * 32));
      tmem_wait_ld();
      const int key0 = j * AT_BN;
      if (key0 + AT_BN - 1 > 256 * t2 + 128 * x || key0 + AT_BN > p.T) {
#pragma unroll
        for (int i = 0; i < AT_BN; ++i)
          if (key0 + i > qpos || key0 + i >= p.T) sv[i] = -INFINITY;
      }
      float mx[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) mx[k] = sv[k];
#pragma unroll
      for (int i = 8; i < AT_BN; ++i) mx[i & 7] = fmaxf(mx[i & 7], sv[i]);
      const float mt =
          p.scale_log2 * fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])), fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
      float corr = 1.f;
      bool rescale = false;
      if (mt > m + AT_RESCALE_LOG2) {
        corr = (m == -INFINITY) ? 0.f : ex2_approx(m - mt);
        l *= corr;
        rescale = j > 0;
        m = mt;
      }
      // P_j = 2^(s * scale - m) in bf16 pairs over the first 64 score columns
      const float sc = p.scale_log2;
      float rsum[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        uint32_t pw[16];
#pragma unroll
        for (int w = 0; w < 16; ++w) {
          const float e0 = ex2_approx(fmaf(sv[q * 32 + 2 * w], sc, -m));
          const float e1 = ex2_approx(fmaf(sv[q * 32 + 2 * w + 1], sc, -m));
          rsum[w & 3] += e0 + e1;
          __nv_bfloat162 t = __floats2bfloat162_rn(e0, e1);
          pw[w] = *reinterpret_cast<uint32_t*>(&t);
        }
        TMEM_ST16(lane_addr + s_col + q * 16, pw);
      }
      l += (rsum[0] + rsum[1]) + (rsum[2] + rsum[3]);
      if (rescale) {
        // O += P_{j-1} V_{j-1} must be complete before this row of O is rescaled
        if (!mbar_wait(odone(x), (j - 1) & 1, abort_flag)) { ok = false; break; }
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < HD / 32; ++c) {
          uint32_t rr[32];
          TMEM_LD32(lane_addr + o_col + c * 32, rr);
          tmem_wait_ld();
#pragma unroll
          for (int i = 0; i < 32; ++i) rr[i] = __float_as_uint(__uint_as_float(rr[i]) * corr);
          TMEM_ST32(lane_addr + o_col + c * 32, rr);
        }
      }
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(pfull(x));
    }
    if (ok && nx > 0) ok = mbar_wait(odone(x), (nx - 1) & 1, abort_flag);
    if (ok && nx > 0) {
      tc_fence_after();
      const float inv = 1.f / l;
      bf16* out = p.ctx + ((long)row_base + qpos) * d + h * HD;
#pragma unroll
      for (int c = 0; c < HD / 32; ++c) {
        uint32_t rr[32];
        TMEM_LD32(lane_addr + o_col + c * 32, rr);
        tmem_wait_ld();
        if (qpos < p.T) {
#pragma unroll
          for (int i = 0; i < 32; i += 8) {
            uint4 pk;
            __nv_bfloat162 t0 = __floats2bfloat162_rn(__uint_as_float(rr[i]) * inv, __uint_as_float(rr[i + 1]) * inv);
            __nv_bfloat162 t1 = __floats2bfloat162_rn(__uint_as_float(rr[i + 2]) * inv, __uint_as_float(rr[i + 3]) * inv);
            __nv_bfloat162 t2v = __floats2bfloat162_rn(__uint_as_float(rr[i + 4]) * inv, __uint_as_float(rr[i + 5]) * inv);
            __nv_bfloat162 t3 = __floats2bfloat162_rn(__uint_as_float(rr[i + 6]) * inv, __uint_as_float(rr[i + 7]) * inv);
            pk.x = *reinterpret_cast<uint32_t*>(&t0); pk.y = *reinterpret_cast<uint32_t*>(&t1);
            pk.z = *reinterpret_cast<uint32_t*>(&t2v); pk.w = *reinterpret_cast<uint32_t*>(&t3);
            *reinterpret_cast<uint4*>(out + c * 32 + i) = pk;
          }
        }
      }
      if (qpos < p.T) p.lse[(long)bh * p.T + qpos] = m + __log2f(l);
    } else if (!ok && lane == 0) {
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
int launch_fwd_tc(int B, int T, int H, int Hkv, const void* qkv, void* ctx, float* lse, int* err, cudaStream_t s,
                  std::string* msg) {
  using L = Attn2Smem<HD>;
  static bool set = false;
  if (!set) {
    if (cudaFuncSetAttribute(attn_fwd2_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, L::TOTAL) !=
        cudaSuccess) {
      if (msg) *msg = "attention smem attribute failed";
      return 4;
    }
    set = true;
  }
  AttnParams p;
  memset(&p, 0, sizeof(p));
  const long dq = (long)(H + 2 * Hkv) * HD;
  if (!tma_map_2d(&p.qkv, qkv, 0, dq, (unsigned long long)B * T, dq, 64, AT_BM, 1, msg)) return 1;
  p.ctx = reinterpret_cast<bf16*>(ctx);
  p.lse = lse;
  p.T = T;
  p.H = H;
  p.Hkv = Hkv;
  p.nq = (T + 255) / 256;  // 256-query blocks
  p.scale_log2 = 1.4426950408889634f / sqrtf((float)HD);
  p.err = err;
  dim3 grid(p.nq, B * H);
  attn_fwd2_kernel<HD><<<grid, AT2_THREADS, L::TOTAL, s>>>(p);
  count_launches(1);
  return 0;
}

}  // namespace

int attn_fwd_tc(int B, int T, int H, int Hkv, int hd, const void* qkv, void* ctx, float* lse, int* dev_err,
                cudaStream_t s, std::string* msg) {
  if (B <= 0 || T <= 0) return 0;
  if (Hkv <= 0 || H % Hkv) { if (msg) *msg = "heads must be a multiple of the key/value heads"; return 1; }
  int r;
  if (hd == 64) r = launch_fwd_tc<64>(B, T, H, Hkv, qkv, ctx, lse, dev_err, s, msg);
  else if (hd == 128) r = launch_fwd_tc<128>(B, T, H, Hkv, qkv, ctx, lse, dev_err, s, msg);
  else { if (msg) *msg = "tcgen05 attention needs head_dim 64 or 128"; return 6; }
  if (r) return r;
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) { if (msg) *msg = std::string("attention forward launch: ") + cudaGetErrorString(e); return 4; }
  return 0;
}

}  // namespace fal
