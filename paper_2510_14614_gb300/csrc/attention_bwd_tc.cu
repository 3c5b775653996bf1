// Causal multi-head attention backward on tcgen05 (bf16 operands, fp32
// accumulation in TMEM) as one persistent launch over two kinds of work item,
// each keeping its accumulators in TMEM for the whole item, so that no atomics
// and no fp32 dQ buffer are needed:
//
//   KV item  (batch, key/value head, 128-key block): resident K and V; streams
//            the 128-query blocks at or after the diagonal of every query head
//            of the group:
//              S^T = K Q^T,  dP^T = V dO^T                       (TMEM)
//              P^T = 2^(S^T*scale*log2e - lse[q]),  dS^T = P^T (dP^T - D[q])
//              dV += P^T dO,  dK += dS^T Q  (P^T and dS^T in bf16 from TMEM)
//   Q item   (batch, query head, 128-query block): resident Q and dO; streams
//            the 128-key blocks up to the diagonal, recomputes S, dP, P, dS
//            row-wise and accumulates dQ += dS K (dS from TMEM).
//
// Every product has N = 128 (or N = head_dim), the shape the tensor pipe runs
// at its full rate.  Each CTA (one per SM) takes items from a launch-wide
// counter; items are ranked in bands of about eight heads (so the CTAs working
// at any time share those heads' Q, K, V and dO in L2), heaviest first within
// a band.  Roles per CTA (576 threads):
//   warp 0      producer: takes the next item and hands it to the other roles,
//               loads the item's resident tiles once its predecessor's last S /
//               dP product has read the old ones, then the streamed tiles
//               through a ring of stages whose two halves are filled and freed
//               separately, their roles alternating with every use; for KV
//               items also lse and D of each query block.
//   warp 1      MMA issuer (one thread).  KV item, per block j: dV_j, S_{j+1},
//               dK_j, dP_{j+1} (dS^T_j is written over the dP^T_j columns, which
//               dP_{j+1} overwrites only after dK_j has read them).  Q item:
//               S_{j+1} as soon as the elementwise warps hold S_j in registers,
//               dQ_j, then dP_{j+1} (head_dim 128, two stages: the K block of
//               j+2 loads into the half V_j leaves after dP_j, so S_{j+2} need
//               not wait for dQ_j); with four stages dP_{j+1} precedes dQ_j.
//               The next item's S_0 and dP_0 run while the elementwise warps
//               store this item's accumulators.
//   warps 2..17 elementwise, four warps per TMEM lane quadrant (32 of the 128
//               streamed columns each), then the item's epilogue: dK (scaled)
//               and dV, or dQ (scaled), through a shared-memory staging tile and
//               TMA stores.
// Waiting warps sleep in the mbarrier (a suspend-time hint) rather than spin,
// leaving their issue slots to the warps that compute.
// TMEM (512 columns): S 0..127, dP 128..255, accumulators from 256 (dV | dK,
// or dQ followed by the Q item's dS in bf16 pairs).
// D = rowsum(dO * O) is an input: in the model it comes from the epilogue of the
// GEMM that produces dO, at the kernel-level entry points from a small pre-pass
// kernel (attention.cu).  Every mbarrier wait is bounded; on expiry the kernel
// records DEV_ERR_TIMEOUT, lets its copies and MMAs finish (again bounded),
// frees TMEM and returns.
#include <cudaTypedefs.h>

#include <cstring>
#include <mutex>

#include "common.cuh"
#include "internal.h"
#include "attn_ptx.cuh"

namespace fal {

namespace {

using namespace ptx;

// Elementwise warps per TMEM lane quadrant: each takes 128 / AB_EW of the
// streamed block's columns.
constexpr int AB_EW = 4;
constexpr int AB_COLS = 128 / AB_EW;
constexpr int AB_THREADS = 64 + 128 * AB_EW;

struct AttnBwdParams {
  CUtensorMap qkv;            // [B*T, dq] bf16, dq = (H + 2 Hkv) hd, box 64 x 128, 128-byte swizzle
  CUtensorMap dout;           // [B*T, d]  bf16, same box
  CUtensorMap dqkv_st;        // dqkv as [B][T][dq] bf16, box 64 x 128 x 1: stores clip at the end of each sequence
  const float* lse;           // [B, H, T] log2 units of the scaled scores
  const float* dvec;          // [B, H, T] rowsum(dO * O)
  bf16* dqkv;                 // [B*T, dq]
  int* next_item;             // work counter, zero at launch
  int B, T, H, Hkv, nblk;     // Hkv key/value heads (each serves H / Hkv query heads); nblk: 128-row blocks
  int band;                   // key/value heads per band of the item order
  float scale, scale_log2;
  int* err;
};

template <int HD>
struct BwdSmem {
  static constexpr int KCH = HD / 64;                  // 64-column chunks of a head
  static constexpr int CH = 128 * 64 * 2;              // one [128 rows][64] bf16 chunk, 16 KB
  static constexpr int STAGES = HD == 64 ? 4 : 2;
  static constexpr int RES_A = 0;                      // K (KV item) or Q (Q item)
  static constexpr int RES_B = KCH * CH;               // V or dO
  static constexpr int HALF = KCH * CH;                // half of a stage: one [128 rows][HD] tile
  static constexpr int ST_OFF = 2 * KCH * CH;
  static constexpr int STAGE = 2 * HALF;
  static constexpr int STG_OFF = ST_OFF + STAGES * STAGE;  // epilogue staging: one accumulator in bf16
  static constexpr int VEC_OFF = STG_OFF + KCH * CH;   // lse[128] | D[128] per stage (KV items)
  static constexpr int BAR_OFF = VEC_OFF + STAGES * 1024;
  static constexpr int TOTAL = BAR_OFF + (HD == 64 ? 512 : 256);  // barriers, TMEM slot, item ring
  static constexpr int LAUNCH = TOTAL + 1024 < 232448 ? TOTAL + 1024 : 232448;  // + alignment slack
};

// Item of rank k.  Items come in bands of p.band key/value heads (with their
// query heads), so that the CTAs working at any time share a few heads' Q, K,
// V and dO in L2; within a band heaviest first: per level (streamed blocks per
// query head, nblk down to 1) the band's KV items, then its Q items.
struct BwdItem {
  int kv, b, head, blk, nit, nit_h;  // head: key/value head (KV) or query head (Q); blk: 128-row block
};
__device__ __forceinline__ BwdItem decode_item(const AttnBwdParams& p, int k) {
  BwdItem it;
  const int gs = p.H / p.Hkv;
  const int per_band = p.nblk * p.band * (1 + gs);
  const int band = k / per_band, rb = k - band * per_band;
  const int nb = min(p.band, p.B * p.Hkv - band * p.band);  // key/value heads in this band
  const int per_level = nb * (1 + gs);
  const int level = rb / per_level, w = rb - level * per_level;
  if (w < nb) {
    const int kvh = band * p.band + w;     // batch-major key/value head index
    it.kv = 1;
    it.b = kvh / p.Hkv;
    it.head = kvh - it.b * p.Hkv;
    it.blk = level;                        // key block: query blocks blk .. nblk-1 see it
    it.nit_h = p.nblk - level;
    it.nit = gs * it.nit_h;
  } else {
    const int q = w - nb;
    const int kvh = band * p.band + q / gs;
    it.kv = 0;
    it.b = kvh / p.Hkv;
    it.head = (kvh - it.b * p.Hkv) * gs + q % gs;
    it.blk = p.nblk - 1 - level;           // query block: key blocks 0 .. blk
    it.nit_h = it.nit = it.blk + 1;
  }
  return it;
}

// Unbounded-by-abort wait used while draining after an error: returns when the
// phase completed or after kWaitNs.
__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity) && global_timer_ns() - t0 < kWaitNs) {}
}

template <int HD>
__global__ void __launch_bounds__(AB_THREADS, 1) attn_bwd_kernel(const __grid_constant__ AttnBwdParams p) {
  using L = BwdSmem<HD>;
  constexpr int KCH = L::KCH, NS = L::STAGES, NR = 2;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  // the layout needs its start 1024-byte aligned inside the launched size
  if (base - raw + L::TOTAL > L::LAUNCH) {
    if (threadIdx.x == 0) set_dev_err(p.err, DEV_ERR_TIMEOUT);
    return;
  }
  uint8_t* sbase = smem_raw + (base - raw);
  const uint32_t bar = base + L::BAR_OFF;
  const uint32_t res_full = bar, res_empty = bar + 8;
  // Each stage has two halves with their own barriers.  Streamed block g uses
  // stage g % NS; its first operand (Q of a KV block, K of a Q block) goes into
  // half ha(g) = (g / NS) & 1 and its second (dO, V) into the other half, so the
  // roles alternate on every use of a stage: a Q block's V half, free once dP has
  // read it, takes the K of the block two later, whose S product is needed soon,
  // while the K half, free only after dQ, takes its V.
  auto hf_full = [&](int s, int hh) { return bar + 8u * (2 + 2 * s + hh); };
  auto hf_empty = [&](int s, int hh) { return bar + 8u * (2 + 2 * NS + 2 * s + hh); };
  auto ha_of = [&](int g) { return (g / NS) & 1; };
  const uint32_t s_full = bar + 8u * (2 + 4 * NS), dp_full = s_full + 8, rd_s = s_full + 16, rd_dp = s_full + 24,
                 p_full = s_full + 32, ds_full = s_full + 40, ds_empty = s_full + 48, stg_full = s_full + 56,
                 stg_empty = s_full + 64, acc_full = s_full + 72, acc_empty = s_full + 80, drain = s_full + 88;
  auto it_full = [&](int i) { return s_full + 96 + 8u * i; };
  auto it_empty = [&](int i) { return s_full + 96 + 8u * (NR + i); };
  uint8_t* misc = sbase + L::BAR_OFF + 8 * (14 + 4 * NS + 2 * NR);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(misc);
  volatile uint32_t* abort_flag = reinterpret_cast<volatile uint32_t*>(misc + 4);
  volatile int* ring = reinterpret_cast<volatile int*>(misc + 8);  // item ranks handed from the producer to the other roles
  const float* vec_base = reinterpret_cast<const float*>(sbase + L::VEC_OFF);

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int gs = p.H / p.Hkv;
  const int d = p.H * HD;
  const int total = p.nblk * p.B * (p.Hkv + p.H);

  if (threadIdx.x == 0) {
    mbar_init(res_full, 1);
    mbar_init(res_empty, 1);
    for (int s = 0; s < NS; ++s)
      for (int hh = 0; hh < 2; ++hh) { mbar_init(hf_full(s, hh), 2); mbar_init(hf_empty(s, hh), 1); }
    mbar_init(s_full, 1);
    mbar_init(dp_full, 1);
    mbar_init(rd_s, 4 * AB_EW);
    mbar_init(rd_dp, 4 * AB_EW);
    mbar_init(p_full, 4 * AB_EW);
    mbar_init(ds_full, 4 * AB_EW);
    mbar_init(ds_empty, 1);
    mbar_init(stg_full, 4 * AB_EW);
    mbar_init(stg_empty, 1);
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, 4 * AB_EW);
    mbar_init(drain, 1);
    for (int i = 0; i < NR; ++i) { mbar_init(it_full(i), 1); mbar_init(it_empty(i), 4 * AB_EW + 1); }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // TMEM columns.  KV item: S^T (then P^T in bf16 pairs) 0..127, dP^T (then
  // dS^T in bf16 pairs) 128..255, dV, dK.  Q item: S, dP, dQ, dS in bf16 pairs.
  constexpr uint32_t T_S = 0, T_DP = 128, T_A1 = 256, T_A2 = 256 + HD, T_DS = 256 + HD;

  // n-th item of this CTA as handed out by the producer (-1: no more work)
  auto next_item = [&](int n, bool& ok) -> int {
    const int i = n % NR;
    if (!mbar_wait_sleep(it_full(i), (n / NR) & 1, abort_flag)) { ok = false; return -1; }
    return ring[i];
  };

  if (warp == 0) {
    // ------------------------------------------------ producer
    bool ok = true;
    int g = 0, n = 0;  // streamed blocks and resident sets issued so far
    for (int r = 0; ok; ++r) {
      // take the next item from the launch-wide counter and hand it to the other roles
      if (!mbar_wait_sleep(it_empty(r % NR), ((r / NR) & 1) ^ 1u, abort_flag)) { ok = false; break; }
      int k = 0;
      if (lane == 0) {
        k = atomicAdd(p.next_item, 1);
        if (k >= total) k = -1;
        ring[r % NR] = k;
        mbar_arrive(it_full(r % NR));
      }
      k = __shfl_sync(0xffffffffu, k, 0);
      if (k < 0) break;
      const BwdItem it = decode_item(p, k);
      const int row_base = it.b * p.T;
      const int kcol = d + (it.kv ? it.head : it.head / gs) * HD;
      const int vcol = kcol + p.Hkv * HD;
      // resident tiles, once the previous item's last S / dP products have read the old ones
      if (!mbar_wait_sleep(res_empty, (n & 1) ^ 1u, abort_flag)) { ok = false; break; }
      if (lane == 0) {
        mbar_arrive_expect_tx(res_full, 2 * KCH * L::CH);
        for (int c = 0; c < KCH; ++c) {
          if (it.kv) {
            tma_load_2d(base + L::RES_A + c * L::CH, &p.qkv, kcol + 64 * c, row_base + it.blk * 128, res_full);
            tma_load_2d(base + L::RES_B + c * L::CH, &p.qkv, vcol + 64 * c, row_base + it.blk * 128, res_full);
          } else {
            tma_load_2d(base + L::RES_A + c * L::CH, &p.qkv, it.head * HD + 64 * c, row_base + it.blk * 128, res_full);
            tma_load_2d(base + L::RES_B + c * L::CH, &p.dout, it.head * HD + 64 * c, row_base + it.blk * 128, res_full);
          }
        }
      }
      __syncwarp();
      ++n;
      for (int j = 0, jj = 0, hq = it.kv ? it.head * gs : it.head; j < it.nit && ok; ++j, ++g) {
        const int s = g % NS, ha = ha_of(g);
        const uint32_t par = ((g / NS) & 1) ^ 1u;
        const int c0 = (it.kv ? it.blk + jj : jj) * 128;   // first streamed row of the block
        const uint32_t sb = base + L::ST_OFF + s * L::STAGE;
        for (int t = 0; t < 2; ++t) {
          // t = 0: Q (KV) or K (Q) into half ha; t = 1: dO or V into the other half
          const int hh = ha ^ t;
          if (!mbar_wait_sleep(hf_empty(s, hh), par, abort_flag)) { ok = false; break; }
          if (lane == 0) {
            mbar_arrive_expect_tx(hf_full(s, hh), L::HALF);
            for (int c = 0; c < KCH; ++c) {
              const uint32_t dst = sb + hh * L::HALF + c * L::CH;
              if (it.kv) tma_load_2d(dst, t ? &p.dout : &p.qkv, hq * HD + 64 * c, row_base + c0, hf_full(s, hh));
              else tma_load_2d(dst, &p.qkv, (t ? vcol : kcol) + 64 * c, row_base + c0, hf_full(s, hh));
            }
          }
          if (it.kv && t == 0) {
            // lse and D of the block's 128 queries (zero beyond the sequence): all
            // eight loads of a lane are in flight together
            float* v = reinterpret_cast<float*>(sbase + L::VEC_OFF + s * 1024);
            const float* lsrc = p.lse + ((long)it.b * p.H + hq) * p.T;
            const float* dsrc = p.dvec + ((long)it.b * p.H + hq) * p.T;
            float lv[4], dvv[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const int tt = c0 + lane + 32 * q;
              lv[q] = tt < p.T ? __ldg(lsrc + tt) : 0.f;
              dvv[q] = tt < p.T ? __ldg(dsrc + tt) : 0.f;
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              v[lane + 32 * q] = lv[q];
              v[128 + lane + 32 * q] = dvv[q];
            }
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(hf_full(s, hh));
          __syncwarp();
        }
        if (++jj == it.nit_h) { jj = 0; ++hq; }
      }
    }
    if (!ok) {
      if (lane == 0) set_dev_err(p.err, DEV_ERR_TIMEOUT);
      // let the copies already issued land before the CTA's shared memory goes away
      if (n > 0) drain_wait(res_full, (uint32_t)((n - 1) & 1));
      for (int s = 0; s < NS && s < g; ++s) {
        const int last = g - 1 - ((g - 1 - s) % NS);      // last block that used stage s
        for (int hh = 0; hh < 2; ++hh) drain_wait(hf_full(s, hh), (uint32_t)((last / NS) & 1));
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    bool ok = true, issued = false;
    if (lane == 0) {
      const uint32_t id_s = make_idesc_bf16(0, 0, 128, 128);   // S, dP: both K-major, N = 128
      const uint32_t id_acc = make_idesc_bf16(0, 1, 128, HD);  // accumulate: B MN-major
      // descriptor words: one high word for every operand (stride 1024 between
      // 8-row groups, 128-byte swizzle); low words step by immediates along K
      const uint32_t hi = desc_hi(1024);
      const uint32_t lo_ra = desc_lo(base + L::RES_A, 16), lo_rb = desc_lo(base + L::RES_B, 16);
      int g = 0, gk = 0, n = 0;
      // S (resident A times the block's first operand) or dP (resident B times its second),
      // the streamed operand in half `half` of stage s
      auto issue_sdp = [&](uint32_t dst, uint32_t lo_res, int s, int half) {
        const uint32_t lo_st = desc_lo(base + L::ST_OFF + s * L::STAGE + half * L::HALF, 16);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
          const uint32_t o = (kk >> 2) * (L::CH >> 4) + (kk & 3) * 2;
          tc_mma_w(tmem + dst, lo_res + o, lo_st + o, hi, id_s, kk > 0);
        }
      };
      // accumulate A (bf16 pairs in TMEM from column a_col, each elementwise warp's
      // AB_COLS values of k packed at a_step * (k / AB_COLS) + (k % AB_COLS) / 2)
      // times a streamed operand as MN-major B
      constexpr int KPW = AB_COLS / 16;  // K16 steps per elementwise warp's columns
      auto issue_acc = [&](uint32_t dst, uint32_t a_col, uint32_t a_step, uint32_t lo_b, bool acc) {
#pragma unroll
        for (int kk = 0; kk < 8; ++kk)
          tc_mma_ts_w(tmem + dst, tmem + a_col + a_step * (kk / KPW) + 8 * (kk % KPW), lo_b + kk * 128, hi, id_acc,
                      (acc || kk > 0));
      };
      for (int r = 0; ok; ++r) {
        const int k = next_item(r, ok);
        if (ok) mbar_arrive(it_empty(r % NR));
        if (k < 0) break;
        const BwdItem it = decode_item(p, k);
        if (!mbar_wait_sleep(res_full, n & 1, abort_flag)) { ok = false; break; }
        {
          // S and dP of the item's first block: the S / dP columns are free once the
          // elementwise warps have read the previous block's
          const int s0 = g % NS, h0 = ha_of(g);
          const uint32_t par0 = (g / NS) & 1;
          if (!mbar_wait_sleep(hf_full(s0, h0), par0, abort_flag)) { ok = false; break; }
          if (g > 0 && !mbar_wait_sleep(rd_s, (g - 1) & 1, abort_flag)) { ok = false; break; }
          tc_fence_after();
          issue_sdp(T_S, lo_ra, s0, h0);
          tc_commit(s_full);
          if (!mbar_wait_sleep(hf_full(s0, h0 ^ 1), par0, abort_flag)) { ok = false; break; }
          if (g > 0 && !mbar_wait_sleep(rd_dp, (g - 1) & 1, abort_flag)) { ok = false; break; }
          tc_fence_after();
          issue_sdp(T_DP, lo_rb, s0, h0 ^ 1);
          tc_commit(dp_full);
          if (!it.kv) tc_commit(hf_empty(s0, h0 ^ 1));  // a Q block's V half: free once dP has read it
          issued = true;
          if (it.nit == 1) tc_commit(res_empty);
        }
        for (int j = 0; j < it.nit; ++j, ++g) {
          const int s = g % NS, ha = ha_of(g);
          const uint32_t sb = base + L::ST_OFF + s * L::STAGE;
          // MN-major B descriptors of this block's two operands (first: Q or K, second: dO or V)
          const uint32_t lo_first = desc_lo(sb + ha * L::HALF, L::CH), lo_second = desc_lo(sb + (ha ^ 1) * L::HALF, L::CH);
          const bool more = j + 1 < it.nit;
          const int s1 = (g + 1) % NS, h1 = ha_of(g + 1);
          const uint32_t par1 = ((g + 1) / NS) & 1;
          if (it.kv) {
            // dV += P^T dO
            if (!mbar_wait_sleep(p_full, gk & 1, abort_flag)) { ok = false; break; }
            if (j == 0 && n > 0 && !mbar_wait_sleep(acc_empty, (n - 1) & 1, abort_flag)) { ok = false; break; }
            tc_fence_after();
            issue_acc(T_A1, T_S, AB_COLS, lo_second, j > 0);
            if (more) {
              // S_{j+1} overwrites P^T_j, which the products above read first (in-order pipe)
              if (!mbar_wait_sleep(hf_full(s1, h1), par1, abort_flag)) { ok = false; break; }
              tc_fence_after();
              issue_sdp(T_S, lo_ra, s1, h1);
              tc_commit(s_full);
            }
            // dK += dS^T Q   (dS^T in bf16 pairs over the dP^T columns)
            if (!mbar_wait_sleep(ds_full, g & 1, abort_flag)) { ok = false; break; }
            tc_fence_after();
            issue_acc(T_A2, T_DP, AB_COLS, lo_first, j > 0);
            tc_commit(ds_empty);
            tc_commit(hf_empty(s, ha));
            tc_commit(hf_empty(s, ha ^ 1));
            if (more) {
              // dP_{j+1} overwrites dS^T_j after the product above has read it
              if (!mbar_wait_sleep(hf_full(s1, h1 ^ 1), par1, abort_flag)) { ok = false; break; }
              tc_fence_after();
              issue_sdp(T_DP, lo_rb, s1, h1 ^ 1);
              tc_commit(dp_full);
              if (j + 2 == it.nit) tc_commit(res_empty);
            }
            ++gk;
          } else {
            // S_{j+1} as soon as its K block is in and S_j has been read; dP_{j+1}
            // once its V block is in and dP_j has been read.  With two stages
            // (head_dim 128) dQ_j goes between them: the V block then arrives into
            // the K half that dQ_j frees, while S_{j+1} and the elementwise warps'
            // P phase proceed; with four stages dP_{j+1} goes first.
            constexpr bool dq_mid = NS == 2;
            if (more) {
              if (!mbar_wait_sleep(hf_full(s1, h1), par1, abort_flag)) { ok = false; break; }
              if (!mbar_wait_sleep(rd_s, g & 1, abort_flag)) { ok = false; break; }
              tc_fence_after();
              issue_sdp(T_S, lo_ra, s1, h1);
              tc_commit(s_full);
            }
            auto issue_dp_next = [&]() -> bool {
              if (!mbar_wait_sleep(hf_full(s1, h1 ^ 1), par1, abort_flag)) return false;
              if (!mbar_wait_sleep(rd_dp, g & 1, abort_flag)) return false;
              tc_fence_after();
              issue_sdp(T_DP, lo_rb, s1, h1 ^ 1);
              tc_commit(dp_full);
              tc_commit(hf_empty(s1, h1 ^ 1));  // its V half
              if (j + 2 == it.nit) tc_commit(res_empty);
              return true;
            };
            if (more && !dq_mid && !issue_dp_next()) { ok = false; break; }
            // dQ += dS K   (dS in bf16 pairs from column T_DS, AB_COLS / 2 columns per warp)
            if (!mbar_wait_sleep(ds_full, g & 1, abort_flag)) { ok = false; break; }
            if (j == 0 && n > 0 && !mbar_wait_sleep(acc_empty, (n - 1) & 1, abort_flag)) { ok = false; break; }
            tc_fence_after();
            issue_acc(T_A1, T_DS, AB_COLS / 2, lo_first, j > 0);
            tc_commit(ds_empty);
            tc_commit(hf_empty(s, ha));  // the K half
            if (more && dq_mid && !issue_dp_next()) { ok = false; break; }
          }
        }
        if (!ok) break;
        tc_commit(acc_full);
        ++n;
      }
      if (!ok) {
        set_dev_err(p.err, DEV_ERR_TIMEOUT);
        *abort_flag = 1;
        if (issued) {
          tc_commit(drain);
          drain_wait(drain, 0);
        }
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------ elementwise (AB_EW warps per lane quadrant)
    constexpr int C = AB_COLS;
    const int q4 = warp & 3, part = (warp - 2) >> 2;
    const int r = q4 * 32 + lane;  // TMEM lane = row inside the 128-row block
    const uint32_t lane_addr = tmem + ((uint32_t)(q4 * 32) << 16);
    const float sl2 = p.scale_log2;
    const bool storer = warp == 2 && lane == 0;  // issues the epilogue's TMA stores
    bool ok = true;
    int g = 0, gk = 0, n = 0, su = 0;  // su: uses of the epilogue staging buffer
    // this thread's HD / AB_EW accumulator columns in its row of the staging tile
    // (128-byte swizzle, 64-column chunks)
    constexpr int EC = HD / AB_EW;
    uint8_t* stg_row = sbase + L::STG_OFF + (part * EC / 64) * L::CH + (r >> 3) * 1024 + (r & 7) * 128;
    const int u0 = (part * EC % 64) / 8;
    for (int rk = 0; ok; ++rk) {
      const int k = next_item(rk, ok);
      __syncwarp();
      if (ok && lane == 0) mbar_arrive(it_empty(rk % NR));
      if (k < 0) break;
      const BwdItem it = decode_item(p, k);
      const int row = it.blk * 128 + r;  // key (KV) or query (Q) position of this thread
      float lse_r = 0.f, d_r = 0.f;
      if (!it.kv && row < p.T) {
        const long o = ((long)it.b * p.H + it.head) * p.T + row;
        lse_r = p.lse[o];
        d_r = p.dvec[o];
      }
      for (int j = 0, jj = 0; j < it.nit; ++j, ++g) {
        const int s = g % NS;
        const int c0 = (it.kv ? it.blk + jj : jj) * 128 + C * part;  // first streamed position of this warp's columns
        if (++jj == it.nit_h) jj = 0;
        // causal / sequence-end mask needed anywhere in this warp's 32 x C piece?
        const bool edge = it.kv ? (c0 < it.blk * 128 + 127 || c0 + C - 1 >= p.T || it.blk * 128 + 127 >= p.T)
                                : (c0 + C - 1 > it.blk * 128 || c0 + C - 1 >= p.T || it.blk * 128 + 127 >= p.T);
        if (!mbar_wait_sleep(s_full, g & 1, abort_flag)) { ok = false; break; }
        tc_fence_after();
        float sv[C];
#pragma unroll
        for (int c = 0; c < C; c += 32) TMEM_LD32(lane_addr + T_S + C * part + c, (reinterpret_cast<uint32_t*>(sv) + c));
        tmem_wait_ld();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(rd_s);  // S of this block is in registers
        if (it.kv) {
          // lse and D arrive with the block's Q half
          if (!mbar_wait_sleep(hf_full(s, ha_of(g)), (g / NS) & 1, abort_flag)) { ok = false; break; }
          const float* vl = vec_base + s * 256 + C * part;   // lse / D of this warp's C queries
          // P^T = 2^(S^T * scale - lse[q])
#pragma unroll
          for (int i = 0; i < C; i += 4) {
            const float4 l4 = *reinterpret_cast<const float4*>(vl + i);
            sv[i] = ex2_approx(fmaf(sv[i], sl2, -l4.x));
            sv[i + 1] = ex2_approx(fmaf(sv[i + 1], sl2, -l4.y));
            sv[i + 2] = ex2_approx(fmaf(sv[i + 2], sl2, -l4.z));
            sv[i + 3] = ex2_approx(fmaf(sv[i + 3], sl2, -l4.w));
          }
          if (edge) {
            // causal mask (query c sees key row iff c >= row) and sequence ends
#pragma unroll
            for (int i = 0; i < C; ++i) {
              const int c = c0 + i;
              if (c >= p.T || row >= p.T || c < row) sv[i] = 0.f;
            }
          }
          // P^T in bf16 pairs over the first C / 2 of this warp's S^T columns
          uint32_t pw[C / 2];
#pragma unroll
          for (int w = 0; w < C / 2; ++w) {
            __nv_bfloat162 t = __floats2bfloat162_rn(sv[2 * w], sv[2 * w + 1]);
            pw[w] = *reinterpret_cast<uint32_t*>(&t);
          }
#pragma unroll
          for (int c = 0; c < C / 2; c += 16) TMEM_ST16(lane_addr + T_S + C * part + c, (pw + c));
          tmem_wait_st();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(p_full);
          // dS^T = P^T (dP^T - D[q]) in bf16 pairs over this warp's dP^T columns, 32 at a time
          if (!mbar_wait_sleep(dp_full, g & 1, abort_flag)) { ok = false; break; }
          tc_fence_after();
#pragma unroll
          for (int hc = 0; hc < C / 32; ++hc) {
            uint32_t dr[32];
            TMEM_LD32(lane_addr + T_DP + C * part + 32 * hc, dr);
            tmem_wait_ld();
            uint32_t dw[16];
#pragma unroll
            for (int w = 0; w < 16; ++w) {
              const int i = 32 * hc + 2 * w;
              const float2 dd = *reinterpret_cast<const float2*>(vl + 128 + i);
              __nv_bfloat162 t = __floats2bfloat162_rn(sv[i] * (__uint_as_float(dr[2 * w]) - dd.x),
                                                       sv[i + 1] * (__uint_as_float(dr[2 * w + 1]) - dd.y));
              dw[w] = *reinterpret_cast<uint32_t*>(&t);
            }
            TMEM_ST16(lane_addr + T_DP + C * part + 16 * hc, dw);
          }
          tmem_wait_st();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) {
            mbar_arrive(rd_dp);
            mbar_arrive(ds_full);
          }
          ++gk;
        } else {
          // With two stages dP_j is issued after dQ_{j-1} and may still be running:
          // P first.  With four, dP_j has been issued beside S_j: read it first, so
          // that dP_{j+1} can follow as early as before.
          constexpr bool p_first = NS == 2;
          float dv[C];
          auto load_dp = [&]() -> bool {
            if (!mbar_wait_sleep(dp_full, g & 1, abort_flag)) return false;
            tc_fence_after();
#pragma unroll
            for (int c = 0; c < C; c += 32) TMEM_LD32(lane_addr + T_DP + C * part + c, (reinterpret_cast<uint32_t*>(dv) + c));
            tmem_wait_ld();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(rd_dp);  // dP of this block is in registers
            return true;
          };
          if (!p_first && !load_dp()) { ok = false; break; }
          const float nl = -lse_r;
#pragma unroll
          for (int i = 0; i < C; ++i) sv[i] = ex2_approx(fmaf(sv[i], sl2, nl));
          if (edge) {
            // causal mask (key c visible to query row iff c <= row) and sequence ends
#pragma unroll
            for (int i = 0; i < C; ++i) {
              const int c = c0 + i;
              if (c >= p.T || row >= p.T || c > row) sv[i] = 0.f;
            }
          }
          if (p_first && !load_dp()) { ok = false; break; }
#pragma unroll
          for (int i = 0; i < C; ++i) dv[i] = sv[i] * (dv[i] - d_r);
          uint32_t dw[C / 2];
#pragma unroll
          for (int w = 0; w < C / 2; ++w) {
            __nv_bfloat162 t = __floats2bfloat162_rn(dv[2 * w], dv[2 * w + 1]);
            dw[w] = *reinterpret_cast<uint32_t*>(&t);
          }
          // dS columns are free once the previous block's dQ (or dK) product has run
          if (g > 0 && !mbar_wait_sleep(ds_empty, (g - 1) & 1, abort_flag)) { ok = false; break; }
          tc_fence_after();
#pragma unroll
          for (int c = 0; c < C / 2; c += 16) TMEM_ST16(lane_addr + T_DS + (C / 2) * part + c, (dw + c));
          tmem_wait_st();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(ds_full);
        }
      }
      if (!ok) break;
      // ---------------------------------------------- epilogue: dK (scaled) and dV, or dQ (scaled)
      // Each accumulator goes through the staging tile (bf16, 128-byte swizzle)
      // and leaves by TMA stores into dqkv viewed as [B][T][dq], which clip the
      // rows past the end of the sequence.
      if (!mbar_wait_sleep(acc_full, n & 1, abort_flag)) { ok = false; break; }
      tc_fence_after();
      const int kcol = d + (it.kv ? it.head : it.head / gs) * HD;
      const int nacc = it.kv ? 2 : 1;
      for (int a = 0; a < nacc && ok; ++a, ++su) {
        // accumulator a: dV (KV) / dQ (Q) from T_A1, then dK (KV) from T_A2
        const uint32_t tcol = a ? T_A2 : T_A1;
        const float sc = (it.kv && a == 0) ? 1.f : p.scale;
        const int ocol = it.kv ? (a ? kcol : kcol + p.Hkv * HD) : it.head * HD;
        uint32_t acc[EC];
        if constexpr (EC >= 32) {
#pragma unroll
          for (int c = 0; c < EC; c += 32) TMEM_LD32(lane_addr + tcol + part * EC + c, (acc + c));
        } else {
          TMEM_LD16(lane_addr + tcol + part * EC, acc);
        }
        tmem_wait_ld();
        if (a + 1 == nacc) {
          // the accumulators are in registers: the next item's products may start
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(acc_empty);
        }
        // the staging tile is free once the previous TMA store has read it
        if (!mbar_wait_sleep(stg_empty, (su & 1) ^ 1u, abort_flag)) { ok = false; break; }
#pragma unroll
        for (int u = 0; u < EC / 8; ++u) {
          uint32_t w4[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            __nv_bfloat162 t = __floats2bfloat162_rn(__uint_as_float(acc[8 * u + 2 * e]) * sc,
                                                     __uint_as_float(acc[8 * u + 2 * e + 1]) * sc);
            w4[e] = *reinterpret_cast<uint32_t*>(&t);
          }
          *reinterpret_cast<uint4*>(stg_row + (((u0 + u) ^ (r & 7)) << 4)) = make_uint4(w4[0], w4[1], w4[2], w4[3]);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(stg_full);
        if (storer) {
          if (!mbar_wait_sleep(stg_full, su & 1, abort_flag)) { ok = false; break; }
          for (int c = 0; c < KCH; ++c)
            tma_store_3d(&p.dqkv_st, base + L::STG_OFF + c * L::CH, ocol + 64 * c, it.blk * 128, it.b);
          bulk_commit();
          bulk_wait_read_all();
          mbar_arrive(stg_empty);
        }
        __syncwarp();
      }
      if (!ok) break;
      ++n;
    }
    if (storer) bulk_wait_all();
    if (!ok && lane == 0) set_dev_err(p.err, DEV_ERR_TIMEOUT);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// 3-D bf16 tensor map (128-byte swizzle) over dqkv viewed as [B][T][dq], box
// 64 x 128 x 1, for the epilogue's stores: rows past the end of a sequence are
// clipped by the T extent instead of landing in the next sequence.
bool dqkv_store_map(CUtensorMap* m, void* ptr, long dq, int T, int B, std::string* msg) {
  static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  if (!encode) {
    if (msg) *msg = "cuTensorMapEncodeTiled not available from the driver";
    return false;
  }
  if ((reinterpret_cast<uintptr_t>(ptr) & 15) || ((dq * 2) & 15)) {
    if (msg) *msg = "dqkv needs a 16-byte aligned base and a 16-byte multiple row pitch";
    return false;
  }
  cuuint64_t dims[3] = {(cuuint64_t)dq, (cuuint64_t)T, (cuuint64_t)B};
  cuuint64_t strides[2] = {(cuuint64_t)dq * 2, (cuuint64_t)dq * 2 * T};
  cuuint32_t box[3] = {64, 128, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  if (encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, ptr, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
             CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) !=
      CUDA_SUCCESS) {
    if (msg) *msg = "cuTensorMapEncodeTiled (dqkv store map) failed";
    return false;
  }
  return true;
}

template <int HD>
int launch_bwd(const AttnBwdParams& p, cudaStream_t s, std::string* msg) {
  constexpr int smem = BwdSmem<HD>::LAUNCH;
  static_assert(BwdSmem<HD>::TOTAL + 512 <= smem, "attention backward shared memory");
  static bool set = false;
  if (!set) {
    if (cudaFuncSetAttribute(attn_bwd_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess) {
      if (msg) *msg = "attention backward smem attribute failed";
      return 4;
    }
    set = true;
  }
  const int total = p.nblk * p.B * (p.Hkv + p.H);
  const int grid = total < num_sms() ? total : num_sms();
  if (cudaMemsetAsync(p.next_item, 0, sizeof(int), s) != cudaSuccess) {
    if (msg) *msg = "attention backward: clearing the work counter failed";
    return 4;
  }
  attn_bwd_kernel<HD><<<grid, AB_THREADS, smem, s>>>(p);
  count_launches(1);
  return 0;
}

}  // namespace

int attn_bwd_tc(int B, int T, int H, int Hkv, int hd, const void* qkv, const void* dctx, const float* lse,
                const float* dvec, int* counter, void* dqkv, int* dev_err, cudaStream_t s, std::string* msg) {
  if (B <= 0 || T <= 0) return 0;
  if (hd != 64 && hd != 128) { if (msg) *msg = "tcgen05 attention needs head_dim 64 or 128"; return 6; }
  if (Hkv <= 0 || H % Hkv) { if (msg) *msg = "heads must be a multiple of the key/value heads"; return 1; }
  AttnBwdParams p;
  memset(&p, 0, sizeof(p));
  const long d = (long)H * hd, dq = (long)(H + 2 * Hkv) * hd;
  const unsigned long long rows = (unsigned long long)B * T;
  if (!tma_map_2d(&p.qkv, qkv, 0, dq, rows, dq, 64, 128, 1, msg) || !tma_map_2d(&p.dout, dctx, 0, d, rows, d, 64, 128, 1, msg) ||
      !dqkv_store_map(&p.dqkv_st, dqkv, dq, T, B, msg))
    return 1;
  const long nblk = (T + 127) / 128;
  if (nblk * B * (long)(Hkv + H) > 0x7fffffffL) { if (msg) *msg = "attention backward: too many work items"; return 1; }
  p.lse = lse;
  p.dvec = dvec;
  p.dqkv = reinterpret_cast<bf16*>(dqkv);
  p.next_item = counter;
  p.B = B;
  p.T = T;
  p.H = H;
  p.Hkv = Hkv;
  p.nblk = (int)nblk;
  // bands of about eight query heads
  const int gs = H / Hkv;
  p.band = gs >= 8 ? 1 : 8 / gs;
  p.scale = 1.f / sqrtf((float)hd);
  p.scale_log2 = 1.4426950408889634f / sqrtf((float)hd);
  p.err = dev_err;
  const int r = hd == 64 ? launch_bwd<64>(p, s, msg) : launch_bwd<128>(p, s, msg);
  if (r) return r;
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) { if (msg) *msg = std::string("attention backward launch: ") + cudaGetErrorString(e); return 4; }
  return 0;
}

}  // namespace fal
