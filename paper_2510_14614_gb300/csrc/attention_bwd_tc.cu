// Causal multi-head attention backward on tcgen05 (bf16 operands, fp32
// accumulation in TMEM), in two passes that each keep their accumulators in
// TMEM for the whole CTA, so that no atomics and no fp32 dQ buffer are needed:
//
//   pass KV  one CTA per (128-key block, head); streams the 64-query blocks
//            that can see those keys:
//              S^T  = K Q^T,  dP^T = V dO^T                    (TMEM, 2 buffers)
//              P^T  = 2^(S^T*scale*log2e - lse[q]),  dS^T = P^T (dP^T - D[q])
//              dV  += P^T dO,  dK += dS^T Q                    (TMEM accumulators)
//   pass Q   one CTA per (128-query block, head); streams the 64-key blocks
//            up to the diagonal, recomputes S, dP, P and dS row-wise and
//            accumulates dQ += dS K.
//
// The two passes share one body template and run in one launch (alternating
// CTAs, heaviest blocks of both first).  Roles per CTA (320 threads):
//   warp 0      producer: the resident 128-row tiles once (K and V, or Q and
//               dO), then the streamed 64-row tiles through a 4-stage ring; in
//               pass KV it also stages lse and D of each query block.
//   warp 1      MMA issuer (one thread), software-pipelined: S / dP of block
//               j+1 are issued before the accumulating products of block j,
//               so the tensor pipe works while the elementwise warps handle j.
//   warps 2..9  elementwise, two warps per TMEM lane quadrant (32 of the 64
//               columns each): P and dS in bf16 written back into TMEM over
//               the scores they came from; the accumulating MMAs read them
//               from there as their A operand (so only B comes from shared
//               memory, whose bandwidth bounds these small-N products).  At
//               the end they scale and store dK, dV or dQ in bf16.
// D = rowsum(dO * O) is an input: in the model it comes from the epilogue of the
// GEMM that produces dO, at the kernel-level entry points from a small pre-pass
// kernel (attention.cu).  Every mbarrier wait
// is bounded; on expiry the kernel records DEV_ERR_TIMEOUT, lets its MMAs
// finish, frees TMEM and returns.
#include <cstring>

#include "common.cuh"
#include "internal.h"
#include "tc_ptx.cuh"

namespace fal {

namespace {

using namespace ptx;

constexpr int AB2_THREADS = 320;
constexpr int AB2_STAGES = 4;

struct AttnBwd2Params {
  CUtensorMap qkv128, qkv64;  // [B*T, dq] bf16, dq = (H + 2 Hkv) hd, boxes 64 x 128 and 64 x 64, 128-byte swizzle
  CUtensorMap do128, do64;    // [B*T, d]  bf16, same boxes
  const float* lse;           // [B, H, T] log2 units of the scaled scores
  const float* dvec;          // [B, H, T] rowsum(dO * O)
  bf16* dqkv;                 // [B*T, dq]
  int T, H, Hkv, nblk;        // Hkv key/value heads (each serves H / Hkv query heads); nblk: 128-row blocks
  float scale, scale_log2;
  int* err;
};

template <int HD, bool KV>
struct Bwd2Smem {
  static constexpr int KCH = HD / 64;
  static constexpr int RES = 128 * 64 * 2;             // [128 rows][64] bf16 chunk (resident tiles)
  static constexpr int STR = 64 * 64 * 2;              // [64 rows][64] bf16 chunk (streamed tiles)
  static constexpr int RES_A = 0;                      // K (KV) or Q (Q)
  static constexpr int RES_B = RES_A + KCH * RES;      // V (KV) or dO (Q)
  static constexpr int STAGE = 2 * KCH * STR;          // Q | dO (KV) or K | V (Q)
  static constexpr int ST_OFF = RES_B + KCH * RES;
  static constexpr int VEC_OFF = ST_OFF + AB2_STAGES * STAGE;  // KV: lse[64] | D[64] per stage
  static constexpr int BAR_OFF = VEC_OFF + (KV ? AB2_STAGES * 512 : 0);
  static constexpr int TOTAL = BAR_OFF + 256 + 1024;   // barriers + alignment slack
};

template <int HD, bool KV>
__device__ __forceinline__ void attn_bwd2_body(const AttnBwd2Params& p, int bx) {
  using L = Bwd2Smem<HD, KV>;
  constexpr int KCH = L::KCH;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* sbase = smem_raw + (base - raw);
  const uint32_t bar = base + L::BAR_OFF;
  const uint32_t res_full = bar;
  auto st_full = [&](int s) { return bar + 8u * (1 + s); };
  auto st_empty = [&](int s) { return bar + 8u * (1 + AB2_STAGES + s); };
  auto sdp_full = [&](int b) { return bar + 8u * (1 + 2 * AB2_STAGES + b); };
  auto ps_full = [&](int b) { return bar + 8u * (3 + 2 * AB2_STAGES + b); };
  const uint32_t fin = bar + 8u * (5 + 2 * AB2_STAGES), drain = bar + 8u * (6 + 2 * AB2_STAGES);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sbase + L::BAR_OFF + 8 * (7 + 2 * AB2_STAGES));
  volatile uint32_t* abort_flag = reinterpret_cast<volatile uint32_t*>(sbase + L::BAR_OFF + 8 * (7 + 2 * AB2_STAGES) + 4);
  const float* vec_base = reinterpret_cast<const float*>(sbase + L::VEC_OFF);

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  // heaviest CTAs first: key block 0 (pass KV) / the last query block (pass Q)
  const int blk = KV ? bx : p.nblk - 1 - bx;
  const int bh = blockIdx.y, b = bh / p.H, h = bh % p.H;
  // Grouped-query attention: query head h uses key / value head g.  Pass KV
  // runs one CTA per key / value head (on the grid row of the group's first
  // query head) and streams the query blocks of every head of the group, so
  // dK and dV sum over the group in TMEM.
  const int gs = p.H / p.Hkv, g = h / gs;
  if (KV && h % gs) return;
  const int d = p.H * HD;
  const long dq = (long)(p.H + 2 * p.Hkv) * HD;    // qkv / dqkv row width
  const int kcol = d + g * HD, vcol = d + (p.Hkv + g) * HD;
  const int row_base = b * p.T;
  const int r0 = blk * 128;  // first key (KV) or query (Q) row of this CTA
  const int nstream = (p.T + 63) / 64;
  int j0, nit, nit_h;
  if (KV) {
    j0 = r0 / 64;             // query blocks that reach key r0 or later
    nit_h = nstream - j0;     // per query head of the group
    nit = gs * nit_h;
  } else {
    j0 = 0;                   // key blocks up to the diagonal
    const int last = min(nstream - 1, (r0 + 127) / 64);
    nit = nit_h = last + 1;
  }

  if (threadIdx.x == 0) {
    mbar_init(res_full, 1);
    for (int s = 0; s < AB2_STAGES; ++s) { mbar_init(st_full(s), KV ? 2 : 1); mbar_init(st_empty(s), 1); }
    for (int i = 0; i < 2; ++i) { mbar_init(sdp_full(i), 1); mbar_init(ps_full(i), 8); }
    mbar_init(fin, 1);
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
  // TMEM columns: S buffers 0 / 64, dP buffers 128 / 192, accumulators from 256.
  // P (KV only) and dS overwrite the first 16 of each warp's 32 score columns
  // in bf16 pairs: query / key k of a 64 block sits in column 32*(k/32) + (k%32)/2.
  constexpr uint32_t T_S = 0, T_DP = 128, T_A1 = 256, T_A2 = 256 + HD;

  if (warp == 0) {
    // ------------------------------------------------ producer
    bool ok = true;
    if (lane == 0) {
      mbar_arrive_expect_tx(res_full, 2 * KCH * L::RES);
      for (int c = 0; c < KCH; ++c) {
        if (KV) {
          tma_load_2d(base + L::RES_A + c * L::RES, &p.qkv128, kcol + 64 * c, row_base + r0, res_full);
          tma_load_2d(base + L::RES_B + c * L::RES, &p.qkv128, vcol + 64 * c, row_base + r0, res_full);
        } else {
          tma_load_2d(base + L::RES_A + c * L::RES, &p.qkv128, h * HD + 64 * c, row_base + r0, res_full);
          tma_load_2d(base + L::RES_B + c * L::RES, &p.do128, h * HD + 64 * c, row_base + r0, res_full);
        }
      }
    }
    // (jj, hq): streamed block index within its query head, and that head
    // (pass KV walks the heads of the group one after another)
    for (int it = 0, jj = 0, hq = KV ? g * gs : h; it < nit && ok; ++it) {
      const int s = it % AB2_STAGES;
      if (!mbar_wait(st_empty(s), ((it / AB2_STAGES) & 1) ^ 1u, abort_flag)) { ok = false; break; }
      const int c0 = (j0 + jj) * 64;                   // first streamed row of this block
      const uint32_t sb = base + L::ST_OFF + s * L::STAGE;
      if (lane == 0) {
        mbar_arrive_expect_tx(st_full(s), L::STAGE);
        for (int c = 0; c < KCH; ++c) {
          if (KV) {
            tma_load_2d(sb + c * L::STR, &p.qkv64, hq * HD + 64 * c, row_base + c0, st_full(s));
            tma_load_2d(sb + (KCH + c) * L::STR, &p.do64, hq * HD + 64 * c, row_base + c0, st_full(s));
          } else {
            tma_load_2d(sb + c * L::STR, &p.qkv64, kcol + 64 * c, row_base + c0, st_full(s));
            tma_load_2d(sb + (KCH + c) * L::STR, &p.qkv64, vcol + 64 * c, row_base + c0, st_full(s));
          }
        }
      }
      if (KV) {
        // lse and D of the block's 64 queries (zero beyond the sequence)
        float* v = reinterpret_cast<float*>(sbase + L::VEC_OFF + s * 512);
        for (int i = lane; i < 64; i += 32) {
          const int t = c0 + i;
          const long bq = (long)b * p.H + hq;
          v[i] = t < p.T ? p.lse[bq * p.T + t] : 0.f;
          v[64 + i] = t < p.T ? p.dvec[bq * p.T + t] : 0.f;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(st_full(s));
      }
      __syncwarp();
      if (++jj == nit_h) { jj = 0; ++hq; }
    }
    if (!ok && lane == 0) set_dev_err(p.err, DEV_ERR_TIMEOUT);
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    bool ok = true, issued = false;
    if (lane == 0) {
      const uint32_t id_s = make_idesc_bf16(0, 0, 128, 64);    // S, dP: both K-major, N = 64
      const uint32_t id_acc = make_idesc_bf16(0, 1, 128, HD);  // accumulate: A K-major, B MN-major
      ok = mbar_wait(res_full, 0, abort_flag);
      for (int it = 0; it <= nit && ok; ++it) {
        if (it < nit) {
          const int bb = it & 1, s = it % AB2_STAGES;
          // (buffer bb was last read by the accumulating MMAs of block it-2, issued
          //  earlier by this thread: the tensor pipe runs them in order)
          if (!mbar_wait(st_full(s), (it / AB2_STAGES) & 1, abort_flag)) { ok = false; break; }
          tc_fence_after();
          const uint32_t sb = base + L::ST_OFF + s * L::STAGE;
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk) {
            const uint32_t oa = (kk >> 2) * L::RES + (kk & 3) * 32, ob = (kk >> 2) * L::STR + (kk & 3) * 32;
            tc_mma(tmem + T_S + 64 * bb, smem_desc(base + L::RES_A + oa, 16, 1024), smem_desc(sb + ob, 16, 1024),
                   id_s, kk > 0);
          }
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk) {
            const uint32_t oa = (kk >> 2) * L::RES + (kk & 3) * 32, ob = (kk >> 2) * L::STR + (kk & 3) * 32;
            tc_mma(tmem + T_DP + 64 * bb, smem_desc(base + L::RES_B + oa, 16, 1024),
                   smem_desc(sb + KCH * L::STR + ob, 16, 1024), id_s, kk > 0);
          }
          tc_commit(sdp_full(bb));
          issued = true;
        }
        if (it >= 1) {
          const int jt = it - 1, bj = jt & 1, sj = jt % AB2_STAGES;
          if (!mbar_wait(ps_full(bj), (jt >> 1) & 1, abort_flag)) { ok = false; break; }
          tc_fence_after();
          const uint32_t sb = base + L::ST_OFF + sj * L::STAGE;
#pragma unroll
          for (int kk = 0; kk < 64 / 16; ++kk) {
            const uint32_t acol = 64 * bj + (kk >> 1) * 32 + (kk & 1) * 8;  // 16 k values in 8 columns
            if (KV) {
              // dV += P^T dO, dK += dS^T Q   (B: the streamed [64 q][hd] tiles read MN-major)
              tc_mma_ts(tmem + T_A1, tmem + T_S + acol, smem_desc(sb + KCH * L::STR + kk * 2048, L::STR, 1024), id_acc,
                        (jt > 0 || kk > 0));
              tc_mma_ts(tmem + T_A2, tmem + T_DP + acol, smem_desc(sb + kk * 2048, L::STR, 1024), id_acc,
                        (jt > 0 || kk > 0));
            } else {
              // dQ += dS K   (B: the streamed [64 keys][hd] tile read MN-major)
              tc_mma_ts(tmem + T_A1, tmem + T_DP + acol, smem_desc(sb + kk * 2048, L::STR, 1024), id_acc,
                        (jt > 0 || kk > 0));
            }
          }
          tc_commit(st_empty(sj));
        }
      }
      if (ok) {
        tc_commit(fin);
      } else {
        set_dev_err(p.err, DEV_ERR_TIMEOUT);
        if (issued) {
          tc_commit(drain);
          const uint64_t t0 = global_timer_ns();
          while (!mbar_try_wait(drain, 0) && global_timer_ns() - t0 < kWaitNs) {}
        }
        *abort_flag = 1;
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------ elementwise (two warps per lane quadrant)
    const int q4 = warp & 3, half = (warp - 2) >> 2;
    const int r = q4 * 32 + lane;  // TMEM lane = row inside the 128-row block
    const int row = r0 + r;        // key (KV) or query (Q) position
    const uint32_t lane_addr = tmem + ((uint32_t)(q4 * 32) << 16);
    float lse_r = 0.f, d_r = 0.f;
    if (!KV && row < p.T) {
      lse_r = p.lse[(long)bh * p.T + row];
      d_r = p.dvec[(long)bh * p.T + row];
    }
    bool ok = true;
    for (int it = 0, jj = -1; it < nit; ++it) {
      if (++jj == nit_h) jj = 0;  // streamed block index within its query head
      const int bb = it & 1, s = it % AB2_STAGES;
      const int c0 = (j0 + jj) * 64 + 32 * half;  // first streamed position of this warp's 32 columns
      // sdp_full(it) also covers the accumulating MMAs of block it-2, the last
      // readers of the P / dS columns of buffer bb
      if (!mbar_wait(sdp_full(bb), (it >> 1) & 1, abort_flag)) { ok = false; break; }
      if (KV && !mbar_wait(st_full(s), (it / AB2_STAGES) & 1, abort_flag)) { ok = false; break; }
      tc_fence_after();
      uint32_t sr[32], dr[32];
      TMEM_LD32(lane_addr + T_S + 64 * bb + 32 * half, sr);
      TMEM_LD32(lane_addr + T_DP + 64 * bb + 32 * half, dr);
      tmem_wait_ld();
      const float* vl = vec_base + s * 128 + 32 * half;  // KV: lse / D of this warp's 32 queries
      float pv[32], dv[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const int c = c0 + i;
        float lse, dd;
        bool masked;
        if (KV) {
          lse = vl[i];
          dd = vl[64 + i];
          masked = c >= p.T || row >= p.T || c < row;   // query c, key row
        } else {
          lse = lse_r;
          dd = d_r;
          masked = c >= p.T || row >= p.T || c > row;   // key c, query row
        }
        const float pr = masked ? 0.f : ex2_approx(__uint_as_float(sr[i]) * p.scale_log2 - lse);
        pv[i] = pr;
        dv[i] = pr * (__uint_as_float(dr[i]) - dd);
      }
      // bf16 pairs back into this warp's own score columns (A operands of the accumulating MMAs)
      uint32_t pw[16], dw[16];
#pragma unroll
      for (int w = 0; w < 16; ++w) {
        __nv_bfloat162 a = __floats2bfloat162_rn(pv[2 * w], pv[2 * w + 1]);
        __nv_bfloat162 g = __floats2bfloat162_rn(dv[2 * w], dv[2 * w + 1]);
        pw[w] = *reinterpret_cast<uint32_t*>(&a);
        dw[w] = *reinterpret_cast<uint32_t*>(&g);
      }
      if (KV) TMEM_ST16(lane_addr + T_S + 64 * bb + 32 * half, pw);
      TMEM_ST16(lane_addr + T_DP + 64 * bb + 32 * half, dw);
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(ps_full(bb));
    }
    // ------------------------------------------------ results: dK (scaled) and dV, or dQ (scaled)
    if (ok && mbar_wait(fin, 0, abort_flag)) {
      tc_fence_after();
      bf16* out1 = p.dqkv + ((long)row_base + row) * dq + (KV ? vcol : h * HD);  // dV or dQ
      bf16* out2 = p.dqkv + ((long)row_base + row) * dq + kcol;                  // dK
      const float s1 = KV ? 1.f : p.scale;
#pragma unroll
      for (int c = half * (HD / 2); c < (half + 1) * (HD / 2); c += 32) {
        uint32_t a[32], k[32];
        TMEM_LD32(lane_addr + T_A1 + c, a);
        if (KV) TMEM_LD32(lane_addr + T_A2 + c, k);
        tmem_wait_ld();
        if (row < p.T) {
#pragma unroll
          for (int i = 0; i < 32; i += 8) {
            uint4 v;
            __nv_bfloat162 y0 = __floats2bfloat162_rn(__uint_as_float(a[i]) * s1, __uint_as_float(a[i + 1]) * s1);
            __nv_bfloat162 y1 = __floats2bfloat162_rn(__uint_as_float(a[i + 2]) * s1, __uint_as_float(a[i + 3]) * s1);
            __nv_bfloat162 y2 = __floats2bfloat162_rn(__uint_as_float(a[i + 4]) * s1, __uint_as_float(a[i + 5]) * s1);
            __nv_bfloat162 y3 = __floats2bfloat162_rn(__uint_as_float(a[i + 6]) * s1, __uint_as_float(a[i + 7]) * s1);
            v.x = *reinterpret_cast<uint32_t*>(&y0); v.y = *reinterpret_cast<uint32_t*>(&y1);
            v.z = *reinterpret_cast<uint32_t*>(&y2); v.w = *reinterpret_cast<uint32_t*>(&y3);
            *reinterpret_cast<uint4*>(out1 + c + i) = v;
            if (KV) {
              uint4 w;
              __nv_bfloat162 x0 = __floats2bfloat162_rn(__uint_as_float(k[i]) * p.scale, __uint_as_float(k[i + 1]) * p.scale);
              __nv_bfloat162 x1 = __floats2bfloat162_rn(__uint_as_float(k[i + 2]) * p.scale, __uint_as_float(k[i + 3]) * p.scale);
              __nv_bfloat162 x2 = __floats2bfloat162_rn(__uint_as_float(k[i + 4]) * p.scale, __uint_as_float(k[i + 5]) * p.scale);
              __nv_bfloat162 x3 = __floats2bfloat162_rn(__uint_as_float(k[i + 6]) * p.scale, __uint_as_float(k[i + 7]) * p.scale);
              w.x = *reinterpret_cast<uint32_t*>(&x0); w.y = *reinterpret_cast<uint32_t*>(&x1);
              w.z = *reinterpret_cast<uint32_t*>(&x2); w.w = *reinterpret_cast<uint32_t*>(&x3);
              *reinterpret_cast<uint4*>(out2 + c + i) = w;
            }
          }
        }
      }
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

// Both passes in one launch (they read the same inputs and write disjoint
// columns of dqkv): even x runs pass KV, odd x pass Q, so the heaviest blocks of
// both go first and the two passes share one wave tail instead of two.
template <int HD>
__global__ void __launch_bounds__(AB2_THREADS, 1) attn_bwd2_kernel(const __grid_constant__ AttnBwd2Params p) {
  if (blockIdx.x & 1) attn_bwd2_body<HD, false>(p, (int)(blockIdx.x >> 1));
  else attn_bwd2_body<HD, true>(p, (int)(blockIdx.x >> 1));
}

template <int HD>
int launch_bwd2(const AttnBwd2Params& p, int BH, cudaStream_t s, std::string* msg) {
  constexpr int smem = Bwd2Smem<HD, true>::TOTAL > Bwd2Smem<HD, false>::TOTAL ? Bwd2Smem<HD, true>::TOTAL
                                                                               : Bwd2Smem<HD, false>::TOTAL;
  static_assert(smem <= 232448, "attention backward shared memory");
  static bool set = false;
  if (!set) {
    if (cudaFuncSetAttribute(attn_bwd2_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess) {
      if (msg) *msg = "attention backward smem attribute failed";
      return 4;
    }
    set = true;
  }
  dim3 grid(2 * p.nblk, BH);
  attn_bwd2_kernel<HD><<<grid, AB2_THREADS, smem, s>>>(p);
  count_launches(1);
  return 0;
}

}  // namespace

int attn_bwd2_tc(int B, int T, int H, int Hkv, int hd, const void* qkv, const void* dctx, const float* lse,
                 const float* dvec, void* dqkv, int* dev_err, cudaStream_t s, std::string* msg) {
  if (B <= 0 || T <= 0) return 0;
  if (hd != 64 && hd != 128) { if (msg) *msg = "tcgen05 attention needs head_dim 64 or 128"; return 6; }
  if (Hkv <= 0 || H % Hkv) { if (msg) *msg = "heads must be a multiple of the key/value heads"; return 1; }
  AttnBwd2Params p;
  memset(&p, 0, sizeof(p));
  const long d = (long)H * hd, dq = (long)(H + 2 * Hkv) * hd;
  const unsigned long long rows = (unsigned long long)B * T;
  if (!tma_map_2d(&p.qkv128, qkv, 0, dq, rows, dq, 64, 128, 1, msg) ||
      !tma_map_2d(&p.qkv64, qkv, 0, dq, rows, dq, 64, 64, 1, msg) ||
      !tma_map_2d(&p.do128, dctx, 0, d, rows, d, 64, 128, 1, msg) ||
      !tma_map_2d(&p.do64, dctx, 0, d, rows, d, 64, 64, 1, msg))
    return 1;
  p.lse = lse;
  p.dvec = dvec;
  p.dqkv = reinterpret_cast<bf16*>(dqkv);
  p.T = T;
  p.H = H;
  p.Hkv = Hkv;
  p.nblk = (T + 127) / 128;
  p.scale = 1.f / sqrtf((float)hd);
  p.scale_log2 = 1.4426950408889634f / sqrtf((float)hd);
  p.err = dev_err;
  int r;
  if (hd == 64) r = launch_bwd2<64>(p, B * H, s, msg);
  else r = launch_bwd2<128>(p, B * H, s, msg);
  if (r) return r;
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) { if (msg) *msg = std::string("attention backward launch: ") + cudaGetErrorString(e); return 4; }
  return 0;
}

}  // namespace fal
