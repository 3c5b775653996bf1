// tcgen05 / TMEM GEMM fed by TMA, for every bf16 contraction of the path
// (QKV projection, MLP up-projection + GELU, the fused [ctx | g] x [W_o ; W_down]
// residual GEMM, LM head, and all data/weight-gradient GEMMs of the backward).
//
// Design (sm_103a, one CTA per SM, persistent over output tiles):
//   warp 0      TMA producer: 128x64 A tile + 256x64 B tile per stage (4 stages),
//               128-byte swizzle, K-major or MN-major operands.
//   warp 1      allocates 512 TMEM columns (two 128x256 fp32 accumulators) and
//               issues tcgen05.mma.cta_group::1.kind::f16 (M=128, N=256, K=16),
//               committing each stage back to the producer.
//   warps 2..9  epilogue (two warps per TMEM lane quadrant, each owning half of
//               the 256 columns): tcgen05.ld 32 lanes x 32 columns, a swizzled
//               shared-memory transpose so that every global access of the
//               epilogue (bias, dGELU input, residual) is row-coalesced, then
//               bias / GELU / dGELU / residual in fp32; outputs are written back
//               into the warp's buffer as a dense tile and leave with one TMA
//               bulk tensor store (reduce-add for fp32 accumulation) per output;
//               the second accumulator lets tile t+1's main loop overlap tile
//               t's epilogue.
// Every mbarrier wait is bounded (about one second): on expiry the CTA records
// DEV_ERR_TIMEOUT in the device error word, drains its in-flight copies and
// MMAs, frees TMEM and returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <cstring>
#include <functional>
#include <map>
#include <mutex>
#include <queue>
#include <utility>
#include <vector>

#include "gemm_epi.cuh"
#include "tc_ptx.cuh"

namespace fal {

namespace {

using namespace ptx;

constexpr int TC_BM = 128, TC_BN = 256, TC_BK = 64, TC_STAGES = 4;
constexpr int TC_A_BYTES = TC_BM * TC_BK * 2;   // 16 KB
constexpr int TC_B_BYTES = TC_BN * TC_BK * 2;   // 32 KB
constexpr int TC_STAGE_BYTES = TC_A_BYTES + TC_B_BYTES;
constexpr int TC_MN_CHUNK_BYTES = 64 * TC_BK * 2;  // one 64-wide MN chunk of an MN-major tile
constexpr int TC_BAR_BYTES = 256;
constexpr int TC_EPI_WARPS = 8;
constexpr int TC_EPI_STAGE_BYTES = 32 * 32 * 4;  // one 32x32 fp32 chunk per epilogue warp
constexpr int TC_SMEM = TC_STAGES * TC_STAGE_BYTES + TC_EPI_WARPS * TC_EPI_STAGE_BYTES + 1024 + TC_BAR_BYTES;
constexpr int TC_THREADS = 64 + 32 * TC_EPI_WARPS;

struct TcGroup {
  int M, N, m_tiles, n_tiles, tile_start, nseg;
  // Tile order: band_m = 0 walks m fastest over the whole group (the B panel of
  // one column of tiles is read once; A must stay in L2).  band_m > 0 walks
  // bands of band_m row tiles, each band across all column tiles, so that the
  // CTAs in flight share their A rows and B stays in L2 (A is read once).
  int band_m;
  int kb[2];
  int amap[2], bmap[2];
  int a_mn, b_mn;
  uint32_t idesc;
  // Output path: TMA bulk tensor stores of 32x32 chunks staged in shared
  // memory (out_tma), else per-thread stores.  omap / omap2: maps of `out`
  // and of the GELU output; out_accum: TMA reduce-add into fp32 `out`.
  int out_tma, out_f32, out_accum, omap, omap2;
  int kind;  // EpiKind specialisation used by the epilogue
  EpiParams epi;
};

constexpr int kMaxMaps = 20;  // operand maps (2 per K segment) and output maps (up to 2) of all groups
struct TcParams {
  CUtensorMap maps[kMaxMaps];
  TcGroup grp[kMaxGemmGroups];
  int ngroups, total_tiles;
  int* err;
  // Tile lists per unit (CTA, or cluster of two): sched[u] .. sched[u + 1] index
  // the tiles of unit u in sched[nunits + 1 + ...].  Null: round robin, unit u
  // takes tiles u, u + nunits, ...
  const int* sched;
};

// The i-th tile of a unit's sequence, or -1 when the unit is done.
__device__ __forceinline__ int tile_at(const TcParams& p, int unit, int nunits, int i) {
  if (p.sched) {
    const int b = __ldg(p.sched + unit), e = __ldg(p.sched + unit + 1);
    return i < e - b ? __ldg(p.sched + nunits + 1 + b + i) : -1;
  }
  const int t = unit + i * nunits;
  return t < p.total_tiles ? t : -1;
}


// One epilogue warp's 32x32 accumulator chunk (rows row0.., columns col0..),
// already loaded from TMEM into r (lane = row).  When every output of the group
// is a TMA target (the usual case) the lane keeps its row: bias / GELU / dGELU /
// residual are applied in registers and the row is written into the warp's
// 4 KB buffer in the swizzled layout of the output's tensor map (64-byte rows
// in bf16, 128-byte rows in fp32, conflict-free), then one TMA bulk tensor store
// (reduce-add for fp32 accumulation) per output leaves the SM.  Otherwise the
// chunk is transposed through the buffer and stored with coalesced per-thread
// stores.  KIND fixes at compile time which inputs the epilogue reads;
// everything the chunk needs arrives by value so that it stays in registers.
struct EpiOut {
  int M, N, out_tma, out_f32, out_accum, omap, omap2, gelu;
};

// EPI_ADAMW chunk: the gradient tile is transposed through the warp's buffer so
// that each row segment is read and written with coalesced 16-byte accesses:
// gradient store, then the AdamW update of the weight (master, moments, bf16
// copy).  The optimizer's operands are read from the parameter block once per
// chunk.
__device__ __forceinline__ void epi_adamw_chunk(const EpiParams* ep, int M, int N, float4* stage, int lane, int row0,
                                                int col0, const uint32_t* r) {
#pragma unroll
  for (int j = 0; j < 8; ++j)
    stage[lane * 8 + (j ^ (lane & 7))] = make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                                                     __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3]));
  __syncwarp();
  float* const g = reinterpret_cast<float*>(ep->out);
  float* const pp = ep->opt_p;
  float* const mm = ep->opt_m;
  float* const vv = ep->opt_v;
  bf16* const sh = reinterpret_cast<bf16*>(ep->opt_sh);
  const long ld = ep->ldo;
  const float lr = ep->opt_lr, b1 = ep->opt_b1, b2 = ep->opt_b2, eps = ep->opt_eps, wd = ep->opt_wd;
  const float rbc1 = ep->opt_rbc1, rbc2 = ep->opt_rbc2;
  const int rb = lane >> 3, ch = lane & 7;
  if (row0 + 32 <= M && col0 + 32 <= N) {
    // Interior chunk: every lane first asks L2 for its row's 128-byte segments
    // of the three optimizer arrays (the whole 32x32 chunk is then in flight
    // at once, at no register cost), then two row groups at a time are loaded,
    // updated and stored.
    {
      const long o = (long)(row0 + lane) * ld + col0;
      asm volatile("prefetch.global.L2 [%0];" ::"l"(pp + o));
      asm volatile("prefetch.global.L2 [%0];" ::"l"(mm + o));
      asm volatile("prefetch.global.L2 [%0];" ::"l"(vv + o));
    }
#pragma unroll 1
    for (int h0 = 0; h0 < 8; h0 += 2) {
      float4 P[2], Mv[2], Vv[2];
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const long o = (long)(row0 + (h0 + j) * 4 + rb) * ld + col0 + ch * 4;
        P[j] = load4(pp + o); Mv[j] = load4(mm + o); Vv[j] = load4(vv + o);
      }
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const int rr = (h0 + j) * 4 + rb;
        const long o = (long)(row0 + rr) * ld + col0 + ch * 4;
        const float4 v4 = stage[rr * 8 + (ch ^ (rr & 7))];
        store4(g + o, v4);
        adamw_elem(P[j].x, Mv[j].x, Vv[j].x, v4.x, lr, b1, b2, eps, wd, rbc1, rbc2);
        adamw_elem(P[j].y, Mv[j].y, Vv[j].y, v4.y, lr, b1, b2, eps, wd, rbc1, rbc2);
        adamw_elem(P[j].z, Mv[j].z, Vv[j].z, v4.z, lr, b1, b2, eps, wd, rbc1, rbc2);
        adamw_elem(P[j].w, Mv[j].w, Vv[j].w, v4.w, lr, b1, b2, eps, wd, rbc1, rbc2);
        store4(pp + o, P[j]); store4(mm + o, Mv[j]); store4(vv + o, Vv[j]);
        if (sh) store4(sh + o, P[j]);
      }
    }
    __syncwarp();
    return;
  }
#pragma unroll 1
  for (int it = 0; it < 8; ++it) {
    const int rr = it * 4 + rb;
    const int row = row0 + rr, c = col0 + ch * 4;
    if (row >= M || c >= N) continue;
    const float4 v4 = stage[rr * 8 + (ch ^ (rr & 7))];
    const long o = (long)row * ld + c;
    if (c + 4 <= N) {
      store4(g + o, v4);
      float4 p = load4(pp + o), m = load4(mm + o), v = load4(vv + o);
      adamw_elem(p.x, m.x, v.x, v4.x, lr, b1, b2, eps, wd, rbc1, rbc2);
      adamw_elem(p.y, m.y, v.y, v4.y, lr, b1, b2, eps, wd, rbc1, rbc2);
      adamw_elem(p.z, m.z, v.z, v4.z, lr, b1, b2, eps, wd, rbc1, rbc2);
      adamw_elem(p.w, m.w, v.w, v4.w, lr, b1, b2, eps, wd, rbc1, rbc2);
      store4(pp + o, p); store4(mm + o, m); store4(vv + o, v);
      if (sh) store4(sh + o, p);
    } else {
      const float gv[4] = {v4.x, v4.y, v4.z, v4.w};
      for (int j = 0; j < 4 && c + j < N; ++j) {
        g[o + j] = gv[j];
        float p = pp[o + j], m = mm[o + j], v = vv[o + j];
        adamw_elem(p, m, v, gv[j], lr, b1, b2, eps, wd, rbc1, rbc2);
        pp[o + j] = p; mm[o + j] = m; vv[o + j] = v;
        if (sh) sh[o + j] = __float2bfloat16_rn(p);
      }
    }
  }
  __syncwarp();
}

template <typename act_t, int KIND>
__device__ __forceinline__ void epi_chunk(const TcParams& p, const EpiParams* ep, const EpiIn q, const EpiOut o,
                                          float4* stage, uint32_t stage_s, int lane, int row0, int col0,
                                          const uint32_t* r) {
  // Every path below writes this buffer: the TMA stores of earlier chunks must
  // have read it (a weight-gradient tile with the AdamW epilogue may follow a
  // data-gradient tile in the same warp when the data gradient is the deeper one).
  if (lane == 0) bulk_wait_read_all();
  __syncwarp();
  if constexpr (KIND == EK_ADAMW) {
    epi_adamw_chunk(ep, o.M, o.N, stage, lane, row0, col0, r);
    return;
  }
  if (!o.out_tma) {
#pragma unroll
    for (int j = 0; j < 8; ++j)
      stage[lane * 8 + (j ^ (lane & 7))] = make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                                                       __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3]));
    __syncwarp();
    const int rb = lane >> 3, ch = lane & 7;
#pragma unroll
    for (int it = 0; it < 8; ++it) {
      const int rr = it * 4 + rb;
      float4 v4 = stage[rr * 8 + (ch ^ (rr & 7))];
      float v[4] = {v4.x, v4.y, v4.z, v4.w};
      epi_row<act_t, 4>(*ep, o.M, o.N, row0 + rr, col0 + ch * 4, v);
    }
    __syncwarp();
    return;
  }
  if constexpr (KIND == EK_DGELU && sizeof(act_t) == 2) {
    if (!o.out_f32 && (q.ldx & 7) == 0 && row0 + 32 <= o.M && col0 + 32 <= o.N) {
      // Interior bf16 chunk: the pre-activation h is read with coalesced
      // 16-byte loads (four lanes per 64-byte row segment, eight rows per
      // load) into the upper half of the warp's buffer, in the swizzled layout
      // of the output, from which each lane then takes its own row.
      uint8_t* sb = reinterpret_cast<uint8_t*>(stage);
      const act_t* aux = reinterpret_cast<const act_t*>(q.aux);
      uint4 hv[4];
#pragma unroll
      for (int it = 0; it < 4; ++it) {
        const int rr = it * 8 + (lane >> 2);
        hv[it] = *reinterpret_cast<const uint4*>(aux + (long)(row0 + rr) * q.ldx + col0 + (lane & 3) * 8);
      }
#pragma unroll
      for (int it = 0; it < 4; ++it) {
        const int rr = it * 8 + (lane >> 2), u = lane & 3;
        *reinterpret_cast<uint4*>(sb + 2048 + rr * 64 + ((u ^ ((rr >> 1) & 3)) << 4)) = hv[it];
      }
      __syncwarp();
      const int sw = (lane >> 1) & 3;
#pragma unroll
      for (int g = 0; g < 4; ++g) {
        const uint4 hp = *reinterpret_cast<const uint4*>(sb + 2048 + lane * 64 + ((g ^ sw) << 4));
        const uint32_t hw[4] = {hp.x, hp.y, hp.z, hp.w};
        uint32_t ow[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float2 h2 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&hw[j]));
          const float a = __uint_as_float(r[8 * g + 2 * j]) * epi_gelu_grad<act_t>(h2.x);
          const float b = __uint_as_float(r[8 * g + 2 * j + 1]) * epi_gelu_grad<act_t>(h2.y);
          __nv_bfloat162 t = __floats2bfloat162_rn(a, b);
          ow[j] = *reinterpret_cast<uint32_t*>(&t);
        }
        *reinterpret_cast<uint4*>(sb + lane * 64 + ((g ^ sw) << 4)) = make_uint4(ow[0], ow[1], ow[2], ow[3]);
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        tma_store_2d(&p.maps[o.omap], stage_s, col0, row0);
        bulk_commit();
      }
      return;
    }
  }
  const int row = row0 + lane;
  float4 y[8];
  if constexpr (KIND == EK_CEGRAD) {
    // (softmax - one-hot) / rows of this lane's row, zero outside M x N
    float lse = 0.f;
    int t = -1;
    if (row < o.M) { lse = ep->ce_lse[row]; t = ep->ce_tgt[row] - ep->ce_v0; }
    const float sc = ep->ce_scale;
#pragma unroll
    for (int g = 0; g < 8; ++g) {
      float v[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int c = col0 + 4 * g + j;
        v[j] = (row < o.M && c < o.N) ? ce_grad1(__uint_as_float(r[4 * g + j]), lse, t, c, sc) : 0.f;
      }
      y[g] = make_float4(v[0], v[1], v[2], v[3]);
    }
  } else {
#pragma unroll
    for (int g = 0; g < 8; ++g)
      y[g] = epi_value4<act_t, KIND>(q, o.M, o.N, row, col0 + 4 * g,
                                     make_float4(__uint_as_float(r[4 * g]), __uint_as_float(r[4 * g + 1]),
                                                 __uint_as_float(r[4 * g + 2]), __uint_as_float(r[4 * g + 3])));
  }
  uint8_t* sb = reinterpret_cast<uint8_t*>(stage);
  const bool gelu = (KIND & EK_GELU) && (KIND != EK_ANY || o.gelu);
  if (o.out_f32) {
#pragma unroll
    for (int g = 0; g < 8; ++g) *reinterpret_cast<float4*>(sb + lane * 128 + ((g ^ (lane & 7)) << 4)) = y[g];
  } else {
    const int sw = (lane >> 1) & 3;
#pragma unroll
    for (int g = 0; g < 4; ++g) {
      uint4 pk;
      __nv_bfloat162 t0 = __floats2bfloat162_rn(y[2 * g].x, y[2 * g].y), t1 = __floats2bfloat162_rn(y[2 * g].z, y[2 * g].w);
      __nv_bfloat162 t2 = __floats2bfloat162_rn(y[2 * g + 1].x, y[2 * g + 1].y);
      __nv_bfloat162 t3 = __floats2bfloat162_rn(y[2 * g + 1].z, y[2 * g + 1].w);
      pk.x = *reinterpret_cast<uint32_t*>(&t0); pk.y = *reinterpret_cast<uint32_t*>(&t1);
      pk.z = *reinterpret_cast<uint32_t*>(&t2); pk.w = *reinterpret_cast<uint32_t*>(&t3);
      *reinterpret_cast<uint4*>(sb + lane * 64 + ((g ^ sw) << 4)) = pk;
    }
    if (gelu) {
#pragma unroll
      for (int g = 0; g < 4; ++g) {
        uint4 pk;
        __nv_bfloat162 t0 = __floats2bfloat162_rn(epi_gelu<act_t>(y[2 * g].x), epi_gelu<act_t>(y[2 * g].y));
        __nv_bfloat162 t1 = __floats2bfloat162_rn(epi_gelu<act_t>(y[2 * g].z), epi_gelu<act_t>(y[2 * g].w));
        __nv_bfloat162 t2 = __floats2bfloat162_rn(epi_gelu<act_t>(y[2 * g + 1].x), epi_gelu<act_t>(y[2 * g + 1].y));
        __nv_bfloat162 t3 = __floats2bfloat162_rn(epi_gelu<act_t>(y[2 * g + 1].z), epi_gelu<act_t>(y[2 * g + 1].w));
        pk.x = *reinterpret_cast<uint32_t*>(&t0); pk.y = *reinterpret_cast<uint32_t*>(&t1);
        pk.z = *reinterpret_cast<uint32_t*>(&t2); pk.w = *reinterpret_cast<uint32_t*>(&t3);
        *reinterpret_cast<uint4*>(sb + 2048 + lane * 64 + ((g ^ sw) << 4)) = pk;
      }
    }
  }
  fence_proxy_async_smem();
  __syncwarp();
  if (lane == 0) {
    if (o.out_accum) tma_reduce_add_2d(&p.maps[o.omap], stage_s, col0, row0);
    else tma_store_2d(&p.maps[o.omap], stage_s, col0, row0);
    if (gelu) tma_store_2d(&p.maps[o.omap2], stage_s + 2048, col0, row0);
    bulk_commit();
  }
}

// Dot product of this lane's 32 output values (rounded to the activation type,
// as stored) with the same 32 columns of rd_src: one head's share of D.
template <typename act_t>
__device__ __forceinline__ float rowdot_chunk(const EpiParams* ep, int M, int row, int col0, const uint32_t* r) {
  if (row >= M) return 0.f;
  const act_t* src = reinterpret_cast<const act_t*>(ep->rd_src) + (long)row * ep->rd_ld + col0;
  float s = 0.f;
#pragma unroll
  for (int j = 0; j < 32; j += 4) {
    const float4 o = load4(src + j);
    s += to_f(from_f<act_t>(__uint_as_float(r[j]))) * o.x + to_f(from_f<act_t>(__uint_as_float(r[j + 1]))) * o.y +
         to_f(from_f<act_t>(__uint_as_float(r[j + 2]))) * o.z + to_f(from_f<act_t>(__uint_as_float(r[j + 3]))) * o.w;
  }
  return s;
}
// The same for a whole interior chunk (rows row0.., all in range): the 32 x 32
// block of rd_src is read with coalesced 16-byte loads into the upper half of
// the warp's buffer (swizzled like the output rows) and each lane takes its row
// from there.  The buffer must be free of pending TMA reads.
__device__ __forceinline__ float rowdot_chunk_staged(const EpiParams* ep, uint8_t* sb, int lane, int row0, int col0,
                                                     const uint32_t* r) {
  const bf16* src = reinterpret_cast<const bf16*>(ep->rd_src);
  uint4 v[4];
#pragma unroll
  for (int it = 0; it < 4; ++it) {
    const int rr = it * 8 + (lane >> 2);
    v[it] = *reinterpret_cast<const uint4*>(src + (long)(row0 + rr) * ep->rd_ld + col0 + (lane & 3) * 8);
  }
#pragma unroll
  for (int it = 0; it < 4; ++it) {
    const int rr = it * 8 + (lane >> 2), u = lane & 3;
    *reinterpret_cast<uint4*>(sb + 2048 + rr * 64 + ((u ^ ((rr >> 1) & 3)) << 4)) = v[it];
  }
  __syncwarp();
  const int sw = (lane >> 1) & 3;
  float s = 0.f;
#pragma unroll
  for (int g = 0; g < 4; ++g) {
    const uint4 op = *reinterpret_cast<const uint4*>(sb + 2048 + lane * 64 + ((g ^ sw) << 4));
    const uint32_t ow[4] = {op.x, op.y, op.z, op.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 o2 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&ow[j]));
      s += to_f(from_f<bf16>(__uint_as_float(r[8 * g + 2 * j]))) * o2.x +
           to_f(from_f<bf16>(__uint_as_float(r[8 * g + 2 * j + 1]))) * o2.y;
    }
  }
  __syncwarp();
  return s;
}

// Row-dot share of one chunk, staged through the warp's buffer when it can be.
template <typename act_t>
__device__ __forceinline__ float rowdot_any(const EpiParams* ep, int M, int N, float4* stage, int lane, int row0,
                                           int col0, const uint32_t* r) {
  if constexpr (sizeof(act_t) == 2) {
    if (row0 + 32 <= M && col0 + 32 <= N) {
      if (lane == 0) bulk_wait_read_all();
      __syncwarp();
      return rowdot_chunk_staged(ep, reinterpret_cast<uint8_t*>(stage), lane, row0, col0, r);
    }
  }
  return rowdot_chunk<act_t>(ep, M, row0 + lane, col0, r);
}

__device__ __forceinline__ void rowdot_store(const EpiParams* ep, int M, int row, int col_end, float s) {
  if (row >= M) return;
  const int T = ep->rd_T, h = (col_end - 1) / ep->rd_hd;
  ep->rd_out[((long)(row / T) * ep->rd_H + h) * T + row % T] = s;
}

// EPI_CE_STATS: folds one 32-column chunk of this lane's row (the columns below
// N) into the running maximum m and sum s of exp(x - m), and stores the logit of
// the row's target t (a column of this group) when the chunk holds it.
__device__ __forceinline__ void ce_stats_chunk(const EpiParams* ep, int M, int N, int row, int col0, int t,
                                               const uint32_t* r, float& m, float& s) {
  if (row >= M) return;
  const int nv = N - col0;  // >= 1: chunks at or beyond N are skipped
  float cm = m;
#pragma unroll
  for (int j = 0; j < 32; ++j)
    if (j < nv) cm = fmaxf(cm, __uint_as_float(r[j]));
  float acc = s * __expf(m - cm);  // 0 on the first chunk (s = 0, m = -inf)
#pragma unroll
  for (int j = 0; j < 32; ++j)
    if (j < nv) acc += __expf(__uint_as_float(r[j]) - cm);
  m = cm;
  s = acc;
  const int tc = t - col0;
  if (tc >= 0 && tc < 32 && tc < nv) {
    float v = 0.f;
#pragma unroll
    for (int j = 0; j < 32; ++j) v = (j == tc) ? __uint_as_float(r[j]) : v;
    ep->ce_tlogit[row] = v;
  }
}

// EPI_CE_STATS over one epilogue warp's 32 x 128 piece of a tile (this lane's
// row `row`, columns col0 .. col0 + 127 at TMEM address taddr): one statistics
// pair per row for the slice.
__device__ __noinline__ void ce_stats_tile(const EpiParams* ep, int M, int N, int row, int col0, uint32_t taddr) {
  const int t = row < M ? ep->ce_tgt[row] - ep->ce_v0 : -1;
  float m = -INFINITY, s = 0.f;
  for (int c = 0; c < kCeSliceTc / 32; ++c) {
    if (col0 + c * 32 >= N) break;
    uint32_t r[32];
    TMEM_LD32(taddr + c * 32, r);
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
    ce_stats_chunk(ep, M, N, row, col0 + c * 32, t, r, m, s);
  }
  if (row < M && col0 < N) ep->ce_stats[(long)(col0 / kCeSliceTc) * ep->ce_ld + row] = make_float2(m, s);
}

// Runs one chunk with the specialisation the group was prepared for.
template <typename act_t>
__device__ __forceinline__ void epi_chunk_dispatch(int kind, const TcParams& p, const EpiParams* ep, const EpiIn q,
                                                   const EpiOut o, float4* stage, uint32_t stage_s, int lane, int row0,
                                                   int col0, const uint32_t* r) {
  switch (kind) {
    case 0: epi_chunk<act_t, 0>(p, ep, q, o, stage, stage_s, lane, row0, col0, r); break;
    case EK_BIAS: epi_chunk<act_t, EK_BIAS>(p, ep, q, o, stage, stage_s, lane, row0, col0, r); break;
    case EK_BIAS | EK_GELU: epi_chunk<act_t, EK_BIAS | EK_GELU>(p, ep, q, o, stage, stage_s, lane, row0, col0, r); break;
    case EK_DGELU: epi_chunk<act_t, EK_DGELU>(p, ep, q, o, stage, stage_s, lane, row0, col0, r); break;
    case EK_BIAS | EK_RESID: epi_chunk<act_t, EK_BIAS | EK_RESID>(p, ep, q, o, stage, stage_s, lane, row0, col0, r); break;
    case EK_BIAS | EK_BIAS2 | EK_RESID:
      epi_chunk<act_t, EK_BIAS | EK_BIAS2 | EK_RESID>(p, ep, q, o, stage, stage_s, lane, row0, col0, r); break;
    case EK_ADAMW: epi_chunk<act_t, EK_ADAMW>(p, ep, q, o, stage, stage_s, lane, row0, col0, r); break;
    case EK_CEGRAD: epi_chunk<act_t, EK_CEGRAD>(p, ep, q, o, stage, stage_s, lane, row0, col0, r); break;
    default: epi_chunk<act_t, EK_ANY>(p, ep, q, o, stage, stage_s, lane, row0, col0, r); break;
  }
}

__device__ __forceinline__ EpiOut epi_out_of(const TcGroup& G) {
  EpiOut o;
  o.M = G.M; o.N = G.N; o.out_tma = G.out_tma; o.out_f32 = G.out_f32; o.out_accum = G.out_accum;
  o.omap = G.omap; o.omap2 = G.omap2; o.gelu = G.epi.op == EPI_GELU;
  return o;
}

// Output tile (row index mt, column index nt) of a group-local tile index.
__device__ __forceinline__ void tile_mn(const TcGroup& G, int local, int& mt, int& nt) {
  if (G.band_m <= 0) {
    mt = local % G.m_tiles;
    nt = local / G.m_tiles;
    return;
  }
  const int per_band = G.band_m * G.n_tiles;
  const int band = local / per_band, r = local - band * per_band;
  const int rows = min(G.band_m, G.m_tiles - band * G.band_m);  // the last band may be short
  mt = band * G.band_m + r % rows;
  nt = r / rows;
}

// Group of a tile index: groups own consecutive tile ranges in group order.
__device__ __forceinline__ int group_of(const TcParams& p, int tile) {
  int g = 0;
#pragma unroll
  for (int k = 1; k < kMaxGemmGroups; ++k)
    if (k < p.ngroups && tile >= p.grp[k].tile_start) g = k;
  return g;
}

__device__ __forceinline__ void decode_tile(const TcParams& p, int tile, int& g, int& m0, int& n0) {
  g = group_of(p, tile);
  const TcGroup& G = p.grp[g];
  int mt, nt;
  tile_mn(G, tile - G.tile_start, mt, nt);
  m0 = mt * TC_BM;
  n0 = nt * TC_BN;
}

template <typename act_t>
__global__ void __launch_bounds__(TC_THREADS, 1) gemm_tc_kernel(const __grid_constant__ TcParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  const uint32_t epi_base = base + TC_STAGES * TC_STAGE_BYTES;
  const uint32_t bar_base = epi_base + TC_EPI_WARPS * TC_EPI_STAGE_BYTES;
  uint8_t* bar_ptr = smem_raw + (bar_base - raw);
  auto full_bar = [&](int s) { return bar_base + 8u * s; };
  auto empty_bar = [&](int s) { return bar_base + 8u * (TC_STAGES + s); };
  auto tfull_bar = [&](int b) { return bar_base + 8u * (2 * TC_STAGES + b); };
  auto tempty_bar = [&](int b) { return bar_base + 8u * (2 * TC_STAGES + 2 + b); };
  const uint32_t drain_bar = bar_base + 8u * (2 * TC_STAGES + 4);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar_ptr + 8 * (2 * TC_STAGES + 5));
  volatile uint32_t* abort_flag = reinterpret_cast<volatile uint32_t*>(bar_ptr + 8 * (2 * TC_STAGES + 5) + 4);

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int unit = (int)blockIdx.x, nunits = (int)gridDim.x;  // this CTA's tile stream
  if (threadIdx.x == 0) {
    for (int s = 0; s < TC_STAGES; ++s) { mbar_init(full_bar(s), 1); mbar_init(empty_bar(s), 1); }
    for (int b = 0; b < 2; ++b) { mbar_init(tfull_bar(b), 1); mbar_init(tempty_bar(b), TC_EPI_WARPS); }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)), "r"(512)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------ TMA producer
    int stage = 0;
    uint32_t phase = 0;
    uint32_t issued_mask = 0, issued_par = 0;
    bool ok = true;
    for (int ti = 0, tile; ok && (tile = tile_at(p, unit, nunits, ti)) >= 0; ++ti) {
      int g, m0, n0;
      decode_tile(p, tile, g, m0, n0);
      const TcGroup& G = p.grp[g];
      for (int s = 0; s < G.nseg && ok; ++s) {
        const CUtensorMap* am = &p.maps[G.amap[s]];
        const CUtensorMap* bm = &p.maps[G.bmap[s]];
        for (int kb = 0; kb < G.kb[s]; ++kb) {
          if (!mbar_wait(empty_bar(stage), phase ^ 1u, abort_flag)) { ok = false; break; }
          if (lane == 0) {
            const uint32_t fb = full_bar(stage);
            const uint32_t sa = base + stage * TC_STAGE_BYTES;
            const uint32_t sb = sa + TC_A_BYTES;
            const int k0 = kb * TC_BK;
            mbar_arrive_expect_tx(fb, TC_STAGE_BYTES);
            if (G.a_mn) {
              tma_load_2d(sa, am, m0, k0, fb);
              tma_load_2d(sa + TC_MN_CHUNK_BYTES, am, m0 + 64, k0, fb);
            } else {
              tma_load_2d(sa, am, k0, m0, fb);
            }
            if (G.b_mn) {
#pragma unroll
              for (int j = 0; j < 4; ++j) tma_load_2d(sb + j * TC_MN_CHUNK_BYTES, bm, n0 + 64 * j, k0, fb);
            } else {
              tma_load_2d(sb, bm, k0, n0, fb);
            }
          }
          __syncwarp();
          issued_mask |= 1u << stage;
          issued_par = (issued_par & ~(1u << stage)) | (phase << stage);
          if (++stage == TC_STAGES) { stage = 0; phase ^= 1u; }
        }
      }
    }
    if (!ok) {
      // Let every copy this CTA issued land before shared memory is released.
      for (int s = 0; s < TC_STAGES; ++s) {
        if (!(issued_mask & (1u << s))) continue;
        const uint32_t par = (issued_par >> s) & 1u;
        const uint64_t t0 = global_timer_ns();
        while (!mbar_try_wait(full_bar(s), par) && global_timer_ns() - t0 < kWaitNs) {}
      }
      if (lane == 0) set_dev_err(p.err, DEV_ERR_TIMEOUT);
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer (one thread)
    // The tensor pipe accepts only a few MMAs ahead, so the issuing thread
    // blocks inside each stage's MMAs and must come back for the next stage
    // before the queued work drains: everything per tile is hoisted into
    // registers and the per-stage path is wait / fence / 4 MMAs / commit.
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true, issued_any = false;
      for (int ti = 0, tile; ok && (tile = tile_at(p, unit, nunits, ti)) >= 0; ++ti) {
        const int g = group_of(p, tile);
        const TcGroup& G = p.grp[g];
        const int nkb = G.kb[0] + (G.nseg > 1 ? G.kb[1] : 0);
        const uint32_t idesc = G.idesc;
        const uint64_t adesc = G.a_mn ? smem_desc(base, TC_MN_CHUNK_BYTES, 1024) : smem_desc(base, 16, 1024);
        const uint64_t bdesc =
            G.b_mn ? smem_desc(base + TC_A_BYTES, TC_MN_CHUNK_BYTES, 1024) : smem_desc(base + TC_A_BYTES, 16, 1024);
        const uint32_t astep = G.a_mn ? (2048u >> 4) : (32u >> 4);  // one K=16 slice, in 16-byte units
        const uint32_t bstep = G.b_mn ? (2048u >> 4) : (32u >> 4);
        if (!mbar_wait(tempty_bar(acc), acc_phase ^ 1u, abort_flag)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * TC_BN;
        uint32_t accum = 0;
        for (int kb = 0; kb < nkb; ++kb) {
          if (!mbar_wait(full_bar(stage), phase, abort_flag)) { ok = false; break; }
          tc_fence_after();
          const uint32_t so = (uint32_t)(stage * TC_STAGE_BYTES) >> 4;
#pragma unroll
          for (int k = 0; k < TC_BK / 16; ++k) {
            tc_mma(d_tmem, adesc + so + k * astep, bdesc + so + k * bstep, idesc, accum);
            accum = 1;
          }
          tc_commit(empty_bar(stage));
          issued_any = true;
          if (++stage == TC_STAGES) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        tc_commit(tfull_bar(acc));
        if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
      }
      if (!ok && issued_any) {
        // Wait for this thread's MMAs to finish before TMEM is freed.
        tc_commit(drain_bar);
        const uint64_t t0 = global_timer_ns();
        while (!mbar_try_wait(drain_bar, 0) && global_timer_ns() - t0 < kWaitNs) {}
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------ epilogue (warps 2..9)
    const int q = warp & 3;             // TMEM lane quadrant this warp may access
    const int half = (warp - 2) >> 2;   // which 128 of the 256 accumulator columns
    const uint32_t stage_s = epi_base + (warp - 2) * TC_EPI_STAGE_BYTES;
    float4* stage = reinterpret_cast<float4*>(smem_raw + (stage_s - raw));
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int ti = 0, tile; (tile = tile_at(p, unit, nunits, ti)) >= 0; ++ti) {
      int g, m0, n0;
      decode_tile(p, tile, g, m0, n0);
      const TcGroup& G = p.grp[g];
      const EpiOut eo = epi_out_of(G);
      const EpiIn ei = epi_in(G.epi);
      const int kind = G.kind;
      if (!mbar_wait(tfull_bar(acc), acc_phase, abort_flag)) break;
      tc_fence_after();
      int* ord_flag = G.epi.ord_role ? G.epi.ord_flags + (long)(tile - G.tile_start) * TC_EPI_WARPS + (warp - 2) : nullptr;
      if (G.epi.ord_role == ORD_WAIT) {
        // the same rows and columns of the signalling group must be in memory first
        bool ok = true;
        if (lane == 0) {
          ok = flag_wait_eq(ord_flag, G.epi.ord_epoch, abort_flag);
          fence_proxy_async_global();
        }
        if (!__shfl_sync(0xffffffffu, ok ? 1 : 0, 0)) {
          if (lane == 0) set_dev_err(p.err, DEV_ERR_TIMEOUT);
          break;
        }
      }
      const bool rd = G.epi.rd_out != nullptr;
      float rdot = 0.f;
      if (kind == EK_CESTATS) ce_stats_tile(&G.epi, eo.M, eo.N, m0 + q * 32 + lane, n0 + half * (TC_BN / 2),
                                            tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * TC_BN + half * (TC_BN / 2)));
      else
      for (int c = 0; c < TC_BN / 64; ++c) {
        const int col0 = n0 + half * (TC_BN / 2) + c * 32;
        if (col0 >= eo.N) break;
        uint32_t r[32];
        const uint32_t taddr =
            tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * TC_BN + half * (TC_BN / 2) + c * 32);
        TMEM_LD32(taddr, r);
        asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
        if (rd) {
          rdot += rowdot_any<act_t>(&G.epi, eo.M, eo.N, stage, lane, m0 + q * 32, col0, r);
          if ((col0 + 32) % G.epi.rd_hd == 0) { rowdot_store(&G.epi, eo.M, m0 + q * 32 + lane, col0 + 32, rdot); rdot = 0.f; }
        }
        epi_chunk_dispatch<act_t>(kind, p, &G.epi, ei, eo, stage, stage_s, lane, m0 + q * 32, col0, r);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty_bar(acc));
      if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
      if (G.epi.ord_role == ORD_SIGNAL) {
        // publish this warp's 32 x 128 piece once its stores have landed
        if (lane == 0) {
          bulk_wait_all();
          fence_proxy_async_global();
          st_release_gpu(ord_flag, G.epi.ord_epoch);
        }
        __syncwarp();
      }
    }
    if (lane == 0) bulk_wait_all();
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(512) : "memory");
  }
}


// ------------------------------------------------------------ CTA-pair kernel
// Same contract as gemm_tc_kernel, but a cluster of two CTAs (two SMs) computes
// a 256x256 output tile with tcgen05.mma.cta_group::2 (M=256, N=256, K=16):
// each CTA stages its own 128 rows of A and 128 of the 256 B rows, so every SM
// moves 32 KB per 64-deep K step instead of 48 KB and keeps six stages in
// flight.  The even CTA issues the MMAs; its full barriers collect both CTAs'
// TMA bytes; commits arrive on both CTAs' barriers; each CTA's epilogue reads
// its own 128 accumulator rows from its TMEM.
constexpr int T2_STAGES = 6;
constexpr int T2_A_BYTES = 128 * TC_BK * 2;  // 16 KB: this CTA's 128 rows of A
constexpr int T2_B_BYTES = 128 * TC_BK * 2;  // 16 KB: this CTA's 128 rows of B
constexpr int T2_STAGE_BYTES = T2_A_BYTES + T2_B_BYTES;
constexpr int T2_SMEM = T2_STAGES * T2_STAGE_BYTES + TC_EPI_WARPS * TC_EPI_STAGE_BYTES + 1024 + TC_BAR_BYTES;
constexpr int T2_TILE = 256;

__device__ __forceinline__ void decode_tile2(const TcParams& p, int tile, int& g, int& m0, int& n0) {
  g = group_of(p, tile);
  const TcGroup& G = p.grp[g];
  int mt, nt;
  tile_mn(G, tile - G.tile_start, mt, nt);
  m0 = mt * T2_TILE;
  n0 = nt * T2_TILE;
}

template <typename act_t>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(TC_THREADS, 1)
    gemm_tc2_kernel(const __grid_constant__ TcParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  const uint32_t epi_base = base + T2_STAGES * T2_STAGE_BYTES;
  const uint32_t bar_base = epi_base + TC_EPI_WARPS * TC_EPI_STAGE_BYTES;
  uint8_t* bar_ptr = smem_raw + (bar_base - raw);
  auto full_bar = [&](int s) { return bar_base + 8u * s; };
  auto empty_bar = [&](int s) { return bar_base + 8u * (T2_STAGES + s); };
  auto tfull_bar = [&](int b) { return bar_base + 8u * (2 * T2_STAGES + b); };
  auto tempty_bar = [&](int b) { return bar_base + 8u * (2 * T2_STAGES + 2 + b); };
  const uint32_t drain_bar = bar_base + 8u * (2 * T2_STAGES + 4);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar_ptr + 8 * (2 * T2_STAGES + 5));
  volatile uint32_t* abort_flag = reinterpret_cast<volatile uint32_t*>(bar_ptr + 8 * (2 * T2_STAGES + 5) + 4);

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int cluster_id = blockIdx.x >> 1, nclusters = gridDim.x >> 1;
  if (threadIdx.x == 0) {
    for (int s = 0; s < T2_STAGES; ++s) { mbar_init(full_bar(s), 1); mbar_init(empty_bar(s), 1); }
    for (int b = 0; b < 2; ++b) { mbar_init(tfull_bar(b), 1); mbar_init(tempty_bar(b), 2 * TC_EPI_WARPS); }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)), "r"(512)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  cluster_sync_all();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------ TMA producer (both CTAs)
    int stage = 0;
    uint32_t phase = 0;
    uint32_t issued_mask = 0, issued_par = 0;
    bool ok = true;
    for (int ti = 0, tile; ok && (tile = tile_at(p, cluster_id, nclusters, ti)) >= 0; ++ti) {
      int g, m0, n0;
      decode_tile2(p, tile, g, m0, n0);
      const TcGroup& G = p.grp[g];
      const int arow = m0 + (int)rank * 128, brow = n0 + (int)rank * 128;
      for (int s = 0; s < G.nseg && ok; ++s) {
        const CUtensorMap* am = &p.maps[G.amap[s]];
        const CUtensorMap* bm = &p.maps[G.bmap[s]];
        for (int kb = 0; kb < G.kb[s]; ++kb) {
          if (!mbar_wait_cluster(empty_bar(stage), phase ^ 1u, abort_flag)) { ok = false; break; }
          if (lane == 0) {
            const uint32_t fb = map_to_rank(full_bar(stage), 0);
            const uint32_t sa = base + stage * T2_STAGE_BYTES;
            const uint32_t sb = sa + T2_A_BYTES;
            const int k0 = kb * TC_BK;
            if (leader) mbar_arrive_expect_tx(full_bar(stage), 2 * T2_STAGE_BYTES);
            if (G.a_mn) {
              tma_load_2d_pair(sa, am, arow, k0, fb);
              tma_load_2d_pair(sa + TC_MN_CHUNK_BYTES, am, arow + 64, k0, fb);
            } else {
              tma_load_2d_pair(sa, am, k0, arow, fb);
            }
            if (G.b_mn) {
              tma_load_2d_pair(sb, bm, brow, k0, fb);
              tma_load_2d_pair(sb + TC_MN_CHUNK_BYTES, bm, brow + 64, k0, fb);
            } else {
              tma_load_2d_pair(sb, bm, k0, brow, fb);
            }
          }
          __syncwarp();
          issued_mask |= 1u << stage;
          issued_par = (issued_par & ~(1u << stage)) | (phase << stage);
          if (++stage == T2_STAGES) { stage = 0; phase ^= 1u; }
        }
      }
    }
    if (!ok) {
      if (leader) {
        // The leader's full barriers collect both CTAs' bytes: wait for every
        // issued stage so no copy lands after shared memory is released.
        for (int s = 0; s < T2_STAGES; ++s) {
          if (!(issued_mask & (1u << s))) continue;
          const uint32_t par = (issued_par >> s) & 1u;
          const uint64_t t0 = global_timer_ns();
          while (!mbar_try_wait_cluster(full_bar(s), par) && global_timer_ns() - t0 < kWaitNs) {}
        }
      }
      if (lane == 0) set_dev_err(p.err, DEV_ERR_TIMEOUT);
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer (one thread of the even CTA)
    if (leader && lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true, issued_any = false;
      for (int ti = 0, tile; ok && (tile = tile_at(p, cluster_id, nclusters, ti)) >= 0; ++ti) {
        const int g = group_of(p, tile);
        const TcGroup& G = p.grp[g];
        const int nkb = G.kb[0] + (G.nseg > 1 ? G.kb[1] : 0);
        const uint32_t idesc = G.idesc;
        const uint64_t adesc = G.a_mn ? smem_desc(base, TC_MN_CHUNK_BYTES, 1024) : smem_desc(base, 16, 1024);
        const uint64_t bdesc =
            G.b_mn ? smem_desc(base + T2_A_BYTES, TC_MN_CHUNK_BYTES, 1024) : smem_desc(base + T2_A_BYTES, 16, 1024);
        const uint32_t astep = G.a_mn ? (2048u >> 4) : (32u >> 4);
        const uint32_t bstep = G.b_mn ? (2048u >> 4) : (32u >> 4);
        if (!mbar_wait_cluster(tempty_bar(acc), acc_phase ^ 1u, abort_flag)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * TC_BN;
        uint32_t accum = 0;
        for (int kb = 0; kb < nkb; ++kb) {
          if (!mbar_wait_cluster(full_bar(stage), phase, abort_flag)) { ok = false; break; }
          tc_fence_after();
          const uint32_t so = (uint32_t)(stage * T2_STAGE_BYTES) >> 4;
#pragma unroll
          for (int k = 0; k < TC_BK / 16; ++k) {
            tc_mma_pair(d_tmem, adesc + so + k * astep, bdesc + so + k * bstep, idesc, accum);
            accum = 1;
          }
          tc_commit_pair_both(empty_bar(stage));
          issued_any = true;
          if (++stage == T2_STAGES) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        tc_commit_pair_both(tfull_bar(acc));
        if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
      }
      if (!ok && issued_any) {
        tc_commit_pair_local(drain_bar);
        const uint64_t t0 = global_timer_ns();
        while (!mbar_try_wait(drain_bar, 0) && global_timer_ns() - t0 < kWaitNs) {}
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------ epilogue (warps 2..9, both CTAs)
    const int q = warp & 3;
    const int half = (warp - 2) >> 2;
    const uint32_t stage_s = epi_base + (warp - 2) * TC_EPI_STAGE_BYTES;
    float4* stage = reinterpret_cast<float4*>(smem_raw + (stage_s - raw));
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int ti = 0, tile; (tile = tile_at(p, cluster_id, nclusters, ti)) >= 0; ++ti) {
      int g, m0, n0;
      decode_tile2(p, tile, g, m0, n0);
      const TcGroup& G = p.grp[g];
      const EpiOut eo = epi_out_of(G);
      const EpiIn ei = epi_in(G.epi);
      const int kind = G.kind;
      if (!mbar_wait_cluster(tfull_bar(acc), acc_phase, abort_flag)) break;
      tc_fence_after();
      int* ord_flag = G.epi.ord_role ? G.epi.ord_flags + (long)(tile - G.tile_start) * (2 * TC_EPI_WARPS) +
                                           (int)rank * TC_EPI_WARPS + (warp - 2)
                                     : nullptr;
      if (G.epi.ord_role == ORD_WAIT) {
        // the same rows and columns of the signalling group must be in memory first
        bool ok = true;
        if (lane == 0) {
          ok = flag_wait_eq(ord_flag, G.epi.ord_epoch, abort_flag);
          fence_proxy_async_global();
        }
        if (!__shfl_sync(0xffffffffu, ok ? 1 : 0, 0)) {
          if (lane == 0) set_dev_err(p.err, DEV_ERR_TIMEOUT);
          break;
        }
      }
      const int row0 = m0 + (int)rank * 128 + q * 32;
      const bool rd = G.epi.rd_out != nullptr;
      float rdot = 0.f;
      if (kind == EK_CESTATS) ce_stats_tile(&G.epi, eo.M, eo.N, row0 + lane, n0 + half * (TC_BN / 2),
                                            tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * TC_BN + half * (TC_BN / 2)));
      else
      for (int c = 0; c < TC_BN / 64; ++c) {
        const int col0 = n0 + half * (TC_BN / 2) + c * 32;
        if (col0 >= eo.N) break;
        uint32_t r[32];
        const uint32_t taddr =
            tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * TC_BN + half * (TC_BN / 2) + c * 32);
        TMEM_LD32(taddr, r);
        asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
        if (rd) {
          rdot += rowdot_any<act_t>(&G.epi, eo.M, eo.N, stage, lane, row0, col0, r);
          if ((col0 + 32) % G.epi.rd_hd == 0) { rowdot_store(&G.epi, eo.M, row0 + lane, col0 + 32, rdot); rdot = 0.f; }
        }
        epi_chunk_dispatch<act_t>(kind, p, &G.epi, ei, eo, stage, stage_s, lane, row0, col0, r);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (leader) mbar_arrive(tempty_bar(acc));
        else mbar_arrive_remote(map_to_rank(tempty_bar(acc), 0));
      }
      if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
      if (G.epi.ord_role == ORD_SIGNAL) {
        // publish this warp's 32 x 128 piece once its stores have landed
        if (lane == 0) {
          bulk_wait_all();
          fence_proxy_async_global();
          st_release_gpu(ord_flag, G.epi.ord_epoch);
        }
        __syncwarp();
      }
    }
    if (lane == 0) bulk_wait_all();
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync_all();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(512) : "memory");
  }
}

// ------------------------------------------------------------ host side
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

bool get_encoder(std::string* msg) {
  std::call_once(g_encode_once, [] {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  if (!g_encode && msg) *msg = "cuTensorMapEncodeTiled not available from the driver";
  return g_encode != nullptr;
}

// 2-D bf16 map over a row-major matrix with `inner` contiguous elements per row.
bool encode_map(CUtensorMap* m, const void* ptr, uint64_t inner, uint64_t outer, uint64_t ld,
                uint32_t box_inner, uint32_t box_outer, std::string* msg) {
  if ((reinterpret_cast<uintptr_t>(ptr) & 15) || ((ld * 2) & 15)) {
    if (msg) *msg = "tcgen05 GEMM operand needs a 16-byte aligned base and a leading dimension multiple of 8";
    return false;
  }
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {ld * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (msg) *msg = "cuTensorMapEncodeTiled failed (code " + std::to_string((int)r) + ")";
    return false;
  }
  return true;
}

// 2-D map for the epilogue's TMA stores: 32x32 boxes whose rows (64 B in bf16,
// 128 B in fp32) are swizzled in shared memory (64-byte / 128-byte swizzle) so
// that each lane can write its own row without bank conflicts.  Returns false
// (no error) when the output cannot be described by a tensor map; the kernel
// then stores with plain per-thread instructions.
bool encode_out_map(CUtensorMap* m, const void* ptr, int f32, uint64_t cols, uint64_t rows, uint64_t ld) {
  const uint64_t esz = f32 ? 4 : 2;
  if (!ptr || (reinterpret_cast<uintptr_t>(ptr) & 15) || ((ld * esz) & 15)) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {ld * esz};
  cuuint32_t box[2] = {32, 32};
  cuuint32_t estr[2] = {1, 1};
  return g_encode(m, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr),
                  dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  f32 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// kind::f16 instruction descriptor: fp32 accumulator, bf16 A and B,
// A/B major-ness, N>>3 at bits 17-22, M>>4 at bits 24-28.
uint32_t make_idesc(int a_mn, int b_mn, int m) {
  uint32_t d = 0;
  d |= 1u << 4;             // D format: f32
  d |= 1u << 7;             // A format: bf16
  d |= 1u << 10;            // B format: bf16
  d |= (uint32_t)a_mn << 15;
  d |= (uint32_t)b_mn << 16;
  d |= (uint32_t)(TC_BN >> 3) << 17;
  d |= (uint32_t)(m >> 4) << 24;
  return d;
}

bool check_ld(long ld, const void* p) { return p == nullptr || ((ld & 3) == 0 && (reinterpret_cast<uintptr_t>(p) & 15) == 0); }

}  // namespace

bool tma_map_2d(void* map128, const void* ptr, int f32, unsigned long long inner, unsigned long long outer,
                unsigned long long ld, unsigned box_inner, unsigned box_outer, int swizzle128, std::string* msg) {
  if (!get_encoder(msg)) return false;
  const uint64_t esz = f32 ? 4 : 2;
  if ((reinterpret_cast<uintptr_t>(ptr) & 15) || ((ld * esz) & 15)) {
    if (msg) *msg = "TMA operand needs a 16-byte aligned base and a 16-byte multiple row pitch";
    return false;
  }
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {ld * esz};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(reinterpret_cast<CUtensorMap*>(map128),
                        f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                        const_cast<void*>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (msg) *msg = "cuTensorMapEncodeTiled failed (code " + std::to_string((int)r) + ")";
    return false;
  }
  return true;
}

namespace {
std::atomic<long long> g_launches{0};
}
void count_launches(long long n) { g_launches.fetch_add(n, std::memory_order_relaxed); }
long long launches_total() { return g_launches.load(std::memory_order_relaxed); }

int num_sms() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}

int gemm_tc(const GemmCall& c, int* dev_err, cudaStream_t s, std::string* msg) {
  // CTA pairs (256 x 256 tiles, each SM reading half of both operand tiles)
  // are faster than single CTAs for every operand layout and shape of the model.
  return gemm_tc_engine(c, TC_PAIR, dev_err, s, msg);
}

// How many clusters of two CTAs of `kernel` (dynamic shared memory `smem`) fit on the GPU at once.
template <typename K>
int max_pair_clusters(K kernel, int smem) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * (num_sms() / 2), 1, 1);
  cfg.blockDim = dim3(TC_THREADS, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = 2; attr.val.clusterDim.y = 1; attr.val.clusterDim.z = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kernel, &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    n = num_sms() / 2;
  }
  return n;
}

// Longest-first assignment of tiles to the units of the persistent grid, for
// launches whose groups differ in depth K (a weight-gradient group with
// K = B*T beside data-gradient groups with K = d or d_ff).  Round robin gives
// every unit the same number of tiles, so the units that draw more of the deep
// ones finish last.  A tile costs its K plus a fixed pipeline overhead; tiles
// go, deepest group first and in tile order within a group, to the unit with
// the least work so far.  The lists live in device memory, built once per
// (units, group tiles and depths) for the life of the process.  Launches with
// an ordered split-K keep round robin: their waits rely on it.
const int* tile_schedule(const GemmCall& c, const TcParams& p, int nunits) {
  long depth[kMaxGemmGroups];
  bool uneven = false;
  for (int g = 0; g < c.ngroups; ++g) {
    if (c.g[g].epi.ord_role) return nullptr;
    depth[g] = 0;
    for (int k = 0; k < c.g[g].nseg; ++k) depth[g] += c.g[g].seg[k].K;
    uneven = uneven || depth[g] != depth[0];
  }
  if (!uneven || nunits <= 1) return nullptr;
  std::vector<long> key = {nunits, c.ngroups};
  for (int g = 0; g < c.ngroups; ++g) {
    key.push_back((long)p.grp[g].m_tiles * p.grp[g].n_tiles);
    key.push_back(depth[g]);
  }
  static std::mutex mu;
  static std::map<std::vector<long>, int*> cache;
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find(key);
  if (it != cache.end()) return it->second;
  int order[kMaxGemmGroups];
  for (int g = 0; g < c.ngroups; ++g) order[g] = g;
  std::stable_sort(order, order + c.ngroups, [&](int a, int b) { return depth[a] > depth[b]; });
  typedef std::pair<long, int> Load;
  std::priority_queue<Load, std::vector<Load>, std::greater<Load>> heap;
  for (int u = 0; u < nunits; ++u) heap.push(Load(0, u));
  std::vector<std::vector<int>> lists(nunits);
  for (int oi = 0; oi < c.ngroups; ++oi) {
    const TcGroup& G = p.grp[order[oi]];
    const long cost = depth[order[oi]] + 384;
    for (int t = G.tile_start; t < G.tile_start + G.m_tiles * G.n_tiles; ++t) {
      Load l = heap.top();
      heap.pop();
      lists[l.second].push_back(t);
      heap.push(Load(l.first + cost, l.second));
    }
  }
  std::vector<int> flat(nunits + 1 + p.total_tiles), seen(p.total_tiles, 0);
  int n = 0;
  for (int u = 0; u < nunits; ++u) {
    flat[u] = n;
    for (int t : lists[u]) { flat[nunits + 1 + n++] = t; ++seen[t]; }
  }
  flat[nunits] = n;
  for (int t = 0; t < p.total_tiles; ++t)
    if (seen[t] != 1) return nullptr;  // cannot happen; round robin is always valid
  int* d = nullptr;
  if (cudaMalloc(&d, flat.size() * sizeof(int)) != cudaSuccess) { cudaGetLastError(); return nullptr; }
  if (cudaMemcpy(d, flat.data(), flat.size() * sizeof(int), cudaMemcpyHostToDevice) != cudaSuccess) {
    cudaGetLastError();
    cudaFree(d);
    return nullptr;
  }
  cache[key] = d;
  return d;
}

int gemm_tc_engine(const GemmCall& c, int kind, int* dev_err, cudaStream_t s, std::string* msg) {
  if (!get_encoder(msg)) return 4;
  static bool attr_set = false;
  static int pair_clusters = 0;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<bf16>, cudaFuncAttributeMaxDynamicSharedMemorySize, TC_SMEM);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(gemm_tc2_kernel<bf16>, cudaFuncAttributeMaxDynamicSharedMemorySize, T2_SMEM);
    if (e != cudaSuccess) { if (msg) *msg = std::string("gemm_tc smem attribute: ") + cudaGetErrorString(e); return 4; }
    pair_clusters = max_pair_clusters(gemm_tc2_kernel<bf16>, T2_SMEM);
    attr_set = true;
  }
  if (kind != TC_ONE && kind != TC_PAIR) { if (msg) *msg = "unknown tcgen05 GEMM kind"; return 1; }
  const bool pair = kind == TC_PAIR;
  const int bm = pair ? T2_TILE : TC_BM, bn = pair ? T2_TILE : TC_BN;
  const int a_rows = 128, b_rows = pair ? 128 : TC_BN;  // K-major TMA box heights per CTA
  TcParams p;
  memset(&p, 0, sizeof(p));
  int nmaps = 0, tiles = 0;
  if (c.ngroups < 1 || c.ngroups > kMaxGemmGroups) { if (msg) *msg = "GEMM launch needs 1 to 4 groups"; return 1; }
  p.ngroups = c.ngroups;
  for (int g = 0; g < c.ngroups; ++g) {
    const GemmGroupDesc& G = c.g[g];
    TcGroup& T = p.grp[g];
    T.M = G.M; T.N = G.N; T.nseg = G.nseg;
    T.m_tiles = (G.M + bm - 1) / bm;
    T.n_tiles = (G.N + bn - 1) / bn;
    T.tile_start = tiles;
    {
      // Bands of about one wave of tiles when a column of tiles is narrower
      // than the machine: the A rows of a band are then read from DRAM once.
      const int conc = pair ? pair_clusters : num_sms();
      T.band_m = (T.n_tiles <= conc) ? (conc / T.n_tiles > 1 ? conc / T.n_tiles : 1) : 0;
    }
    T.epi = G.epi;
    const EpiParams& e = G.epi;
    if (!check_ld(e.ldo, e.out) || !check_ld(e.ldo2, e.out2) || !check_ld(e.ldr, e.resid) ||
        !check_ld(e.ldr2, e.resid2) || !check_ld(e.ldx, e.aux) || !check_ld(0, e.bias) || !check_ld(0, e.bias2)) {
      if (msg) *msg = "tcgen05 GEMM epilogue pointers must be 16-byte aligned with leading dimensions multiple of 4";
      return 1;
    }
    if (G.nseg < 1 || G.nseg > 2 || G.M <= 0 || G.N <= 0) { if (msg) *msg = "bad GEMM group"; return 1; }
    T.a_mn = G.seg[0].A.mn_major;
    T.b_mn = G.seg[0].B.mn_major;
    for (int sg = 0; sg < G.nseg; ++sg) {
      const GemmSeg& S = G.seg[sg];
      if (S.A.mn_major != T.a_mn || S.B.mn_major != T.b_mn || S.K <= 0) {
        if (msg) *msg = "GEMM segments of one group must share operand majors";
        return 1;
      }
      T.kb[sg] = (S.K + TC_BK - 1) / TC_BK;
      if (nmaps + 2 > kMaxMaps) { if (msg) *msg = "too many GEMM operands in one launch"; return 1; }
      // A: logical [M, K]
      if (S.A.mn_major) {
        if (!encode_map(&p.maps[nmaps], S.A.ptr, G.M, S.K, S.A.ld, 64, TC_BK, msg)) return 1;
      } else {
        if (!encode_map(&p.maps[nmaps], S.A.ptr, S.K, G.M, S.A.ld, TC_BK, a_rows, msg)) return 1;
      }
      T.amap[sg] = nmaps++;
      if (S.B.mn_major) {
        if (!encode_map(&p.maps[nmaps], S.B.ptr, G.N, S.K, S.B.ld, 64, TC_BK, msg)) return 1;
      } else {
        if (!encode_map(&p.maps[nmaps], S.B.ptr, S.K, G.N, S.B.ld, TC_BK, b_rows, msg)) return 1;
      }
      T.bmap[sg] = nmaps++;
    }
    T.idesc = make_idesc(T.a_mn, T.b_mn, pair ? 256 : TC_BM);
    // output maps (TMA stores) when every output of the group allows them
    {
      const int k = epi_kind(e);
      const bool special = k == 0 || k == EK_BIAS || k == (EK_BIAS | EK_GELU) || k == EK_DGELU ||
                           k == (EK_BIAS | EK_RESID) || k == (EK_BIAS | EK_BIAS2 | EK_RESID) || k == EK_ADAMW ||
                           k == EK_CEGRAD || k == EK_CESTATS;
      T.kind = special ? k : EK_ANY;
    }
    if ((e.op == EPI_CE_GRAD || e.op == EPI_CE_STATS) &&
        (e.bias || e.bias2 || e.resid || e.resid2 || e.pre_f32 || e.rd_out || e.ord_role || !e.ce_tgt ||
         (e.op == EPI_CE_GRAD ? (e.out_mode != OUT_ACT || !e.out || !e.ce_lse)
                              : (e.out != nullptr || !e.ce_stats || !e.ce_tlogit || e.ce_ld < G.M)))) {
      if (msg) *msg = "cross-entropy epilogue needs its row vectors, a plain output (gradient) or none (statistics)";
      return 1;
    }
    if (e.rd_out && (e.op != EPI_NONE || e.bias || e.bias2 || e.resid || e.resid2 || e.pre_f32 ||
                     e.out_mode != OUT_ACT || e.rd_hd <= 0 || e.rd_hd % 32 || G.N % e.rd_hd || e.rd_T <= 0 ||
                     e.rd_H <= 0 || !check_ld(e.rd_ld, e.rd_src) || (e.rd_ld & 7))) {
      if (msg) *msg = "row-dot epilogue needs a plain activation output and head-aligned columns";
      return 1;
    }
    if (e.op == EPI_ADAMW &&
        (e.out_mode != OUT_F32 || !e.opt_p || !e.opt_m || !e.opt_v || !check_ld(e.ldo, e.opt_p) ||
         !check_ld(e.ldo, e.opt_m) || !check_ld(e.ldo, e.opt_v) ||
         (e.opt_sh && (reinterpret_cast<uintptr_t>(e.opt_sh) & 7)))) {
      if (msg) *msg = "fused AdamW epilogue needs an fp32 gradient output and aligned optimizer arrays";
      return 1;
    }
    T.out_f32 = e.out_mode != OUT_ACT && e.op != EPI_GELU;
    T.out_accum = e.out_mode == OUT_F32_ACCUM;
    T.out_tma = 0;
    T.omap = T.omap2 = 0;
    if (e.op != EPI_ADAMW && nmaps + 2 <= kMaxMaps && encode_out_map(&p.maps[nmaps], e.out, T.out_f32, G.N, G.M, e.ldo)) {
      T.omap = nmaps;
      bool ok = true;
      if (e.op == EPI_GELU) {
        ok = encode_out_map(&p.maps[nmaps + 1], e.out2, 0, G.N, G.M, e.ldo2);
        T.omap2 = nmaps + 1;
      }
      if (ok) {
        T.out_tma = 1;
        nmaps += (e.op == EPI_GELU) ? 2 : 1;
      }
    }
    tiles += T.m_tiles * T.n_tiles;
  }
  // Groups of one launch that add into the same output must do so with TMA
  // reduce-adds: the per-thread fallback is a plain read-modify-write.
  for (int g = 0; g < c.ngroups; ++g)
    for (int o = 0; o < c.ngroups; ++o)
      if (o != g && p.grp[g].out_accum && !p.grp[g].out_tma && c.g[g].epi.out == c.g[o].epi.out) {
        if (msg) *msg = "GEMM groups accumulating into one output need TMA-storable outputs";
        return 1;
      }
  // Ordered split-K: every waiting group follows a signalling group of the same
  // shape and output (its tiles come first in the static schedule, and tiles of
  // a signalling group never wait, so every wait ends).
  for (int g = 0; g < c.ngroups; ++g) {
    const EpiParams& e = c.g[g].epi;
    if (!e.ord_role) continue;
    const TcGroup& T = p.grp[g];
    const long flags_per_tile = pair ? 2 * TC_EPI_WARPS : TC_EPI_WARPS;
    bool ok = T.out_tma && e.ord_flags && e.ord_role >= ORD_SIGNAL &&
              e.ord_role <= ORD_WAIT && (long)T.m_tiles * T.n_tiles * flags_per_tile <= (long)e.ord_cap &&
              e.rd_out == nullptr;
    if (ok && e.ord_role == ORD_WAIT) {
      ok = false;
      if (e.out_mode == OUT_F32_ACCUM)
        for (int o = 0; o < g; ++o)
          if (c.g[o].epi.ord_role == ORD_SIGNAL && c.g[o].epi.ord_flags == e.ord_flags &&
              c.g[o].epi.ord_epoch == e.ord_epoch && c.g[o].epi.out == e.out && c.g[o].M == c.g[g].M &&
              c.g[o].N == c.g[g].N)
            ok = true;
    }
    if (!ok) {
      if (msg) *msg = "ordered split-K needs the one-CTA or pair engine, TMA outputs and a matching signalling group first";
      return 1;
    }
  }
  p.total_tiles = tiles;
  p.err = dev_err;
  if (tiles == 0) return 0;
  const int cap = pair ? pair_clusters : num_sms();
  const int nunits = tiles < cap ? tiles : cap;
  p.sched = tile_schedule(c, p, nunits);
  if (pair) {
    const int clusters = nunits;
    gemm_tc2_kernel<bf16><<<2 * clusters, TC_THREADS, T2_SMEM, s>>>(p);
  } else {
    gemm_tc_kernel<bf16><<<nunits, TC_THREADS, TC_SMEM, s>>>(p);
  }
  count_launches(1);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) { if (msg) *msg = std::string("gemm_tc launch: ") + cudaGetErrorString(e); return 4; }
  return 0;
}

}  // namespace fal
