// Row-streaming LayerNorm forward and backward: the LN_1, LN_2, LN_F and final
// LayerNorms of the blocks (Eq. 1, Eq. 2) with their backward, for rows of up
// to 4096 features.
//
// These kernels are bound by HBM bandwidth.  Warp-per-row kernels that load a
// row into registers keep too few bytes in flight per SM (every load holds an
// L1 miss slot until it returns).  Here persistent CTAs (two per SM) stream their
// rows through a ring of shared-memory stages filled by bulk copies
// (cp.async.bulk, issued by one producer thread, completion counted on an
// mbarrier), so several rows per SM are always on their way from HBM without
// holding registers.  Eight consumer warps share each row: every thread owns
// up to four 4-column groups of it, row statistics are reduced with warp
// shuffles and one named barrier, and each row's outputs leave with coalesced
// 16-byte stores.  The backward also accumulates the affine parameters'
// gradient column sums in registers across all rows of the CTA, so no second
// pass over the rows is needed.
//
// Every mbarrier wait is bounded; on expiry the CTA's consumers agree (barrier
// reduction) to stop, record DEV_ERR_TIMEOUT in the device error word, the
// producer waits for the copies it issued, and the launch returns normally.
// Two CTAs share an SM, so that one CTA's row reductions overlap the other's.
// The backward can also sum the columns of its output dx (the bias gradients
// of the linear maps whose outputs feed the normalised residual).
#include <atomic>

#include "tc_ptx.cuh"

namespace fal {

namespace {

using namespace ptx;

constexpr float LR_EPS = 1e-5f;
constexpr int LR_WARPS = 8;                 // consumer warps
constexpr int LR_CONS = LR_WARPS * 32;      // consumer threads
constexpr int LR_THREADS = LR_CONS + 32;    // + one producer warp
constexpr int LR_MAX_D = 4 * 4 * LR_CONS;   // up to four 4-column groups per consumer thread
constexpr int LR_MAX_STAGES = 8;
constexpr uint32_t LR_STAGE_BUDGET = 96 * 1024;  // two CTAs per SM (rows of up to 2048 features)
constexpr uint32_t LR_WIDE_BUDGET = 192 * 1024;  // one CTA per SM (wider rows: four column groups)
constexpr uint32_t LR_TAIL_BYTES = 16 * LR_MAX_STAGES + 32 * 4 + 16;  // barriers, reduction slots, abort flag
constexpr uint32_t LR_SMEM_MAX = LR_STAGE_BUDGET + LR_TAIL_BYTES;
constexpr uint32_t LR_WIDE_SMEM_MAX = LR_WIDE_BUDGET + LR_TAIL_BYTES;
// Column groups per consumer thread for rows of d features, and CTAs per SM.
__host__ __device__ constexpr int lr_nch(int d) { return d <= 4 * LR_CONS ? 1 : d <= 8 * LR_CONS ? 2 : 4; }
__host__ __device__ constexpr int lr_ctas_per_sm(int nch) { return nch > 2 ? 1 : 2; }

// fp32 row-major [rows, d] inputs copied into each stage, in slot order.
struct RowSrc {
  const float* p[4];
  int n;
};

struct Ring {
  uint32_t base, stage_bytes, bar_base;
  int stages;
  __device__ uint32_t full(int s) const { return bar_base + 8u * s; }
  __device__ uint32_t empty(int s) const { return bar_base + 8u * (stages + s); }
};

// Bounded wait with a budget of wait_ns (the default when <= 0).
__device__ __forceinline__ bool ring_wait(uint32_t bar, uint32_t parity, volatile uint32_t* abort_flag,
                                          long long wait_ns) {
  if (wait_ns <= 0) return mbar_wait(bar, parity, abort_flag);
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (global_timer_ns() - t0 > (uint64_t)wait_ns) { *abort_flag = 1; return false; }
  }
}

// One thread: copies every row r = blockIdx.x + k * gridDim.x of the sources
// into the ring, then waits until each copy it issued has landed (with the
// default budget, whatever wait_ns is).  stall_rows >= 0 (test hook): stop
// after that many rows.
__device__ void produce_rows(const RowSrc src, int rows, int d, const Ring ring, volatile uint32_t* abort_flag,
                             long long wait_ns, int stall_rows) {
  const uint32_t rb = (uint32_t)d * 4u;
  int s = 0, n = 0;
  uint32_t ph = 0, issued_mask = 0, issued_par = 0;
  for (int r = blockIdx.x; r < rows; r += gridDim.x, ++n) {
    if (stall_rows >= 0 && n >= stall_rows) break;
    if (!ring_wait(ring.empty(s), ph ^ 1u, abort_flag, wait_ns)) break;
    mbar_arrive_expect_tx(ring.full(s), (uint32_t)src.n * rb);
    const uint32_t dst = ring.base + (uint32_t)s * ring.stage_bytes;
    for (int k = 0; k < src.n; ++k) bulk_load_1d(dst + (uint32_t)k * rb, src.p[k] + (long)r * d, rb, ring.full(s));
    issued_mask |= 1u << s;
    issued_par = (issued_par & ~(1u << s)) | (ph << s);
    if (++s == ring.stages) { s = 0; ph ^= 1u; }
  }
  for (int k = 0; k < ring.stages; ++k) {
    if (!(issued_mask & (1u << k))) continue;
    const uint64_t t0 = global_timer_ns();
    while (!mbar_try_wait(ring.full(k), (issued_par >> k) & 1u) && global_timer_ns() - t0 < kWaitNs) {}
  }
}

__device__ __forceinline__ Ring setup_ring(uint8_t* smem, int stages, uint32_t stage_bytes, float** red,
                                           volatile uint32_t** abort_flag) {
  Ring ring;
  ring.base = smem_u32(smem);
  ring.stage_bytes = stage_bytes;
  ring.stages = stages;
  ring.bar_base = ring.base + (uint32_t)stages * stage_bytes;
  *red = reinterpret_cast<float*>(smem + (size_t)stages * stage_bytes + 16 * stages);
  *abort_flag = reinterpret_cast<volatile uint32_t*>(*red + 32);
  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) { mbar_init(ring.full(s), 1); mbar_init(ring.empty(s), LR_WARPS); }
    **abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  return ring;
}

__device__ __forceinline__ float4 f4_add(float4 a, float4 b) { return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w); }
__device__ __forceinline__ float4 f4_mul(float4 a, float4 b) { return make_float4(a.x * b.x, a.y * b.y, a.z * b.z, a.w * b.w); }
__device__ __forceinline__ float f4_sum(float4 a) { return a.x + a.y + a.z + a.w; }
__device__ __forceinline__ float4 f4_zero() { return make_float4(0.f, 0.f, 0.f, 0.f); }

// y = LN(x) (* gamma + beta); optional fp32 copy; out2 = y + add_src * add_g + add_b.
template <typename act_t, int NCH>
__global__ void __launch_bounds__(LR_THREADS, lr_ctas_per_sm(NCH)) ln_fwd_rows_kernel(const LnFwdArgs a, int stages, uint32_t stage_bytes,
                                                                    long long wait_ns, int stall_rows) {
  extern __shared__ __align__(16) uint8_t smem[];
  float* red;
  volatile uint32_t* abort_flag;
  const Ring ring = setup_ring(smem, stages, stage_bytes, &red, &abort_flag);
  const int d = a.d, d4 = d >> 2;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const bool has2 = a.out2 != nullptr && a.add_src != nullptr;
  if (warp == LR_WARPS) {
    if (lane == 0) {
      RowSrc src;
      src.p[0] = a.x; src.p[1] = has2 ? a.add_src : nullptr; src.p[2] = src.p[3] = nullptr;
      src.n = has2 ? 2 : 1;
      produce_rows(src, a.rows, d, ring, abort_flag, wait_ns, stall_rows);
    }
    return;
  }
  float4 gam[NCH], bet[NCH], ag[NCH], ab[NCH];
#pragma unroll
  for (int k = 0; k < NCH; ++k) {
    const int c4 = tid + k * LR_CONS;
    const bool in = c4 < d4;
    gam[k] = (in && a.gamma) ? load4(a.gamma + 4 * c4) : make_float4(1.f, 1.f, 1.f, 1.f);
    bet[k] = (in && a.beta) ? load4(a.beta + 4 * c4) : f4_zero();
    ag[k] = (in && a.add_g) ? load4(a.add_g + 4 * c4) : make_float4(1.f, 1.f, 1.f, 1.f);
    ab[k] = (in && a.add_b) ? load4(a.add_b + 4 * c4) : f4_zero();
  }
  int s = 0;
  uint32_t ph = 0, it = 0;
  for (int r = blockIdx.x; r < a.rows; r += gridDim.x, ++it) {
    const bool ok = ring_wait(ring.full(s), ph, abort_flag, wait_ns);
    float4 x[NCH], z[NCH];
    float sum = 0.f;
    const float4* st = reinterpret_cast<const float4*>(smem + (size_t)s * stage_bytes);
#pragma unroll
    for (int k = 0; k < NCH; ++k) {
      const int c4 = tid + k * LR_CONS;
      x[k] = (ok && c4 < d4) ? st[c4] : f4_zero();
      z[k] = (ok && has2 && c4 < d4) ? st[d4 + c4] : f4_zero();
      sum += f4_sum(x[k]);
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(ring.empty(s));
    if (++s == stages) { s = 0; ph ^= 1u; }
    float* rb = red + (it & 1u) * 16;
    sum = warp_sum(sum);
    if (lane == 0) rb[warp] = sum;
    if (named_bar_or(1, LR_CONS, !ok)) {
      if (tid == 0) set_dev_err(a.err, DEV_ERR_TIMEOUT);
      break;
    }
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < LR_WARPS; ++w) tot += rb[w];
    const float mean = tot / d;
    float q = 0.f;
#pragma unroll
    for (int k = 0; k < NCH; ++k) {
      const int c4 = tid + k * LR_CONS;
      if (c4 < d4) {
        const float dx = x[k].x - mean, dy = x[k].y - mean, dz = x[k].z - mean, dw = x[k].w - mean;
        q += dx * dx + dy * dy + dz * dz + dw * dw;
      }
    }
    q = warp_sum(q);
    if (lane == 0) rb[8 + warp] = q;
    named_bar_or(1, LR_CONS, false);
    float qt = 0.f;
#pragma unroll
    for (int w = 0; w < LR_WARPS; ++w) qt += rb[8 + w];
    const float rstd = rsqrtf(qt / d + LR_EPS);
    if (tid == 0) {
      if (a.mean) a.mean[r] = mean;
      if (a.rstd) a.rstd[r] = rstd;
    }
    const long off = (long)r * d;
#pragma unroll
    for (int k = 0; k < NCH; ++k) {
      const int c4 = tid + k * LR_CONS;
      if (c4 >= d4) continue;
      const float4 xh = make_float4((x[k].x - mean) * rstd, (x[k].y - mean) * rstd, (x[k].z - mean) * rstd,
                                    (x[k].w - mean) * rstd);
      const float4 y = f4_add(f4_mul(xh, gam[k]), bet[k]);
      if (a.out) store4(reinterpret_cast<act_t*>(a.out) + off + 4 * c4, y);
      if (a.out_f32) store4(a.out_f32 + off + 4 * c4, y);
      if (has2) store4(reinterpret_cast<act_t*>(a.out2) + off + 4 * c4, f4_add(y, f4_add(f4_mul(z[k], ag[k]), ab[k])));
    }
  }
}

// dx = rstd * (g - mean(g) - xhat * mean(g * xhat)) + dres with g = (dy + dy2) * gamma;
// optional per-CTA column sums of (dy + dy2) * xhat and (dy + dy2).
template <typename act_t, int NCH>
__global__ void __launch_bounds__(LR_THREADS, lr_ctas_per_sm(NCH)) ln_bwd_rows_kernel(const LnBwdArgs a, int stages, uint32_t stage_bytes,
                                                                    long long wait_ns, int stall_rows) {
  extern __shared__ __align__(16) uint8_t smem[];
  float* red;
  volatile uint32_t* abort_flag;
  const Ring ring = setup_ring(smem, stages, stage_bytes, &red, &abort_flag);
  const int d = a.d, d4 = d >> 2;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int i_dy2 = a.dy2 ? 2 : -1;
  const int i_dres = a.dres ? (a.dy2 ? 3 : 2) : -1;
  if (warp == LR_WARPS) {
    if (lane == 0) {
      RowSrc src;
      src.p[0] = a.x; src.p[1] = a.dy; src.p[2] = src.p[3] = nullptr;
      src.n = 2;
      if (a.dy2) src.p[src.n++] = a.dy2;
      if (a.dres) src.p[src.n++] = a.dres;
      produce_rows(src, a.rows, d, ring, abort_flag, wait_ns, stall_rows);
    }
    return;
  }
  float4 gam[NCH], cs0[NCH], cs1[NCH], cs2[NCH];
  const bool sum_dx = a.cs_part && (a.dxs_out || a.dxs_out2);
#pragma unroll
  for (int k = 0; k < NCH; ++k) {
    const int c4 = tid + k * LR_CONS;
    gam[k] = (a.gamma && c4 < d4) ? load4(a.gamma + 4 * c4) : make_float4(1.f, 1.f, 1.f, 1.f);
    cs0[k] = cs1[k] = cs2[k] = f4_zero();
  }
  int s = 0;
  uint32_t ph = 0, it = 0;
  for (int r = blockIdx.x; r < a.rows; r += gridDim.x, ++it) {
    const float mean = a.mean[r], rstd = a.rstd[r];
    const bool ok = ring_wait(ring.full(s), ph, abort_flag, wait_ns);
    float4 xh[NCH], gd[NCH], dr[NCH];
    float s1 = 0.f, s2 = 0.f;
    const float4* st = reinterpret_cast<const float4*>(smem + (size_t)s * stage_bytes);
#pragma unroll
    for (int k = 0; k < NCH; ++k) {
      const int c4 = tid + k * LR_CONS;
      if (ok && c4 < d4) {
        const float4 x = st[c4];
        float4 g = st[d4 + c4];
        if (i_dy2 >= 0) g = f4_add(g, st[i_dy2 * d4 + c4]);
        dr[k] = i_dres >= 0 ? st[i_dres * d4 + c4] : f4_zero();
        xh[k] = make_float4((x.x - mean) * rstd, (x.y - mean) * rstd, (x.z - mean) * rstd, (x.w - mean) * rstd);
        cs0[k] = f4_add(cs0[k], g);
        cs1[k] = f4_add(cs1[k], f4_mul(g, xh[k]));
        gd[k] = f4_mul(g, gam[k]);
        s1 += f4_sum(gd[k]);
        s2 += f4_sum(f4_mul(gd[k], xh[k]));
      } else {
        xh[k] = gd[k] = dr[k] = f4_zero();
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(ring.empty(s));
    if (++s == stages) { s = 0; ph ^= 1u; }
    float* rb = red + (it & 1u) * 16;
    s1 = warp_sum(s1);
    s2 = warp_sum(s2);
    if (lane == 0) { rb[warp] = s1; rb[8 + warp] = s2; }
    if (named_bar_or(1, LR_CONS, !ok)) {
      if (tid == 0) set_dev_err(a.err, DEV_ERR_TIMEOUT);
      break;
    }
    float m1 = 0.f, m2 = 0.f;
#pragma unroll
    for (int w = 0; w < LR_WARPS; ++w) { m1 += rb[w]; m2 += rb[8 + w]; }
    m1 /= d;
    m2 /= d;
    const long off = (long)r * d;
#pragma unroll
    for (int k = 0; k < NCH; ++k) {
      const int c4 = tid + k * LR_CONS;
      if (c4 >= d4) continue;
      const float4 o = make_float4(rstd * (gd[k].x - m1 - xh[k].x * m2) + dr[k].x,
                                   rstd * (gd[k].y - m1 - xh[k].y * m2) + dr[k].y,
                                   rstd * (gd[k].z - m1 - xh[k].z * m2) + dr[k].z,
                                   rstd * (gd[k].w - m1 - xh[k].w * m2) + dr[k].w);
      store4(a.dx + off + 4 * c4, o);
      if (a.dx_act) store4(reinterpret_cast<act_t*>(a.dx_act) + off + 4 * c4, o);
      if (sum_dx) cs2[k] = f4_add(cs2[k], o);
    }
  }
  if (a.cs_part) {
    const int ns = sum_dx ? 3 : 2;
#pragma unroll
    for (int k = 0; k < NCH; ++k) {
      const int c4 = tid + k * LR_CONS;
      if (c4 >= d4) continue;
      store4(a.cs_part + ((long)blockIdx.x * ns + 0) * d + 4 * c4, cs0[k]);
      store4(a.cs_part + ((long)blockIdx.x * ns + 1) * d + 4 * c4, cs1[k]);
      if (sum_dx) store4(a.cs_part + ((long)blockIdx.x * ns + 2) * d + 4 * c4, cs2[k]);
    }
  }
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

// Stage count for `nin` input rows of d floats, 0 when fewer than two fit.
int ring_stages(int nin, int d, uint32_t* stage_bytes) {
  *stage_bytes = (uint32_t)nin * (uint32_t)d * 4u;
  const uint32_t budget = lr_nch(d) > 2 ? LR_WIDE_BUDGET : LR_STAGE_BUDGET;
  int st = (int)(budget / *stage_bytes);
  if (st > LR_MAX_STAGES) st = LR_MAX_STAGES;
  return st >= 2 ? st : 0;
}

template <typename K>
bool set_smem_attr(K kernel, uint32_t bytes = LR_SMEM_MAX) {
  return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes) == cudaSuccess;
}

std::atomic<int> g_stall_rows{-1};
std::atomic<long long> g_wait_ns{0};

int rows_grid(int rows, int d) {
  int g = lr_ctas_per_sm(lr_nch(d)) * num_sms();
  if (g > kMaxColsumChunks) g = kMaxColsumChunks;  // per-CTA column partials must fit colsum_partial_floats(d)
  return rows < g ? rows : g;
}

template <typename act_t>
int ln_fwd_rows(const LnFwdArgs& a, cudaStream_t s) {
  static const bool attr = set_smem_attr(ln_fwd_rows_kernel<act_t, 1>) && set_smem_attr(ln_fwd_rows_kernel<act_t, 2>) &&
                           set_smem_attr(ln_fwd_rows_kernel<act_t, 4>, LR_WIDE_SMEM_MAX);
  if (!attr) return 1;
  const bool has2 = a.out2 != nullptr && a.add_src != nullptr;
  uint32_t sb;
  const int st = ring_stages(has2 ? 2 : 1, a.d, &sb);
  if (!st) return 1;
  const uint32_t smem = (uint32_t)st * sb + LR_TAIL_BYTES;
  const int grid = rows_grid(a.rows, a.d);
  const long long w = g_wait_ns.load();
  const int sr = g_stall_rows.load();
  const int nch = lr_nch(a.d);
  if (nch == 1) ln_fwd_rows_kernel<act_t, 1><<<grid, LR_THREADS, smem, s>>>(a, st, sb, w, sr);
  else if (nch == 2) ln_fwd_rows_kernel<act_t, 2><<<grid, LR_THREADS, smem, s>>>(a, st, sb, w, sr);
  else ln_fwd_rows_kernel<act_t, 4><<<grid, LR_THREADS, smem, s>>>(a, st, sb, w, sr);
  return 0;
}

template <typename act_t>
int ln_bwd_rows(const LnBwdArgs& a, cudaStream_t s) {
  static const bool attr = set_smem_attr(ln_bwd_rows_kernel<act_t, 1>) && set_smem_attr(ln_bwd_rows_kernel<act_t, 2>) &&
                           set_smem_attr(ln_bwd_rows_kernel<act_t, 4>, LR_WIDE_SMEM_MAX);
  if (!attr) return 1;
  uint32_t sb;
  const int st = ring_stages(2 + (a.dy2 ? 1 : 0) + (a.dres ? 1 : 0), a.d, &sb);
  if (!st) return 1;
  const uint32_t smem = (uint32_t)st * sb + LR_TAIL_BYTES;
  const int grid = rows_grid(a.rows, a.d);
  const long long w = g_wait_ns.load();
  const int sr = g_stall_rows.load();
  const int nch = lr_nch(a.d);
  if (nch == 1) ln_bwd_rows_kernel<act_t, 1><<<grid, LR_THREADS, smem, s>>>(a, st, sb, w, sr);
  else if (nch == 2) ln_bwd_rows_kernel<act_t, 2><<<grid, LR_THREADS, smem, s>>>(a, st, sb, w, sr);
  else ln_bwd_rows_kernel<act_t, 4><<<grid, LR_THREADS, smem, s>>>(a, st, sb, w, sr);
  return 0;
}

bool rows_eligible(int rows, int d) { return rows > 0 && d >= 4 && d % 4 == 0 && d <= LR_MAX_D; }

}  // namespace

int ln_fwd_bulk(int act_bf16, const LnFwdArgs& a, cudaStream_t s) {
  if (!rows_eligible(a.rows, a.d) || !aligned16(a.x) || (a.add_src && !aligned16(a.add_src))) return 1;
  return act_bf16 ? ln_fwd_rows<bf16>(a, s) : ln_fwd_rows<float>(a, s);
}

int ln_bwd_bulk(int act_bf16, const LnBwdArgs& a, cudaStream_t s) {
  if (!rows_eligible(a.rows, a.d) || !aligned16(a.x) || !aligned16(a.dy) || (a.dy2 && !aligned16(a.dy2)) ||
      (a.dres && !aligned16(a.dres)))
    return 1;
  const int r = act_bf16 ? ln_bwd_rows<bf16>(a, s) : ln_bwd_rows<float>(a, s);
  if (r) return r;
  if (a.cs_part) {
    const bool sum_dx = a.dxs_out || a.dxs_out2;
    return colsum_finish(a.cs_part, rows_grid(a.rows, a.d), a.d, a.cs_out1, a.cs_out0, nullptr, a.cs_accumulate, s,
                         sum_dx ? 3 : 2, a.dxs_out, a.dxs_out2);
  }
  return 0;
}

void ln_debug_stall(int stall_rows, long long wait_ns) {
  g_stall_rows.store(stall_rows);
  g_wait_ns.store(wait_ns);
}

}  // namespace fal
