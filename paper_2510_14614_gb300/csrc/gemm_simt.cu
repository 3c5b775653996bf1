// Plain fp32-FMA tiled GEMM: the fp32 debug path (no tensor cores, no TF32)
// and a GPU-side cross-check for the tcgen05 GEMM.  Same problem description
// and epilogue as the tensor-core GEMM.
#include "gemm_epi.cuh"

namespace fal {

namespace {

constexpr int SB_M = 64, SB_N = 64, SB_K = 16;

struct SimtParams {
  GemmCall c;
  int tiles[kMaxGemmGroups];  // tiles per group
};

template <typename in_t>
__device__ __forceinline__ float ld_op(const GemmOperand& o, int row, int k, int rows, int K) {
  if (row >= rows || k >= K) return 0.f;
  const in_t* p = reinterpret_cast<const in_t*>(o.ptr);
  return to_f(o.mn_major ? p[(long)k * o.ld + row] : p[(long)row * o.ld + k]);
}

// EPI_CE_STATS of one 64 x 64 tile: every row's maximum and sum of exp(x - max)
// over the tile's columns below N, reduced over the 16 threads that share the
// row (lanes that differ in tx only), and the logit of the row's target.
__device__ __forceinline__ void simt_ce_stats(const EpiParams& e, int M, int N, int m0, int n0, int ty, int tx,
                                              const float (*acc)[4]) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int row = m0 + ty * 4 + i;
    float m = -INFINITY;
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (n0 + tx * 4 + j < N) m = fmaxf(m, acc[i][j]);
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    float s = 0.f;
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (n0 + tx * 4 + j < N) s += __expf(acc[i][j] - m);
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (row < M) {
      if (tx == 0) e.ce_stats[(long)(n0 / kCeSliceSimt) * e.ce_ld + row] = make_float2(m, s);
      const int t = e.ce_tgt[row] - e.ce_v0 - n0 - tx * 4;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (t == j && n0 + tx * 4 + j < N) e.ce_tlogit[row] = acc[i][j];
    }
  }
}

template <typename in_t, typename act_t>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const __grid_constant__ SimtParams p) {
  __shared__ float As[SB_K][SB_M + 4];
  __shared__ float Bs[SB_K][SB_N + 4];
  int tile = blockIdx.x;
  int g = 0;
  while (g + 1 < kMaxGemmGroups && tile >= p.tiles[g]) { tile -= p.tiles[g]; ++g; }
  const GemmGroupDesc& G = p.c.g[g];
  const int mt = (G.M + SB_M - 1) / SB_M;
  const int m0 = (tile % mt) * SB_M, n0 = (tile / mt) * SB_N;
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  float acc[4][4] = {};
  for (int s = 0; s < G.nseg; ++s) {
    const GemmSeg& S = G.seg[s];
    for (int k0 = 0; k0 < S.K; k0 += SB_K) {
      for (int i = threadIdx.x; i < SB_M * SB_K; i += 256) {
        int r, kk;
        if (S.A.mn_major) { r = i % SB_M; kk = i / SB_M; } else { r = i / SB_K; kk = i % SB_K; }
        As[kk][r] = ld_op<in_t>(S.A, m0 + r, k0 + kk, G.M, S.K);
        if (S.B.mn_major) { r = i % SB_N; kk = i / SB_N; } else { r = i / SB_K; kk = i % SB_K; }
        Bs[kk][r] = ld_op<in_t>(S.B, n0 + r, k0 + kk, G.N, S.K);
      }
      __syncthreads();
#pragma unroll
      for (int kk = 0; kk < SB_K; ++kk) {
        float a[4], b[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) { a[i] = As[kk][ty * 4 + i]; b[i] = Bs[kk][tx * 4 + i]; }
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
      }
      __syncthreads();
    }
  }
  if (G.epi.op == EPI_CE_STATS) {
    simt_ce_stats(G.epi, G.M, G.N, m0, n0, ty, tx, acc);
    return;
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) epi_row<act_t, 4>(G.epi, G.M, G.N, m0 + ty * 4 + i, n0 + tx * 4, acc[i]);
}

}  // namespace

int gemm_simt(const GemmCall& c, int in_bf16, int act_bf16, cudaStream_t s, std::string* msg) {
  SimtParams p;
  p.c = c;
  int total = 0;
  if (c.ngroups < 1 || c.ngroups > kMaxGemmGroups) { if (msg) *msg = "GEMM launch needs 1 to 4 groups"; return 1; }
  for (int g = 0; g < kMaxGemmGroups; ++g) {
    p.tiles[g] = 0;
    if (g < c.ngroups) {
      const GemmGroupDesc& G = c.g[g];
      p.tiles[g] = ((G.M + SB_M - 1) / SB_M) * ((G.N + SB_N - 1) / SB_N);
    }
    total += p.tiles[g];
  }
  if (total == 0) return 0;
  if (in_bf16 && act_bf16) gemm_simt_kernel<bf16, bf16><<<total, 256, 0, s>>>(p);
  else if (in_bf16) gemm_simt_kernel<bf16, float><<<total, 256, 0, s>>>(p);
  else if (act_bf16) gemm_simt_kernel<float, bf16><<<total, 256, 0, s>>>(p);
  else gemm_simt_kernel<float, float><<<total, 256, 0, s>>>(p);
  count_launches(1);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) { if (msg) *msg = std::string("gemm_simt launch: ") + cudaGetErrorString(e); return 4; }
  return 0;
}

}  // namespace fal
