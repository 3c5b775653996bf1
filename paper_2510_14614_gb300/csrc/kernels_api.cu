// Kernel-level C ABI (include/fal_kernels.h): single GEMM / attention calls.
#include <cstring>

#include "../../include/fal.h"
#include "../../include/fal_kernels.h"
#include "internal.h"

using namespace fal;

namespace {
int map_rc(int r) { return r == 0 ? FAL_OK : r == 1 ? FAL_ERR_ARG : r == 6 ? FAL_ERR_UNSUPPORTED : FAL_ERR_CUDA; }
}  // namespace

extern "C" {

int fal_kernel_gemm(int M, int N, int K, const void* A, long lda, int a_mn_major, const void* B, long ldb,
                    int b_mn_major, int in_f32, const float* bias, void* C, long ldc, int c_f32, int engine,
                    int* dev_err, void* stream) {
  if (M < 0 || N < 0 || K <= 0 || !A || !B || !C) return FAL_ERR_ARG;
  if (engine != FAL_ENGINE_TCGEN05 && engine != FAL_ENGINE_SIMT && engine != FAL_ENGINE_TCGEN05_PAIR)
    return FAL_ERR_ARG;
  if (engine != FAL_ENGINE_SIMT && in_f32) return FAL_ERR_ARG;
  if (ldc < N || lda < (a_mn_major ? M : K) || ldb < (b_mn_major ? N : K)) return FAL_ERR_ARG;
  if (M == 0 || N == 0) return FAL_OK;
  GemmCall c;
  memset(&c, 0, sizeof(c));
  c.ngroups = 1;
  GemmGroupDesc& g = c.g[0];
  g.M = M; g.N = N; g.nseg = 1;
  g.seg[0].A = {A, lda, a_mn_major ? 1 : 0};
  g.seg[0].B = {B, ldb, b_mn_major ? 1 : 0};
  g.seg[0].K = K;
  g.epi.out = C; g.epi.ldo = ldc; g.epi.out_mode = c_f32 ? OUT_F32 : OUT_ACT; g.epi.bias = bias;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  std::string msg;
  int r = engine == FAL_ENGINE_SIMT ? gemm_simt(c, in_f32 ? 0 : 1, 1, s, &msg)
                                    : gemm_tc_engine(c, engine == FAL_ENGINE_TCGEN05_PAIR ? TC_PAIR : TC_ONE,
                                                     dev_err, s, &msg);
  return map_rc(r);
}

int fal_kernel_attention_fwd(int B, int T, int H, int hd, const void* qkv, void* ctx, float* lse, void* stream) {
  if (B < 0 || T < 0 || H <= 0 || !qkv || !ctx || !lse) return FAL_ERR_ARG;
  std::string msg;
  return map_rc(attn_fwd(1, B, T, H, hd, qkv, ctx, lse, nullptr, reinterpret_cast<cudaStream_t>(stream), &msg));
}

size_t fal_kernel_attention_bwd_scratch(int B, int T, int H, int hd) {
  (void)hd;
  if (B <= 0 || T <= 0 || H <= 0) return 64;
  return fal::attn_bwd_scratch_floats(B, T, H);
}

int fal_kernel_attention_bwd(int B, int T, int H, int hd, const void* qkv, const void* ctx, const float* lse,
                             const void* dctx, void* dqkv, float* scratch, void* stream) {
  if (B < 0 || T < 0 || H <= 0 || !qkv || !ctx || !lse || !dctx || !dqkv || !scratch) return FAL_ERR_ARG;
  std::string msg;
  return map_rc(attn_bwd(1, B, T, H, hd, qkv, ctx, lse, dctx, dqkv, scratch, nullptr,
                         reinterpret_cast<cudaStream_t>(stream),
                         &msg));
}

}  // extern "C"
