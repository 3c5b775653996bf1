// PTX wrappers used by the attention kernels on top of tc_ptx.cuh: MMAs that
// take each shared-memory descriptor as two 32-bit words (the issuing thread
// builds the constant high word once and steps the low word by immediates
// along K), and the 3-D TMA store of the backward's epilogue.
#pragma once

#include "tc_ptx.cuh"

namespace fal {
namespace ptx {

// High word of a tcgen05 shared-memory descriptor: stride byte offset >> 4,
// version 1 (bit 46 of the descriptor), 128-byte swizzle (bits 61-63 = 2).
__device__ __forceinline__ uint32_t desc_hi(uint32_t sbo) {
  return ((sbo >> 4) & 0x3FFFu) | (1u << 14) | (2u << 29);
}
// Low word: start address >> 4 and leading byte offset >> 4.
__device__ __forceinline__ uint32_t desc_lo(uint32_t saddr, uint32_t lbo) {
  return ((saddr >> 4) & 0x3FFFu) | (((lbo >> 4) & 0x3FFFu) << 16);
}
// D (+)= A B with both operands in shared memory.
__device__ __forceinline__ void tc_mma_w(uint32_t d_tmem, uint32_t a_lo, uint32_t b_lo, uint32_t hi, uint32_t idesc,
                                         uint32_t accum) {
  asm volatile(
      "{\n .reg .pred p;\n .reg .b64 da, db;\n setp.ne.b32 p, %5, 0;\n mov.b64 da, {%1, %3};\n"
      " mov.b64 db, {%2, %3};\n tcgen05.mma.cta_group::1.kind::f16 [%0], da, db, %4, p;\n}\n" ::"r"(d_tmem),
      "r"(a_lo), "r"(b_lo), "r"(hi), "r"(idesc), "r"(accum)
      : "memory");
}
// D (+)= A B with A in TMEM (bf16 pairs) and B in shared memory.
__device__ __forceinline__ void tc_mma_ts_w(uint32_t d_tmem, uint32_t a_tmem, uint32_t b_lo, uint32_t hi, uint32_t idesc,
                                            uint32_t accum) {
  asm volatile(
      "{\n .reg .pred p;\n .reg .b64 db;\n setp.ne.b32 p, %4, 0;\n mov.b64 db, {%2, %3};\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], db, %5, p;\n}\n" ::"r"(d_tmem),
      "r"(a_tmem), "r"(b_lo), "r"(hi), "r"(accum), "r"(idesc)
      : "memory");
}
// TMA store of a shared-memory tile to global memory through a 3-D tensor map.
__device__ __forceinline__ void tma_store_3d(const CUtensorMap* map, uint32_t src, int x, int y, int z) {
  asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(src), "r"(x), "r"(y), "r"(z)
               : "memory");
}

}  // namespace ptx
}  // namespace fal
