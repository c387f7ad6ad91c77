// Helpers shared by the register-operand (mma.sync) GEMVs of libunisvq:
// the m16n8k16 fp16 tensor-core instruction, the per-token fp16 scale of the
// folded activations, the guarded 8-wide bf16 activation load and the fp16
// unpacking of stored affine maps.
#pragma once

#include <cuda_fp16.h>

#include "common.cuh"

namespace unisvq {

// D[16 x 8] += A[16 x 16] B[16 x 8], fp16 operands, fp32 accumulators, with
// the standard m16n8k16 register fragments (A row-major, B column-major).
__device__ __forceinline__ void mma_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                          uint2 b) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b.x), "r"(b.y));
}

// 2^P with P = 15 - e, e the binary exponent of bound in [2^(e-1), 2^e): puts
// every value of magnitude <= bound below 2^15, the fp16 range.
__device__ __forceinline__ int token_scale_exp(float bound) {
  if (!(bound > 0.f)) return 0;
  const int e = static_cast<int>(__float_as_uint(bound) >> 23) - 126;
  return max(-100, min(100, 15 - e));
}

// Eight activations x[k .. k+7] of one token as packed bf16 (zero at or past kend).
__device__ __forceinline__ uint4 load_x8(const uint16_t* row, int k, int kend, bool vec8) {
  if (vec8 && k + 7 < kend) return ldg_v4(row + k);
  uint32_t e[8];
#pragma unroll
  for (int q = 0; q < 8; ++q) e[q] = (k + q < kend) ? static_cast<uint32_t>(row[k + q]) : 0u;
  return make_uint4(e[0] | (e[1] << 16), e[2] | (e[3] << 16), e[4] | (e[5] << 16), e[6] | (e[7] << 16));
}

// The low and high fp16 of a 32-bit word as floats (exact).
__device__ __forceinline__ float f16_lo(uint32_t v) {
  return __half2float(__ushort_as_half(static_cast<unsigned short>(v & 0xFFFFu)));
}
__device__ __forceinline__ float f16_hi(uint32_t v) {
  return __half2float(__ushort_as_half(static_cast<unsigned short>(v >> 16)));
}

}  // namespace unisvq
