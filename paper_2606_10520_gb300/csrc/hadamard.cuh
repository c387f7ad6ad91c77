// Block-local pieces of the Hadamard transform H_n = H_{2^a} (Sylvester)
// Kronecker H_m (Paley) of Eq. def:hadamard, shared by the rotation kernel
// (rht.cu) and the fold kernel's fused input rotation (decode.cu). A row of
// n = p2 * m values is viewed as p2 blocks of m; entry (p, q) sits at p m + q.
// Every helper is run by all NT threads of the CTA on shared memory; the
// caller synchronises between calls.
#pragma once

#include <cstdint>

namespace unisvq {

// Row vector times H_m for every block of M_ consecutive entries of src,
// into dst: four threads per block, each forming M_/4 of its outputs. neg[c]
// has bit q set where H_m[q][c] = -1.
template <int NT, int M_>
__device__ __forceinline__ void paley_blocks(const float* src, float* dst, int nblk, const uint32_t* neg) {
  constexpr int C = M_ / 4;
  for (int it = threadIdx.x; it < nblk * 4; it += NT) {
    const int p = it >> 2, c0 = (it & 3) * C;
    const float* blk = src + p * M_;
    float v[M_];
#pragma unroll
    for (int q = 0; q < M_; ++q) v[q] = blk[q];
#pragma unroll
    for (int c = 0; c < C; ++c) {
      const uint32_t mask = neg[c0 + c];
      float acc = 0.f;
#pragma unroll
      for (int q = 0; q < M_; ++q) acc += ((mask >> q) & 1u) ? -v[q] : v[q];
      dst[p * M_ + c0 + c] = acc;
    }
  }
}

// Sylvester stages s0 .. s0 + R - 1 (butterfly distances 2^s0 .. 2^(s0+R-1)
// blocks) for every column of the p2 x m view, R stages per pass in registers.
template <int NT, int R>
__device__ __forceinline__ void sylvester_pass(float* buf, int p2, int m, int s0) {
  constexpr int G = 1 << R;
  const int h = 1 << s0;
  const int groups = (p2 >> R) * m;
  for (int gi = threadIdx.x; gi < groups; gi += NT) {
    const int col = gi % m, rest = gi / m;
    const int lo = (rest & (h - 1)) | ((rest >> s0) << (s0 + R));   // R zero bits inserted at s0
    float v[G];
#pragma unroll
    for (int j = 0; j < G; ++j) v[j] = buf[(lo + j * h) * m + col];
#pragma unroll
    for (int st = 0; st < R; ++st) {
      const int d = 1 << st;
#pragma unroll
      for (int j = 0; j < G; ++j)
        if (!(j & d)) {
          const float a = v[j], b = v[j + d];
          v[j] = a + b;
          v[j + d] = a - b;
        }
    }
#pragma unroll
    for (int j = 0; j < G; ++j) buf[(lo + j * h) * m + col] = v[j];
  }
}

// The whole Sylvester transform over the p2 blocks of buf, three stages per
// pass, a barrier after each pass.
template <int NT>
__device__ __forceinline__ void sylvester_all(float* buf, int p2, int m) {
  int lg = 0;
  while ((1 << lg) < p2) ++lg;
  for (int s0 = 0; s0 < lg;) {
    const int r = lg - s0 < 3 ? lg - s0 : 3;
    if (r == 3) sylvester_pass<NT, 3>(buf, p2, m, s0);
    else if (r == 2) sylvester_pass<NT, 2>(buf, p2, m, s0);
    else sylvester_pass<NT, 1>(buf, p2, m, s0);
    s0 += r;
    __syncthreads();
  }
}

}  // namespace unisvq
