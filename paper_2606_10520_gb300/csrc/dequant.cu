// Test hook: W_hat [N][K] in fp32 from the packed device layout.
//
// Each warp unpacks one 16 x 128 tile with the same position-extraction helper
// the layer kernels use (layout.h), rebuilds the vector index of every
// d-vector (coordinate c in bits [2c+1:2c]) and reads the fp32 codeword
// RN_fp32(A z + B) of Eq. (def:unisvq) from the handle's codebook.
#include "common.cuh"
#include "internal.h"

namespace unisvq {
namespace {

__global__ void __launch_bounds__(256) dequant_kernel(const uint8_t* __restrict__ codes,
                                                      const float* __restrict__ lut, float* W,
                                                      int N, int K, int KT, int d, int ntiles) {
  const int tile = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (tile >= ntiles) return;
  const int lane = threadIdx.x & 31;
  const int rt = tile / KT, kt = tile - (tile / KT) * KT;
  const int g = lane >> 2, t = lane & 3;
  const uint4 wv = *reinterpret_cast<const uint4*>(codes + static_cast<size_t>(tile) * kTileBytes + lane * 16);
  const uint32_t words[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int grp = q >> 1, rh = q & 1;
    const int row = rt * kTileRows + g + 8 * rh;
    const uint32_t w = words[q], ws = w >> 10;
    // 4-column groups: i selects the k16 block, positions 2i (cols +0,+1) and 2i+1 (cols +2,+3).
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const uint32_t f0 = extract_pos(w, ws, 2 * i), f1 = extract_pos(w, ws, 2 * i + 1);
      const uint32_t z[4] = {frag_code_lo(f0, 2 * i), frag_code_hi(f0, 2 * i),
                             frag_code_lo(f1, 2 * i + 1), frag_code_hi(f1, 2 * i + 1)};
      const int k0 = kt * kTileCols + 64 * grp + 16 * i + 4 * t;
      if (row >= N) continue;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int k = k0 + e;
        if (k >= K) continue;
        const int v0 = e & ~(d - 1);   // first coordinate of this column's vector
        uint32_t idx = 0;
        for (int c = 0; c < d; ++c) idx |= z[v0 + c] << (2 * c);
        W[static_cast<size_t>(row) * K + k] = lut[idx * d + (e & (d - 1))];
      }
    }
  }
}

}  // namespace

unisvq_status launch_dequant(const unisvq_layer* L, float* W, cudaStream_t s) {
  const int ntiles = (L->Np / kTileRows) * L->KT;
  dequant_kernel<<<(ntiles + 7) / 8, 256, 0, s>>>(L->codes, L->lut32, W, L->N, L->K, L->KT, L->d,
                                                  ntiles);
  return cudaGetLastError() == cudaSuccess ? UNISVQ_OK : UNISVQ_ERR_CUDA;
}

}  // namespace unisvq
