// Test hook: W_hat [N][K] in fp32 from the packed device layout.
//
// Each thread unpacks the four words of one (row, half) -- 64 codes -- with
// the same extraction helper the layer kernels use (layout.h), adds the high
// bits of 3-bit codes, rebuilds the index z0 | z1 << bits | ... of every
// d-vector and reads the fp32 codeword RN_fp32(A z + B) of Eq. (def:unisvq)
// from the handle's codebook.
#include <cuda_fp16.h>

#include "common.cuh"
#include "internal.h"

namespace unisvq {
namespace {

__global__ void __launch_bounds__(256) dequant_kernel(const uint8_t* __restrict__ codes,
                                                      const uint8_t* __restrict__ hi,
                                                      const float* __restrict__ lut, float* W,
                                                      int N, int K, int KT, int d, int bits, int nchunks) {
  const int id = blockIdx.x * 256 + threadIdx.x;
  if (id >= nchunks) return;
  const int tile = id >> 8;               // 256 (row, half) pairs per tile
  const int h = (id >> 7) & 1, r = id & 127;
  const int rb = tile / KT, kt = tile - rb * KT;
  const int row = rb * kTileRows + r;
  if (row >= N) return;
  const uint8_t* tb = codes + static_cast<size_t>(tile) * kTileBytes;
  uint32_t words[4];
#pragma unroll
  for (int t = 0; t < 4; ++t) words[t] = *reinterpret_cast<const uint32_t*>(tb + tile_word_offset(r, h, t));
#pragma unroll
  for (int wi = 0; wi < 4; ++wi) {
    // The 16 codes of the word: z[4s + b] = column 4s + b (16 consecutive
    // columns, so a d-vector, d <= 8, never leaves the word). 3-bit codes add
    // bit 4b + s of the word's halfword in the high-bit plane as bit 2.
    uint32_t hw = 0;
    if (bits == 3)
      hw = *reinterpret_cast<const uint16_t*>(hi + static_cast<size_t>(tile) * (kTileBytes / 2) +
                                              (r >> 4) * (kUnitBytes / 2) + ((r & 7) * 4 + wi) * 8 +
                                              2 * (2 * h + ((r >> 3) & 1)));
    uint32_t z[16];
#pragma unroll
    for (int s = 0; s < 4; ++s) {
      const uint32_t e = extract4(words[wi], s);   // columns 4s .. 4s+3 of the word
#pragma unroll
      for (int b = 0; b < 4; ++b) z[4 * s + b] = ((e >> (8 * b)) & 3u) | (((hw >> (4 * b + s)) & 1u) << 2);
    }
    const int k0 = kt * kTileCols + 64 * h + 16 * wi;
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const int k = k0 + j;
      if (k >= K) continue;
      const int v0 = j & ~(d - 1);              // first coordinate of this column's vector
      uint32_t idx = 0;
      for (int c = 0; c < d; ++c) idx |= z[v0 + c] << (bits * c);
      W[static_cast<size_t>(row) * K + k] = lut[idx * d + (j & (d - 1))];
    }
  }
}

// Per-(row, group) layers: one thread per weight. Column k of row n is
// coordinate r = k mod d of vector v of group g = k / 128; coordinate c of
// that vector sits at chunk q = c (8/d) + v / 16, quarter t = (v mod 16) / 4,
// byte b = e(v mod 4) of the permuted tile (pack_codes_grouped_host), and
// RN_fp32(sum_c A[n][g][r][c] z_c + B[n][g][r]) is formed exactly in fp64.
__global__ void __launch_bounds__(256) dequant_grouped_kernel(const uint8_t* __restrict__ codes,
                                                              const uint16_t* __restrict__ meta, float* W, int N,
                                                              int K, int KT, int d) {
  const size_t id = static_cast<size_t>(blockIdx.x) * 256 + threadIdx.x;
  if (id >= static_cast<size_t>(N) * K) return;
  const int n = static_cast<int>(id / K), k = static_cast<int>(id % K);
  const int g = k / kTileCols, col = k % kTileCols;
  const int v = col / d, r = col % d, nq = 8 / d;
  const int rb = n / kTileRows, rr = n % kTileRows;
  const uint8_t* tile = codes + (static_cast<size_t>(rb) * KT + g) * kTileBytes;
  const int md = d * d + d;
  const uint16_t* rec = meta + ((static_cast<size_t>(rb) * KT + g) * kTileRows + rr) * md;
  const int q = v / 16, t = (v % 16) / 4, e = v % 4;
  const int b = (e >> 1) | ((e & 1) << 1);
  double w = static_cast<double>(__half2float(__ushort_as_half(rec[d * d + r])));
  for (int c = 0; c < d; ++c) {
    const int qc = c * nq + q;
    const uint32_t word = *reinterpret_cast<const uint32_t*>(tile + tile_word_offset(rr, qc >> 2, t));
    const uint32_t z = (word >> (8 * b + 2 * (qc & 3))) & 3u;
    w += static_cast<double>(__half2float(__ushort_as_half(rec[r * d + c]))) * static_cast<double>(z);
  }
  W[id] = static_cast<float>(w);
}

// Test hook for the unwind path of a bounded wait: one CTA allocates 32
// TMEM columns, starts a bulk copy of `src` (16 bytes) into shared memory
// counted on one mbarrier, and waits on a second mbarrier that nothing
// arrives at. That wait runs out after the library's limit and records
// kErrTimeoutFull; the CTA then waits (bounded) for its own copy, frees TMEM
// and returns, the steps every kernel of the library takes when a wait runs
// out.
__global__ void __launch_bounds__(32) wait_probe_kernel(const uint8_t* src, int* err, int* out) {
  __shared__ __align__(16) uint8_t buf[16];
  __shared__ __align__(8) uint64_t bars[2];
  __shared__ uint32_t tmem_slot;
  const uint32_t copy_bar = smem_u32(&bars[0]), never = smem_u32(&bars[1]);
  if (threadIdx.x == 0) {
    mbar_init(copy_bar, 1);
    mbar_init(never, 1);
    fence_mbar_init();
  }
  __syncwarp();
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 32;" ::"r"(smem_u32(&tmem_slot))
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncwarp();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t taddr = tmem_slot;
  int waited = 0, copied = 0;
  if (threadIdx.x == 0) {
    mbar_arrive_expect_tx(copy_bar, 16);
    bulk_g2s(smem_u32(buf), src, 16, copy_bar, policy_evict_first());
    waited = mbar_wait(never, 0, err, kErrTimeoutFull) ? 1 : 0;    // runs out: nothing arrives
    copied = mbar_wait(copy_bar, 0, err, kErrTimeoutFull) ? 1 : 0;  // the own copy still lands
    out[0] = waited;
    out[1] = copied;
    out[2] = copied ? static_cast<int>(buf[0]) : -1;
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncwarp();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 32;" ::"r"(taddr) : "memory");
}

}  // namespace

unisvq_status launch_dequant(const unisvq_layer* L, float* W, cudaStream_t s) {
  if (L->grouped) {
    const size_t total = static_cast<size_t>(L->N) * L->K;
    dequant_grouped_kernel<<<static_cast<unsigned>((total + 255) / 256), 256, 0, s>>>(L->codes, L->meta, W, L->N,
                                                                                      L->K, L->KT, L->d);
    return cudaGetLastError() == cudaSuccess ? UNISVQ_OK : UNISVQ_ERR_CUDA;
  }
  const int nchunks = (L->Np / kTileRows) * L->KT * 256;
  dequant_kernel<<<(nchunks + 255) / 256, 256, 0, s>>>(L->codes, L->hi, L->lut32, W, L->N, L->K, L->KT, L->d,
                                                       L->bits, nchunks);
  return cudaGetLastError() == cudaSuccess ? UNISVQ_OK : UNISVQ_ERR_CUDA;
}

unisvq_status launch_wait_probe(const void* src16, int* out3, cudaStream_t s) {
  wait_probe_kernel<<<1, 32, 0, s>>>(static_cast<const uint8_t*>(src16), device_error_word(), out3);
  return cudaGetLastError() == cudaSuccess ? UNISVQ_OK : UNISVQ_ERR_CUDA;
}

}  // namespace unisvq
