// Prefill GEMM (M > 32 tokens): tcgen05 tensor cores with the dequantised
// weight tile built in shared memory and never written to HBM.
//
// y[m, n] = sum_k x[m, k] W_hat[n, k] (Eq. def:ptq_loss), W_hat of
// Eq. (col:dequant). One output tile is 128 weight rows x BN tokens:
//   D[128 x BN] (fp32, TMEM) = W_tile[128 x K] (bf16, smem) * x_tile[BN x K]^T
// so the weights are the M=128 operand A and the tokens the N operand B of
// tcgen05.mma.kind::f16, both K-major in the 128-byte swizzled layout.
//
// Roles of the 14 warps of a CTA (persistent over tiles):
//   warp 0        TMA producer: x tile [BN x 64] per k-block, and TMEM owner
//   warp 1        MMA issuer (one thread): 4 x tcgen05.mma (K = 16) per k-block
//   warps 2..9    converters: one 16-row unit per warp, two rows x 16 columns
//                 per lane; every d-vector index selects its exact bf16
//                 codeword RN(A z + B) from a pack-time table (per-matrix
//                 maps, d <= 4; for d = 8 the sum of two quad-table rows,
//                 fp32), or from a table of the row's map that the warp
//                 builds for every 128-column group (per-group maps, d = 2),
//                 or as A z + B from the row's map (per-group maps, d = 4)
//   warps 10..13  epilogue: tcgen05.ld of the accumulator, bf16, global store
// The accumulator is double-buffered in TMEM so the epilogue of one tile runs
// under the main loop of the next.
#include <cudaTypedefs.h>

#include <type_traits>

#include "common.cuh"
#include "mma_sync.cuh"
#include "internal.h"

namespace unisvq {
namespace {

// Warps: TMA producer, MMA issuer, NCONV converters (8, or 16 for per-matrix
// 2-bit layers with d <= 4), four epilogue warps.
__host__ __device__ constexpr int pf_threads(int nconv) { return (2 + nconv + 4) * 32; }
constexpr int kPfThreads = pf_threads(8);
constexpr int kBM = 128;
constexpr int kBK = 64;                  // bf16 columns per stage (one 128B swizzle row)
constexpr int kATileBytes = kBM * 128;   // 16 KB
constexpr int kConvWarp0 = 2;
constexpr int kCodeAhead = 8;   // stages of codes in flight per converter lane (8: 1081 vs 1066 TFLOP/s for 3)

// Layers of one launch (several only for 2-bit layers with one d <= 4 that
// read the same x, all per-matrix or all per-group): their tiles are numbered
// one layer after the other, layer i from tile0[i] on; a per-matrix layer
// keeps its codeword table in a 2 KB slot of shared memory, a per-group layer
// has its own maps.
constexpr int kPfMaxLayers = UNISVQ_MAX_GROUP;

struct PrefillArgs {
  const uint8_t* codes[kPfMaxLayers];
  // d <= 2: 16 x bf16x2 pair codewords (3-bit: 64); d == 4: 256 x 4 bf16 (3-bit: [2][64][4] fp32
  // pair tables); d == 8: [2][256][8] fp32 quad tables
  const uint32_t* lut[kPfMaxLayers];
  uint16_t* y[kPfMaxLayers];
  int N[kPfMaxLayers];
  int tile0[kPfMaxLayers];
  int nlayers;
  // per-group layers: fp16 [Np/128][KT][128][d*d + d] (A row-major, B) per layer, else null
  const uint16_t* meta[kPfMaxLayers];
  const uint8_t* hi;     // 3-bit codes (d <= 2): the high-bit plane; the table has 64 pairs, index z0 | z1 << 3
  int M, K, KT, d;
  int nkb;               // k-blocks of 64 columns: ceil(K / 64)
  int mtiles, tiles;
  int* err;
};

// The launch's layer of a tile (constant parameter offsets only).
__device__ __forceinline__ int tile_layer(const PrefillArgs& a, int tile) {
  int li = 0;
#pragma unroll
  for (int i = 1; i < kPfMaxLayers; ++i)
    if (i < a.nlayers && tile >= a.tile0[i]) li = i;
  return li;
}
template <class T>
__device__ __forceinline__ T pick_layer(const T (&v)[kPfMaxLayers], int li) {
  T r = v[0];
#pragma unroll
  for (int i = 1; i < kPfMaxLayers; ++i)
    if (i == li) r = v[i];
  return r;
}

template <int BN, int STAGES>
struct PfCfg {
  static constexpr int kBTileBytes = BN * 128;
  static constexpr int kStageBytes = kATileBytes + kBTileBytes;
  static constexpr int kOffA = 0;
  static constexpr int kOffB = STAGES * kATileBytes;
  static constexpr int kOffLut = STAGES * kStageBytes;            // 2 KB (d = 8: the 16 KB region)
  static constexpr int kOffGrp = kOffLut + 2048;                   // 8 x 1 KB: per-group tables
  static constexpr int kOffBars = kOffLut + 20 * 1024;            // per-group d = 8: 8 x 2304 B of maps
  // bars: bfull[S], afull[S], empty[S], accfull[2], accempty[2]
  static constexpr int kOffTmemPtr = kOffBars + (3 * STAGES + 5) * 8;   // + drain barrier
  static constexpr int kOffFlag = kOffTmemPtr + 8;
  static constexpr int kSmem = kOffFlag + 8 + 1024;                // + alignment slack
  static constexpr uint32_t kTmemCols = 2 * BN < 32 ? 32 : 2 * BN;
};

// ---- tcgen05 / TMA wrappers --------------------------------------------------

__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, rows of
// 128 bytes, 8-row core groups 1024 bytes apart (SBO), version 1 (sm_100+).
__device__ __forceinline__ uint64_t make_sw128_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);       // start address
  d |= static_cast<uint64_t>(1) << 16;                       // LBO (unused for swizzled K-major)
  d |= static_cast<uint64_t>(1024 >> 4) << 32;               // SBO
  d |= static_cast<uint64_t>(1) << 46;                       // descriptor version
  d |= static_cast<uint64_t>(2) << 61;                       // SWIZZLE_128B
  return d;
}

// Instruction descriptor, kind::f16: D f32, A and B bf16, both K-major, M = 128.
template <int BN>
__device__ __forceinline__ uint32_t make_idesc() {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(BN >> 3) << 17) |
         (static_cast<uint32_t>(kBM >> 4) << 24);
}

__device__ __forceinline__ void mma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                         uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int c0, int c1,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar)
      : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]),
        "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]),
        "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void sts128(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}
__device__ __forceinline__ void sts64(uint32_t addr, uint32_t a, uint32_t b) {
  asm volatile("st.shared.v2.b32 [%0], {%1, %2};" ::"r"(addr), "r"(a), "r"(b) : "memory");
}
__device__ __forceinline__ uint32_t lds32(uint32_t addr) {
  uint32_t v;
  asm volatile("ld.shared.b32 %0, [%1];" : "=r"(v) : "r"(addr));
  return v;
}
__device__ __forceinline__ void sts32(uint32_t addr, uint32_t v) {
  asm volatile("st.shared.b32 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}
__device__ __forceinline__ uint2 lds64(uint32_t addr) {
  uint2 v;
  asm volatile("ld.shared.v2.b32 {%0, %1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(addr));
  return v;
}
__device__ __forceinline__ float4 lds128f(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(addr));
  return v;
}

template <int BN, int STAGES, int NCONV>
__global__ void __launch_bounds__(pf_threads(NCONV), 1)
    prefill_kernel(const __grid_constant__ CUtensorMap tmap_x, const __grid_constant__ PrefillArgs a) {
  using C = PfCfg<BN, STAGES>;
  constexpr int kEpiWarp0 = kConvWarp0 + NCONV;
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte alignment for the 128B-swizzled tiles.
  const uint32_t raw_addr = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024 - (raw_addr & 1023)) & 1023);
  const uint32_t sbase = smem_u32(smem);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t bar0 = sbase + C::kOffBars;
  auto bfull = [&](int s) { return bar0 + 8u * s; };
  auto afull = [&](int s) { return bar0 + 8u * (STAGES + s); };
  auto empty = [&](int s) { return bar0 + 8u * (2 * STAGES + s); };
  auto accfull = [&](int b) { return bar0 + 8u * (3 * STAGES + b); };
  auto accempty = [&](int b) { return bar0 + 8u * (3 * STAGES + 2 + b); };
  const uint32_t drain = bar0 + 8u * (3 * STAGES + 4);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::kOffFlag);
  uint32_t* tmem_ptr = reinterpret_cast<uint32_t*>(smem + C::kOffTmemPtr);

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(bfull(s), 1);
      mbar_init(afull(s), NCONV);
      mbar_init(empty(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(accfull(b), 1);
      mbar_init(accempty(b), 4);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmap_x)) : "memory");
  }
  // Codeword table -> shared memory (per-matrix maps only; per-group layers
  // build theirs in the converters).
  if (!a.meta[0]) {   // layer i's table at kOffLut + 2 KB i (one layer for d = 8: 16 KB)
    const int words = a.hi ? (a.d == 4 ? 512 : 64) : (a.d == 8 ? 4096 : (a.d == 4 ? 512 : 16));
#pragma unroll
    for (int l = 0; l < kPfMaxLayers; ++l) {
      if (l < a.nlayers) {
        uint32_t* lut_s = reinterpret_cast<uint32_t*>(smem + C::kOffLut + 2048 * l);
        const uint32_t* src = a.lut[l];
        for (int i = threadIdx.x; i < words; i += pf_threads(NCONV)) lut_s[i] = src[i];
      }
    }
  }
  if (warp == 0) {
    tmem_alloc(sbase + C::kOffTmemPtr, C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_ptr;

  if (warp == 0) {
    // ---------------- TMA producer: activations ----------------
    if (lane == 0) {
      int it = 0;
      for (int tile = blockIdx.x; tile < a.tiles && !*abort_flag; tile += gridDim.x) {
        const int m0 = ((tile - pick_layer(a.tile0, tile_layer(a, tile))) % a.mtiles) * BN;
        for (int kb = 0; kb < a.nkb; ++kb, ++it) {
          const int s = it % STAGES;
          if (it >= STAGES && !mbar_wait(empty(s), ((it / STAGES) - 1) & 1, a.err, kErrTimeoutEmpty)) {
            *abort_flag = 1;
            break;
          }
          mbar_arrive_expect_tx(bfull(s), C::kBTileBytes);
          tma_load_2d(sbase + C::kOffB + s * C::kBTileBytes, &tmap_x, kb * kBK, m0, bfull(s));
        }
      }
      // After an abort, loads nobody consumed must still land before exit.
      if (*abort_flag)
        for (int j = it - STAGES > 0 ? it - STAGES : 0; j < it; ++j)
          mbar_wait(bfull(j % STAGES), (j / STAGES) & 1, a.err, kErrTimeoutFull);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      const uint32_t idesc = make_idesc<BN>();
      int it = 0, lt = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < a.tiles && ok; tile += gridDim.x, ++lt) {
        const int b = lt & 1;
        if (lt >= 2) {
          ok = mbar_wait(accempty(b), ((lt >> 1) - 1) & 1, a.err, kErrTimeoutAcc);
          if (!ok) break;
        }
        tc_fence_after();
        const uint32_t dcol = tmem_base + static_cast<uint32_t>(b * BN);
        for (int kb = 0; kb < a.nkb; ++kb, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (it / STAGES) & 1;
          ok = !*abort_flag && mbar_wait(bfull(s), ph, a.err, kErrTimeoutFull) &&
               mbar_wait(afull(s), ph, a.err, kErrTimeoutFull);
          if (!ok) break;
          tc_fence_after();
          const uint64_t ad = make_sw128_desc(sbase + C::kOffA + s * kATileBytes);
          const uint64_t bd = make_sw128_desc(sbase + C::kOffB + s * C::kBTileBytes);
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)   // +32 bytes per K=16 step inside the swizzle row
            mma_bf16(dcol, ad + 2 * k, bd + 2 * k, idesc, (kb > 0 || k > 0) ? 1u : 0u);
          mma_commit(empty(s));
        }
        if (!ok) break;
        mma_commit(accfull(b));
      }
      if (!ok) *abort_flag = 1;
      // Everything issued so far must retire before TMEM is released.
      mma_commit(drain);
      mbar_wait(drain, 0, a.err, kErrTimeoutMma);
    }
  } else if (NCONV == 16 && warp < kEpiWarp0) {
    // ---------------- converters, 16 warps (per-matrix maps, 2-bit, d <= 4) ----------------
    // Warp c covers row half hr = c / 8 of unit u = c % 8: lane 4g + t converts
    // row 16u + g + 8hr, column quarter t of the stage's half, i.e. the chunks
    // 2t and 2t + 1 of that row (one code word per stage).
    const int c = warp - kConvWarp0, u = c & 7, hr = c >> 3;
    const int g = lane >> 2, t = lane & 3;
    const int r = 16 * u + g + 8 * hr;
    const uint32_t lut_base = sbase + C::kOffLut;   // layer i's table at + 2 KB i
    int it = 0;
    for (int tile = blockIdx.x; tile < a.tiles; tile += gridDim.x) {
      const int li = tile_layer(a, tile);
      const int n_blk = (tile - pick_layer(a.tile0, li)) / a.mtiles;
      // word (h, hr) of the lane's 16-byte chunk: byte 4 (2h + hr)
      const uint8_t* rbase = pick_layer(a.codes, li) + static_cast<size_t>(n_blk) * a.KT * kTileBytes +
                             u * kUnitBytes + lane * 16 + 4 * hr;
      const uint32_t lut_s = lut_base + 2048u * static_cast<uint32_t>(li);
      auto load = [&](int kb) -> uint32_t {
        return kb < a.nkb ? __ldg(reinterpret_cast<const uint32_t*>(rbase + (kb >> 1) * kTileBytes + (kb & 1) * 8))
                          : 0u;
      };
      uint32_t qr[kCodeAhead];
#pragma unroll
      for (int j = 0; j < kCodeAhead; ++j) qr[j] = load(j);
      bool ok = !*abort_flag;
      for (int kb0 = 0; kb0 < a.nkb; kb0 += kCodeAhead) {
#pragma unroll
        for (int j = 0; j < kCodeAhead; ++j) {
          const int kb = kb0 + j;
          if (kb >= a.nkb) break;
          const int s = it % STAGES;
          const uint32_t w = qr[j];
          qr[j] = load(kb + kCodeAhead);   // refill the slot just read
          if (ok && it >= STAGES) {
            ok = !*abort_flag && mbar_wait(empty(s), ((it / STAGES) - 1) & 1, a.err, kErrTimeoutEmpty);
            if (!ok) *abort_flag = 1;
          }
          if (ok) {
            const uint32_t row_addr = sbase + C::kOffA + s * kATileBytes + r * 128;
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int cc = 2 * t + e;                       // chunk: stage columns 8cc .. 8cc+7
              const uint32_t e0 = extract4(w, 2 * e);         // columns 8cc .. 8cc+3
              const uint32_t e1 = extract4(w, 2 * e + 1);     // columns 8cc+4 .. 8cc+7
              uint32_t o0, o1, o2, o3;
              if (a.d == 4) {
                const uint32_t i0 = (e0 & 3u) | ((e0 >> 6) & 0xCu) | ((e0 >> 12) & 0x30u) | ((e0 >> 18) & 0xC0u);
                const uint32_t i1 = (e1 & 3u) | ((e1 >> 6) & 0xCu) | ((e1 >> 12) & 0x30u) | ((e1 >> 18) & 0xC0u);
                const uint2 v0 = lds64(lut_s + i0 * 8), v1 = lds64(lut_s + i1 * 8);
                o0 = v0.x; o1 = v0.y; o2 = v1.x; o3 = v1.y;
              } else {
                o0 = lds32(lut_s + (((e0 & 3u) | ((e0 >> 6) & 0xCu)) << 2));
                o1 = lds32(lut_s + ((((e0 >> 16) & 3u) | ((e0 >> 22) & 0xCu)) << 2));
                o2 = lds32(lut_s + (((e1 & 3u) | ((e1 >> 6) & 0xCu)) << 2));
                o3 = lds32(lut_s + ((((e1 >> 16) & 3u) | ((e1 >> 22) & 0xCu)) << 2));
              }
              sts128(row_addr + ((cc ^ g) << 4), o0, o1, o2, o3);
            }
            fence_proxy_async_smem();
          }
          __syncwarp();
          if (lane == 0 && ok) mbar_arrive(afull(s));
          ++it;
        }
      }
    }
  } else if (NCONV == 8 && warp < kEpiWarp0) {
    // ---------------- converters: codes -> bf16 codeword tile ----------------
    // Warp c covers unit c (rows 16c .. 16c+15): lane 4g + t reads the 8-byte
    // pair of words of rows 16c + g and 16c + g + 8 for column quarter t of the
    // stage's half (layout.h) and writes their 16 columns of each row.
    const int c = warp - kConvWarp0;
    const int g = lane >> 2, t = lane & 3;
    const int r0 = 16 * c + g, r1 = r0 + 8;
    const uint32_t lut_base = sbase + C::kOffLut;   // layer i's table at + 2 KB i
    int it = 0;
    if (a.meta[0] && a.d == 8) {
      // Per-(row, 128-column group) maps, d = 8, codes permuted within each group
      // (pack_codes_grouped_host): packed position (h, t, s, b) holds coordinate
      // 4 h + s of vector v = 4 t + e(b), natural columns 8 v .. 8 v + 7. So a
      // lane's 16-byte load holds every coordinate of four vectors of rows g and
      // g + 8, all in stage half t / 2. Lanes t and t ^ 2 share the work: in
      // stage half hs the lane with t / 2 == hs forms the vectors of bytes
      // b = 0, 1 from its own words, its partner those of b = 2, 3 from the
      // same words (one shuffle per word and k-tile). Each output is
      // sum_c' A[c][c'] z_c' + B[c] in fp32 (one 16-byte store per vector); the
      // warp stages its 16 rows' maps (72 fp16 each) in shared memory per k-tile.
      const uint32_t map_s = sbase + C::kOffLut + c * 2304;   // [16 rows][72] fp16
      for (int tile = blockIdx.x; tile < a.tiles; tile += gridDim.x) {
        const int li = tile_layer(a, tile);
        const int n_blk = (tile - pick_layer(a.tile0, li)) / a.mtiles;
        const uint8_t* rbase =
            pick_layer(a.codes, li) + static_cast<size_t>(n_blk) * a.KT * kTileBytes + c * kUnitBytes + lane * 16;
        const uint32_t* mbase = reinterpret_cast<const uint32_t*>(pick_layer(a.meta, li) +
                                                                  static_cast<size_t>(n_blk) * a.KT * kBM * 72 +
                                                                  static_cast<size_t>(16 * c) * 72);
        const int nkt = (a.nkb + 1) >> 1;
        auto load_codes = [&](int kt) -> uint4 {
          return kt < nkt ? __ldg(reinterpret_cast<const uint4*>(rbase + static_cast<size_t>(kt) * kTileBytes))
                          : make_uint4(0, 0, 0, 0);
        };
        // this lane's 18 of the 576 words of the warp's 16 row maps of group kt
        auto load_maps = [&](int kt, uint32_t (&w)[18]) {
#pragma unroll
          for (int i = 0; i < 18; ++i)
            w[i] = kt < nkt ? __ldg(mbase + static_cast<size_t>(kt) * kBM * 36 + lane + 32 * i) : 0u;
        };
        uint4 cn = load_codes(0), own = cn, par = cn;
        uint32_t mw[18];
        load_maps(0, mw);
        bool ok = !*abort_flag;
        for (int kb = 0; kb < a.nkb; ++kb, ++it) {
          const int s = it % STAGES;
          const int hs = kb & 1;
          if (hs == 0) {
            own = cn;
            par.x = __shfl_xor_sync(0xffffffffu, own.x, 2);
            par.y = __shfl_xor_sync(0xffffffffu, own.y, 2);
            par.z = __shfl_xor_sync(0xffffffffu, own.z, 2);
            par.w = __shfl_xor_sync(0xffffffffu, own.w, 2);
            __syncwarp();   // every lane is done with the previous group's maps
#pragma unroll
            for (int i = 0; i < 18; ++i) sts32(map_s + (lane + 32 * i) * 4, mw[i]);
            __syncwarp();
            cn = load_codes((kb >> 1) + 1);
            load_maps((kb >> 1) + 1, mw);
          }
          if (ok && it >= STAGES) {
            ok = !*abort_flag && mbar_wait(empty(s), ((it / STAGES) - 1) & 1, a.err, kErrTimeoutEmpty);
            if (!ok) *abort_flag = 1;
          }
          if (ok) {
            const uint32_t tile_addr = sbase + C::kOffA + s * kATileBytes;
            const bool mine = (t >> 1) == hs;                    // own words, bytes 0, 1; else the partner's, 2, 3
            const int tq = mine ? t : (t ^ 2);                   // the quarter whose vectors this lane forms
            const uint4 src = mine ? own : par;
#pragma unroll
            for (int q = 0; q < 2; ++q) {
              const uint32_t wh[2] = {q ? src.y : src.x, q ? src.w : src.z};   // halves 0 and 1 of the row
              const uint32_t row_addr = tile_addr + (q ? r1 : r0) * 128;
              const uint32_t rec = map_s + (g + 8 * q) * 144;
              float z[2][8];
#pragma unroll
              for (int jb = 0; jb < 2; ++jb) {
                const int bb = mine ? jb : 2 + jb;
#pragma unroll
                for (int cc2 = 0; cc2 < 8; ++cc2)
                  z[jb][cc2] = static_cast<float>((wh[cc2 >> 2] >> (8 * bb + 2 * (cc2 & 3))) & 3u);
              }
              float w[2][8];
#pragma unroll
              for (int cr = 0; cr < 8; ++cr) {
                const uint32_t bw = lds32(rec + 128 + 4 * (cr >> 1));
                const float bc = (cr & 1) ? f16_hi(bw) : f16_lo(bw);
                float ar[8];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                  const uint32_t aw = lds32(rec + 16 * cr + 4 * i);
                  ar[2 * i] = f16_lo(aw);
                  ar[2 * i + 1] = f16_hi(aw);
                }
#pragma unroll
                for (int jb = 0; jb < 2; ++jb) {
                  float acc = bc;
#pragma unroll
                  for (int c2 = 0; c2 < 8; ++c2) acc = fmaf(ar[c2], z[jb][c2], acc);
                  w[jb][cr] = acc;
                }
              }
#pragma unroll
              for (int jb = 0; jb < 2; ++jb) {
                const int bb = mine ? jb : 2 + jb;
                const int ev = (bb >> 1) | ((bb & 1) << 1);     // vector 4 tq + e(b): chunk 4 (tq & 1) + e(b)
                const int cc = 4 * (tq & 1) + ev;
                sts128(row_addr + ((cc ^ g) << 4), pack_bf16x2(w[jb][0], w[jb][1]), pack_bf16x2(w[jb][2], w[jb][3]),
                       pack_bf16x2(w[jb][4], w[jb][5]), pack_bf16x2(w[jb][6], w[jb][7]));
              }
            }
            fence_proxy_async_smem();
          }
          __syncwarp();
          if (lane == 0 && ok) mbar_arrive(afull(s));
        }
      }
    } else if (a.meta[0] && a.d == 4) {
      // Per-(row, 128-column group) maps, d = 4: 256 codewords per row and group
      // are too many to tabulate per k-tile, so each output is formed directly,
      // sum_c' A[c][c'] z_c' + B[c] in fp32. Natural columns 64 h + 8 cc + j
      // (cc = 2t, 2t + 1: the lane's own chunks) are vector 16 h + 2 cc + j/4,
      // coordinate c = j mod 4; its coordinate c' sits in the word of half c'/2
      // at shift 2 (c' mod 2) + h and byte e(2 (cc mod 2) + j/4), quarter t. The
      // warp stages its 16 rows' maps (20 fp16 each, 640 contiguous bytes) in
      // shared memory once per k-tile.
      const uint32_t map_s = sbase + C::kOffGrp + c * 1024;   // [16 rows][20] fp16
      for (int tile = blockIdx.x; tile < a.tiles; tile += gridDim.x) {
        const int li = tile_layer(a, tile);
        const int n_blk = (tile - pick_layer(a.tile0, li)) / a.mtiles;
        const uint8_t* rbase =
            pick_layer(a.codes, li) + static_cast<size_t>(n_blk) * a.KT * kTileBytes + c * kUnitBytes + lane * 16;
        const uint32_t* mbase = reinterpret_cast<const uint32_t*>(pick_layer(a.meta, li) + static_cast<size_t>(n_blk) * a.KT * kBM * 20 +
                                                                  static_cast<size_t>(16 * c) * 20);
        const int nkt = (a.nkb + 1) >> 1;
        auto load_codes = [&](int kt) -> uint4 {
          return kt < nkt ? __ldg(reinterpret_cast<const uint4*>(rbase + static_cast<size_t>(kt) * kTileBytes))
                          : make_uint4(0, 0, 0, 0);
        };
        // this lane's 5 of the 160 words of the warp's 16 row maps of group kt
        auto load_maps = [&](int kt, uint32_t (&w)[5]) {
#pragma unroll
          for (int i = 0; i < 5; ++i)
            w[i] = kt < nkt ? __ldg(mbase + static_cast<size_t>(kt) * kBM * 10 + lane + 32 * i) : 0u;
        };
        uint4 cn = load_codes(0), cur = cn;
        uint32_t mw[5];
        load_maps(0, mw);
        float am[2][16], bm[2][4];   // the maps of rows r0, r1 for the current group
        bool ok = !*abort_flag;
        for (int kb = 0; kb < a.nkb; ++kb, ++it) {
          const int s = it % STAGES;
          const int hs = kb & 1;
          if (hs == 0) {
            cur = cn;
            __syncwarp();   // the previous group's maps are in registers already
#pragma unroll
            for (int i = 0; i < 5; ++i) sts32(map_s + (lane + 32 * i) * 4, mw[i]);
            __syncwarp();
            cn = load_codes((kb >> 1) + 1);
            load_maps((kb >> 1) + 1, mw);
#pragma unroll
            for (int q = 0; q < 2; ++q) {
              const uint32_t rec = map_s + (g + 8 * q) * 40;
#pragma unroll
              for (int i = 0; i < 8; ++i) {
                const uint32_t w = lds32(rec + 4 * i);
                am[q][2 * i] = f16_lo(w);
                am[q][2 * i + 1] = f16_hi(w);
              }
#pragma unroll
              for (int i = 0; i < 2; ++i) {
                const uint32_t w = lds32(rec + 32 + 4 * i);
                bm[q][2 * i] = f16_lo(w);
                bm[q][2 * i + 1] = f16_hi(w);
              }
            }
          }
          if (ok && it >= STAGES) {
            ok = !*abort_flag && mbar_wait(empty(s), ((it / STAGES) - 1) & 1, a.err, kErrTimeoutEmpty);
            if (!ok) *abort_flag = 1;
          }
          if (ok) {
            const uint32_t tile_addr = sbase + C::kOffA + s * kATileBytes;
#pragma unroll
            for (int q = 0; q < 2; ++q) {
              const uint32_t wh[2] = {q ? cur.y : cur.x, q ? cur.w : cur.z};   // halves 0 and 1 of the row
              const uint32_t row_addr = tile_addr + (q ? r1 : r0) * 128;
#pragma unroll
              for (int u = 0; u < 2; ++u) {
                const int cc = 2 * t + u;
                uint32_t o[4];
#pragma unroll
                for (int vv = 0; vv < 2; ++vv) {
                  const int e = 2 * u + vv;
                  const int bsh = 8 * ((e >> 1) | ((e & 1) << 1));
                  float z[4];
#pragma unroll
                  for (int c2 = 0; c2 < 4; ++c2)
                    z[c2] = static_cast<float>((wh[c2 >> 1] >> (bsh + 2 * (2 * (c2 & 1) + hs))) & 3u);
                  float w[4];
#pragma unroll
                  for (int cr = 0; cr < 4; ++cr)
                    w[cr] = fmaf(am[q][4 * cr + 3], z[3],
                                 fmaf(am[q][4 * cr + 2], z[2], fmaf(am[q][4 * cr + 1], z[1], fmaf(am[q][4 * cr], z[0], bm[q][cr]))));
                  o[2 * vv] = pack_bf16x2(w[0], w[1]);
                  o[2 * vv + 1] = pack_bf16x2(w[2], w[3]);
                }
                sts128(row_addr + ((cc ^ g) << 4), o[0], o[1], o[2], o[3]);
              }
            }
            fence_proxy_async_smem();
          }
          __syncwarp();
          if (lane == 0 && ok) mbar_arrive(afull(s));
        }
      }
    } else if (a.meta[0] && a.d == 1) {
      // Per-(row, 128-column group) maps, d = 1, codes permuted within each group
      // (pack_codes_grouped_host): packed position (h, t, s, b) holds group
      // column 64 h + 16 s + 4 t + e(b). So stage half h needs the words of half
      // h only, and lane t's word of a row gives, for each s, the natural
      // columns 16 s + 4 t + j (j = e(b); e swaps b = 1 and 2) of the stage:
      // 8 bytes of the 16-byte chunk 2 s + t/2. Per k-tile the warp builds, for
      // each of its 16 rows, the 16 bf16 pairs (a z0 + b, a z1 + b) of the
      // row's map (four entries per lane and row); the columns j, j + 1 (bytes
      // e(j), e(j + 1)) index it.
      const uint32_t tab_s = sbase + C::kOffGrp + c * 1024;   // [16 rows][16 entries] bf16x2
      for (int tile = blockIdx.x; tile < a.tiles; tile += gridDim.x) {
        const int li = tile_layer(a, tile);
        const int n_blk = (tile - pick_layer(a.tile0, li)) / a.mtiles;
        const uint8_t* rbase =
            pick_layer(a.codes, li) + static_cast<size_t>(n_blk) * a.KT * kTileBytes + c * kUnitBytes + lane * 16;
        const uint16_t* mbase = pick_layer(a.meta, li) + static_cast<size_t>(n_blk) * a.KT * kBM * 2;
        const int nkt = (a.nkb + 1) >> 1;
        auto load_codes = [&](int kt) -> uint4 {
          return kt < nkt ? __ldg(reinterpret_cast<const uint4*>(rbase + static_cast<size_t>(kt) * kTileBytes))
                          : make_uint4(0, 0, 0, 0);
        };
        // a row's map (a, b) as one word
        auto load_map = [&](int kt, int row) -> uint32_t {
          return kt < nkt ? __ldg(reinterpret_cast<const uint32_t*>(mbase + (static_cast<size_t>(kt) * kBM + row) * 2))
                          : 0u;
        };
        uint4 cn = load_codes(0), cur = cn;
        uint32_t mn0 = load_map(0, r0), mn1 = load_map(0, r1);
        bool ok = !*abort_flag;
        for (int kb = 0; kb < a.nkb; ++kb, ++it) {
          const int s = it % STAGES;
          const int hs = kb & 1;
          if (hs == 0) {
            cur = cn;
            const uint32_t m0 = mn0, m1 = mn1;
            cn = load_codes((kb >> 1) + 1);
            mn0 = load_map((kb >> 1) + 1, r0);
            mn1 = load_map((kb >> 1) + 1, r1);
            __syncwarp();   // every lane is done with the previous group's table
#pragma unroll
            for (int q = 0; q < 2; ++q) {
              const uint32_t m = q ? m1 : m0;
              const float am = f16_lo(m), bm = f16_hi(m);
              const int rr = g + 8 * q;
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                const int idx = 4 * t + k;
                const float z0 = static_cast<float>(idx & 3), z1 = static_cast<float>(idx >> 2);
                sts32(tab_s + (rr * 16 + idx) * 4, pack_bf16x2(fmaf(am, z0, bm), fmaf(am, z1, bm)));
              }
            }
            __syncwarp();
          }
          if (ok && it >= STAGES) {
            ok = !*abort_flag && mbar_wait(empty(s), ((it / STAGES) - 1) & 1, a.err, kErrTimeoutEmpty);
            if (!ok) *abort_flag = 1;
          }
          if (ok) {
            const uint32_t tile_addr = sbase + C::kOffA + s * kATileBytes;
#pragma unroll
            for (int q = 0; q < 2; ++q) {
              const uint32_t w = hs ? (q ? cur.w : cur.z) : (q ? cur.y : cur.x);   // half hs of the row
              const uint32_t row_addr = tile_addr + (q ? r1 : r0) * 128;
              const uint32_t trow = tab_s + (g + 8 * q) * 64;
#pragma unroll
              for (int sq = 0; sq < 4; ++sq) {
                const uint32_t i0 = ((w >> (2 * sq)) & 3u) | (((w >> (16 + 2 * sq)) & 3u) << 2);       // columns j = 0, 1
                const uint32_t i1 = ((w >> (8 + 2 * sq)) & 3u) | (((w >> (24 + 2 * sq)) & 3u) << 2);  // j = 2, 3
                const int cc = 2 * sq + (t >> 1);
                sts64(row_addr + ((cc ^ g) << 4) + ((t & 1) << 3), lds32(trow + i0 * 4), lds32(trow + i1 * 4));
              }
            }
            fence_proxy_async_smem();
          }
          __syncwarp();
          if (lane == 0 && ok) mbar_arrive(afull(s));
        }
      }
    } else if (a.meta[0]) {
      // Per-(row, 128-column group) maps, d = 2, codes permuted within each group
      // (pack_codes_grouped_host): coordinate c of vector v = 16 s + 4 t + e(b)
      // sits in the word of half c at shift s and byte b. The A tile keeps the
      // natural column order, so lane t writes the chunks t and t + 4 of a stage:
      // natural columns 64 h + 8 cc + j are vector 32 h + 4 cc + j/2 (quarter t,
      // shift 2h + cc/4, byte e(j/2)), coordinate j mod 2 -- all in the lane's own
      // 16-byte load. Per k-tile the warp builds, for each of its 16 rows, the 16
      // bf16 pairs RN(A z + B) of the row's map (four entries per lane and row).
      const uint32_t tab_s = sbase + C::kOffGrp + c * 1024;   // [16 rows][16 entries] bf16x2
      for (int tile = blockIdx.x; tile < a.tiles; tile += gridDim.x) {
        const int li = tile_layer(a, tile);
        const int n_blk = (tile - pick_layer(a.tile0, li)) / a.mtiles;
        const uint8_t* rbase =
            pick_layer(a.codes, li) + static_cast<size_t>(n_blk) * a.KT * kTileBytes + c * kUnitBytes + lane * 16;
        const uint16_t* mbase = pick_layer(a.meta, li) + static_cast<size_t>(n_blk) * a.KT * kBM * 6;
        const int nkt = (a.nkb + 1) >> 1;
        auto load_codes = [&](int kt) -> uint4 {
          return kt < nkt ? __ldg(reinterpret_cast<const uint4*>(rbase + static_cast<size_t>(kt) * kTileBytes))
                          : make_uint4(0, 0, 0, 0);
        };
        // the six fp16 of a row's map, as three words
        auto load_map = [&](int kt, int row) -> uint3 {
          if (kt >= nkt) return make_uint3(0, 0, 0);
          const uint32_t* m = reinterpret_cast<const uint32_t*>(mbase + (static_cast<size_t>(kt) * kBM + row) * 6);
          return make_uint3(__ldg(m), __ldg(m + 1), __ldg(m + 2));
        };
        uint4 cn = load_codes(0), cur = cn;
        uint3 mn0 = load_map(0, r0), mn1 = load_map(0, r1);
        bool ok = !*abort_flag;
        for (int kb = 0; kb < a.nkb; ++kb, ++it) {
          const int s = it % STAGES;
          const int hs = kb & 1;
          if (hs == 0) {
            cur = cn;
            const uint3 m0 = mn0, m1 = mn1;
            cn = load_codes((kb >> 1) + 1);
            mn0 = load_map((kb >> 1) + 1, r0);
            mn1 = load_map((kb >> 1) + 1, r1);
            __syncwarp();   // every lane is done with the previous group's table
#pragma unroll
            for (int q = 0; q < 2; ++q) {
              const uint3 m = q ? m1 : m0;
              const float a00 = f16_lo(m.x), a01 = f16_hi(m.x), a10 = f16_lo(m.y), a11 = f16_hi(m.y);
              const float b0 = f16_lo(m.z), b1 = f16_hi(m.z);
              const int rr = g + 8 * q;
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                const int idx = 4 * t + k;
                const float z0 = static_cast<float>(idx & 3), z1 = static_cast<float>(idx >> 2);
                const float w0 = fmaf(a00, z0, fmaf(a01, z1, b0));
                const float w1 = fmaf(a10, z0, fmaf(a11, z1, b1));
                sts32(tab_s + (rr * 16 + idx) * 4, pack_bf16x2(w0, w1));
              }
            }
            __syncwarp();
          }
          if (ok && it >= STAGES) {
            ok = !*abort_flag && mbar_wait(empty(s), ((it / STAGES) - 1) & 1, a.err, kErrTimeoutEmpty);
            if (!ok) *abort_flag = 1;
          }
          if (ok) {
            const uint32_t tile_addr = sbase + C::kOffA + s * kATileBytes;
#pragma unroll
            for (int q = 0; q < 2; ++q) {
              const uint32_t wh0 = q ? cur.y : cur.x, wh1 = q ? cur.w : cur.z;   // halves 0 and 1 of the row
              const uint32_t row_addr = tile_addr + (q ? r1 : r0) * 128;
              const uint32_t trow = tab_s + (g + 8 * q) * 64;
#pragma unroll
              for (int u = 0; u < 2; ++u) {
                const int cc = t + 4 * u;
                const int sh = 2 * (2 * hs + u);   // 2 s
                uint32_t o[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  const int bsh = 8 * ((e >> 1) | ((e & 1) << 1)) + sh;
                  const uint32_t idx = ((wh0 >> bsh) & 3u) | (((wh1 >> bsh) & 3u) << 2);
                  o[e] = lds32(trow + idx * 4);
                }
                sts128(row_addr + ((cc ^ g) << 4), o[0], o[1], o[2], o[3]);
              }
            }
            fence_proxy_async_smem();
          }
          __syncwarp();
          if (lane == 0 && ok) mbar_arrive(afull(s));
        }
      }
    } else {
      // Per-matrix maps. The loop is compiled four times (HI = 3-bit codes,
      // with P4 = d = 4 through two pair tables; D8 = 2-bit vectors of 8
      // through the quad tables; or none of these) so that each loop carries
      // only its own loads and no extra branches.
      auto convert = [&](auto hi_tag, auto d8_tag, auto p4_tag) {
        constexpr bool HI = decltype(hi_tag)::value;
        constexpr bool D8 = decltype(d8_tag)::value;
        constexpr bool P4 = decltype(p4_tag)::value;
        for (int tile = blockIdx.x; tile < a.tiles; tile += gridDim.x) {
          const int li = tile_layer(a, tile);
          const int n_blk = (tile - pick_layer(a.tile0, li)) / a.mtiles;
          const uint8_t* rbase =
              pick_layer(a.codes, li) + static_cast<size_t>(n_blk) * a.KT * kTileBytes + c * kUnitBytes + lane * 16;
          const uint32_t lut_s = lut_base + 2048u * static_cast<uint32_t>(li);
          // Code words of stage kb live at tile kb/2, half kb%2; prefetched
          // kCodeAhead stages ahead (a register ring).
          auto load = [&](int kb) -> uint2 {
            return kb < a.nkb ? __ldg(reinterpret_cast<const uint2*>(rbase + (kb >> 1) * kTileBytes + (kb & 1) * 8))
                              : make_uint2(0, 0);
          };
          // 3-bit codes: the halfwords of those two words in the high-bit plane
          const uint8_t* hbase =
              HI ? a.hi + static_cast<size_t>(n_blk) * a.KT * (kTileBytes / 2) + c * (kUnitBytes / 2) + lane * 8
                 : nullptr;
          auto load_hi = [&](int kb) -> uint32_t {
            if constexpr (HI)
              return kb < a.nkb
                         ? __ldg(reinterpret_cast<const uint32_t*>(hbase + (kb >> 1) * (kTileBytes / 2) + (kb & 1) * 4))
                         : 0u;
            return 0u;
          };
          uint2 qr[kCodeAhead];
          uint32_t hr[kCodeAhead];
#pragma unroll
          for (int j = 0; j < kCodeAhead; ++j) {
            qr[j] = load(j);
            hr[j] = load_hi(j);
          }
          // The stage loop is unrolled by the ring depth so that slot j is read
          // and refilled in place: shifting a register ring would read slots
          // whose loads are still in flight and wait for them every stage.
          bool ok = !*abort_flag;
          for (int kb0 = 0; kb0 < a.nkb; kb0 += kCodeAhead) {
#pragma unroll
          for (int j = 0; j < kCodeAhead; ++j) {
            const int kb = kb0 + j;
            if (kb >= a.nkb) break;
            const int s = it % STAGES;
            const uint2 cw = qr[j];
            const uint32_t hw = hr[j];
            qr[j] = load(kb + kCodeAhead);
            if constexpr (HI) hr[j] = load_hi(kb + kCodeAhead);
            if (ok && it >= STAGES) {
              ok = !*abort_flag && mbar_wait(empty(s), ((it / STAGES) - 1) & 1, a.err, kErrTimeoutEmpty);
              if (!ok) *abort_flag = 1;
            }
            if (ok) {
              const uint32_t tile_addr = sbase + C::kOffA + s * kATileBytes;
#pragma unroll
              for (int q = 0; q < 2; ++q) {
                const uint32_t w = q ? cw.y : cw.x;
                const uint32_t hq = q ? (hw >> 16) : (hw & 0xFFFFu);   // bit 4b + s: high bit of byte b, shift s
                const uint32_t row_addr = tile_addr + (q ? r1 : r0) * 128;
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                  const int cc = 2 * t + e;                       // chunk: stage columns 8cc .. 8cc+7
                  const uint32_t e0 = extract4(w, 2 * e);         // columns 8cc .. 8cc+3
                  const uint32_t e1 = extract4(w, 2 * e + 1);     // columns 8cc+4 .. 8cc+7
                  uint32_t o0, o1, o2, o3;
                  if constexpr (HI) {
                    // 3-bit codes of columns 8cc + 4u + b: low bits (e_u >> 8b) & 3, high bit
                    // bit 4b + 2e + u of hq; pairs (b = 0, 1) and (2, 3) index the 64-pair table
                    auto code3 = [&](uint32_t eu, int u, int b) -> uint32_t {
                      return ((eu >> (8 * b)) & 3u) | (((hq >> (4 * b + 2 * e + u)) & 1u) << 2);
                    };
                    const uint32_t p00 = code3(e0, 0, 0) | (code3(e0, 0, 1) << 3);
                    const uint32_t p01 = code3(e0, 0, 2) | (code3(e0, 0, 3) << 3);
                    const uint32_t p10 = code3(e1, 1, 0) | (code3(e1, 1, 1) << 3);
                    const uint32_t p11 = code3(e1, 1, 2) | (code3(e1, 1, 3) << 3);
                    if constexpr (P4) {
                      // columns 8cc .. +3 and 8cc + 4 .. +7 are two vectors; their coordinate
                      // pairs index two 64-row fp32 tables: w = T_0[z0 z1] + T_1[z2 z3]
                      const float4 va = lds128f(lut_s + p00 * 16), vb = lds128f(lut_s + 1024 + p01 * 16);
                      const float4 vc = lds128f(lut_s + p10 * 16), vd = lds128f(lut_s + 1024 + p11 * 16);
                      o0 = pack_bf16x2(va.x + vb.x, va.y + vb.y);
                      o1 = pack_bf16x2(va.z + vb.z, va.w + vb.w);
                      o2 = pack_bf16x2(vc.x + vd.x, vc.y + vd.y);
                      o3 = pack_bf16x2(vc.z + vd.z, vc.w + vd.w);
                    } else {
                      o0 = lds32(lut_s + (p00 << 2));
                      o1 = lds32(lut_s + (p01 << 2));
                      o2 = lds32(lut_s + (p10 << 2));
                      o3 = lds32(lut_s + (p11 << 2));
                    }
                  } else if constexpr (D8) {
                    // the chunk is one vector: coordinates 0..3 in bytes 0..3 of e0, 4..7 of e1;
                    // w = T_0[z0 z1 z2 z3] + T_1[z4 z5 z6 z7] (quad tables, fp32)
                    const uint32_t i0 = (e0 & 3u) | ((e0 >> 6) & 0xCu) | ((e0 >> 12) & 0x30u) | ((e0 >> 18) & 0xC0u);
                    const uint32_t i1 = (e1 & 3u) | ((e1 >> 6) & 0xCu) | ((e1 >> 12) & 0x30u) | ((e1 >> 18) & 0xC0u);
                    // (a row's two halves are swapped when bit 2 of its index is set)
                    const uint32_t t0 = lut_s + i0 * 32, t1 = lut_s + 8192 + i1 * 32;
                    const uint32_t s0 = (i0 << 2) & 16u, s1 = (i1 << 2) & 16u;
                    const float4 a0 = lds128f(t0 + s0), a1 = lds128f(t0 + (s0 ^ 16u));
                    const float4 b0 = lds128f(t1 + s1), b1 = lds128f(t1 + (s1 ^ 16u));
                    o0 = pack_bf16x2(a0.x + b0.x, a0.y + b0.y);
                    o1 = pack_bf16x2(a0.z + b0.z, a0.w + b0.w);
                    o2 = pack_bf16x2(a1.x + b1.x, a1.y + b1.y);
                    o3 = pack_bf16x2(a1.z + b1.z, a1.w + b1.w);
                  } else if (a.d == 4) {
                    const uint32_t i0 = (e0 & 3u) | ((e0 >> 6) & 0xCu) | ((e0 >> 12) & 0x30u) | ((e0 >> 18) & 0xC0u);
                    const uint32_t i1 = (e1 & 3u) | ((e1 >> 6) & 0xCu) | ((e1 >> 12) & 0x30u) | ((e1 >> 18) & 0xC0u);
                    const uint2 v0 = lds64(lut_s + i0 * 8), v1 = lds64(lut_s + i1 * 8);
                    o0 = v0.x; o1 = v0.y; o2 = v1.x; o3 = v1.y;
                  } else {
                    o0 = lds32(lut_s + (((e0 & 3u) | ((e0 >> 6) & 0xCu)) << 2));
                    o1 = lds32(lut_s + ((((e0 >> 16) & 3u) | ((e0 >> 22) & 0xCu)) << 2));
                    o2 = lds32(lut_s + (((e1 & 3u) | ((e1 >> 6) & 0xCu)) << 2));
                    o3 = lds32(lut_s + ((((e1 >> 16) & 3u) | ((e1 >> 22) & 0xCu)) << 2));
                  }
                  sts128(row_addr + ((cc ^ g) << 4), o0, o1, o2, o3);
                }
              }
              fence_proxy_async_smem();
            }
            __syncwarp();
            if (lane == 0 && ok) mbar_arrive(afull(s));
            ++it;
          }
          }
        }
      };
      if (a.hi && a.d == 4) convert(std::true_type{}, std::false_type{}, std::true_type{});
      else if (a.hi) convert(std::true_type{}, std::false_type{}, std::false_type{});
      else if (a.d == 8) convert(std::false_type{}, std::true_type{}, std::false_type{});
      else convert(std::false_type{}, std::false_type{}, std::false_type{});
    }
  } else {
    // ---------------- epilogue ----------------
    const int q = warp & 3;                      // TMEM lane quarter of this warp
    int lt = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < a.tiles && ok; tile += gridDim.x, ++lt) {
      const int b = lt & 1;
      const int li = tile_layer(a, tile);
      const int local = tile - pick_layer(a.tile0, li);
      const int n0 = (local / a.mtiles) * kBM;
      const int m0 = (local % a.mtiles) * BN;
      uint16_t* const yl = pick_layer(a.y, li);
      const int Nl = pick_layer(a.N, li);
      ok = !*abort_flag && mbar_wait(accfull(b), (lt >> 1) & 1, a.err, kErrTimeoutMma);
      if (!ok) {
        *abort_flag = 1;
        break;
      }
      tc_fence_after();
      const int n = n0 + 32 * q + lane;
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 32) {
        uint32_t r[32];
        tmem_ld32(tmem_base + (static_cast<uint32_t>(32 * q) << 16) + static_cast<uint32_t>(b * BN + c0), r);
        if (n < Nl) {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const int m = m0 + c0 + j;
            if (m < a.M) yl[static_cast<size_t>(m) * Nl + n] = f32_to_bf16_rn(__uint_as_float(r[j]));
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(accempty(b));
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem_base, C::kTmemCols);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

template <int BN, int STAGES, int NCONV>
unisvq_status launch_bn(const unisvq_layer* const* Ls, int n, const PrefillPlan& p, const void* x,
                        void* const* ys, int M, cudaStream_t s) {
  using C = PfCfg<BN, STAGES>;
  const unisvq_layer* L = Ls[0];
  static bool attr_set[64] = {};
  const int dev = L->device;
  if (dev < 0 || dev >= 64) return UNISVQ_ERR_CUDA;
  if (!attr_set[dev]) {
    if (cudaFuncSetAttribute(prefill_kernel<BN, STAGES, NCONV>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             C::kSmem) != cudaSuccess)
      return UNISVQ_ERR_CUDA;
    attr_set[dev] = true;
  }
  PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode();
  if (!enc) return UNISVQ_ERR_CUDA;
  CUtensorMap map;
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(L->K), static_cast<cuuint64_t>(M)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(L->K) * 2};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), static_cast<cuuint32_t>(BN)};
  const cuuint32_t estr[2] = {1, 1};
  if (enc(&map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(x), dims, strides, box, estr,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return UNISVQ_ERR_CUDA;

  PrefillArgs a{};
  a.mtiles = (M + BN - 1) / BN;
  int tile = 0;
  for (int i = 0; i < n; ++i) {
    a.codes[i] = Ls[i]->codes;
    a.lut[i] = Ls[i]->tlut;
    a.y[i] = static_cast<uint16_t*>(ys[i]);
    a.N[i] = Ls[i]->N;
    a.meta[i] = Ls[i]->grouped ? Ls[i]->meta : nullptr;
    a.tile0[i] = tile;
    tile += (Ls[i]->Np / kBM) * a.mtiles;
  }
  a.nlayers = n;
  a.hi = L->bits == 3 ? L->hi : nullptr;
  a.M = M;
  a.K = L->K;
  a.KT = L->KT;
  a.d = L->d;
  a.nkb = (L->K + kBK - 1) / kBK;
  a.tiles = p.tiles;
  a.err = device_error_word();
  if (tile != p.tiles) return UNISVQ_ERR_INVALID_ARG;
  prefill_kernel<BN, STAGES, NCONV><<<p.grid, pf_threads(NCONV), C::kSmem, s>>>(map, a);
  return cudaGetLastError() == cudaSuccess ? UNISVQ_OK : UNISVQ_ERR_CUDA;
}

int pick_bn(int M) { return M <= 64 ? 64 : (M <= 128 ? 128 : 256); }

}  // namespace

bool prefill_supported(const unisvq_layer* L, int M) {
  // per-group layers: d = 1 or 2 (a 16-pair table per row and group) or d = 4
  // and 8 (direct sums); 3-bit layers: d <= 4 (a 64-pair codeword table for d <= 2, two
  // 64-row pair tables for d = 4); per-matrix 2-bit layers: every d (d = 8
  // through two quad tables)
  const bool maps_ok = L->grouped ? true : (L->bits == 3 ? L->d <= 4 : true);
  return M > 0 && maps_ok && (L->K % 8) == 0 && get_encode() != nullptr;
}

bool prefill_group_supported(const unisvq_layer* const* Ls, int n, int M) {
  if (n < 1 || n > kPfMaxLayers) return false;
  if (n == 1) return prefill_supported(Ls[0], M);
  // several layers in one launch: 2-bit layers with one d <= 4 and one K, all
  // per-matrix (their tables, <= 2 KB each, share the table region) or all
  // per-group (each converter reads its tile's layer's maps)
  for (int i = 0; i < n; ++i)
    if (Ls[i]->grouped != Ls[0]->grouped || Ls[i]->bits != 2 || Ls[i]->d > 4 || Ls[i]->d != Ls[0]->d ||
        Ls[i]->K != Ls[0]->K || !prefill_supported(Ls[i], M))
      return false;
  return true;
}

PrefillPlan plan_prefill_group(const unisvq_layer* const* Ls, int n, int M) {
  PrefillPlan p{};
  p.bn = pick_bn(M);
  const int mtiles = (M + p.bn - 1) / p.bn;
  p.tiles = 0;
  for (int i = 0; i < n; ++i) p.tiles += (Ls[i]->Np / kBM) * mtiles;
  p.grid = p.tiles < Ls[0]->num_sms ? p.tiles : Ls[0]->num_sms;
  if (p.grid < 1) p.grid = 1;
  p.smem = p.bn == 64 ? PfCfg<64, 8>::kSmem : (p.bn == 128 ? PfCfg<128, 6>::kSmem : PfCfg<256, 4>::kSmem);
  return p;
}

PrefillPlan plan_prefill(const unisvq_layer* L, int M) { return plan_prefill_group(&L, 1, M); }

unisvq_status launch_prefill_group(const unisvq_layer* const* Ls, int n, const void* x, void* const* ys, int M,
                                   cudaStream_t s) {
  if (!prefill_group_supported(Ls, n, M)) return UNISVQ_ERR_UNSUPPORTED;
  const PrefillPlan p = plan_prefill_group(Ls, n, M);
  // per-matrix 2-bit layers with d <= 4: sixteen converter warps (a row each
  // per unit), else eight
  bool pm = true;
  for (int i = 0; i < n; ++i) pm = pm && !Ls[i]->grouped && Ls[i]->bits == 2 && Ls[i]->d <= 4;
  if (pm) {
    if (p.bn == 64) return launch_bn<64, 8, 16>(Ls, n, p, x, ys, M, s);
    if (p.bn == 128) return launch_bn<128, 6, 16>(Ls, n, p, x, ys, M, s);
    return launch_bn<256, 4, 16>(Ls, n, p, x, ys, M, s);
  }
  if (p.bn == 64) return launch_bn<64, 8, 8>(Ls, n, p, x, ys, M, s);
  if (p.bn == 128) return launch_bn<128, 6, 8>(Ls, n, p, x, ys, M, s);
  return launch_bn<256, 4, 8>(Ls, n, p, x, ys, M, s);
}

unisvq_status launch_prefill(const unisvq_layer* L, const void* x, void* y, int M, cudaStream_t s) {
  void* ys[1] = {y};
  return launch_prefill_group(&L, 1, x, ys, M, s);
}

}  // namespace unisvq
