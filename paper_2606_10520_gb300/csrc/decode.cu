// Skinny GEMM for decode batches (M <= 32 tokens per launch): tcgen05 tensor
// cores with the 2-bit codes as an 8-bit operand resident in tensor memory.
//
// Computes y = x W_hat^T through the fold of Eq. (col:matmul):
//   y[m, n] = sum_k x'[m, k] z[n, k] + c[m],
//   x'[m, g d + c] = sum_r x[m, g d + r] A[r][c]      (the row vectors X_i A)
//   c[m]          = sum_g x[m, g d .. g d + d - 1] . B  (the X_i B terms)
// so the codes are never turned into weights.
//
// Operands. A code z becomes a byte of an e4m3 A operand: with w a code word
// (columns 16t + 4s + b at bits 8b + 2s, layout.h),
//   w & 0x03030303        bytes z          (columns s = 0, e4m3 z * 2^-9)
//   w & 0x0c0c0c0c        bytes 4 z        (s = 1, e4m3 4z * 2^-9: bytes 0..15
//   (w >> 4) & 0x03030303 bytes z           are exact, subnormal or first binade)
//   (w >> 4) & 0x0c0c0c0c bytes 4 z        (s = 3)
// one shift and four ANDs for 16 codes; the factor 4 of odd s is taken out of
// the B operand. tcgen05.st writes the bytes into a TMEM A slot (128 rows in
// the 128 TMEM lanes, 32 columns of four bytes per k-tile). The folded
// activations, scaled per token and K slice by 2^P (|x' 2^P| < 256), are
// split into three e4m3 terms h + m + l (about 12 significant bits, the
// precision of fp16); the terms of token m are B rows 3m, 3m+1, 3m+2, so one
// MMA of N = 16/32/48/96 columns covers every term of up to 5/10/16/32 tokens and a
// 128 x 128 k-tile takes four tcgen05.mma.kind::f8f6f4 (K = 32). The epilogue
// adds the three term columns of a token and multiplies by 2^(9 - P).
//
// Two kernels per launch:
//  fold_kernel    one CTA per (K slice, token, layer): scale 2^P and c over the
//                 slice, then the B tiles of the slice, in the exact image of
//                 the 128B-swizzled shared-memory operand, into the layer's
//                 fold workspace (device memory owned by the handle). The fold
//                 is done once per launch instead of once per row block.
//  decode_kernel  CTA = 128 output rows x one K slice; the KS CTAs sharing the
//                 rows form a thread-block cluster and add their partial sums
//                 in distributed shared memory. Pipeline stages hold two
//                 k-tiles: 8 KB of codes and the two B tiles. Warp roles (10):
//     0      producer: code and B stages -> shared-memory ring (cp.async.bulk)
//     1      TMEM owner; one thread issues the MMAs
//     2..9   converters: shared ring -> TMEM A slots; warp w serves TMEM lane
//            quarter w % 4 (rows 32 (w%4) ..) for every other stage; warps
//            2..5 then run the epilogue (tcgen05.ld of their 32 rows)
// The codes never depend on the previous kernel: the producer fetches the
// first stages of codes before the programmatic-launch wait and the B tiles
// after it, so codes stream while the fold kernel runs. Layers that share x
// (same K) run in one launch of each kernel: their row blocks are stacked
// along grid.y of decode_kernel, their folds along grid.z of fold_kernel.
#include <atomic>
#include <cstring>
#include <cmath>

#include "common.cuh"
#include "hadamard.cuh"
#include "internal.h"

namespace unisvq {
namespace {

constexpr int kWarps = 10;
constexpr int kThreads = kWarps * 32;
constexpr int kConvWarp0 = 2;
constexpr int kConvWarps = 8;
constexpr int kMaxTokPerLaunch = 32;
constexpr int kMaxSplit = 8;                        // K slices (cluster size)
constexpr int kMaxGroup = UNISVQ_MAX_GROUP;
constexpr int kFoldThreads = 256;

// Fold workspace of a handle (unisvq_layer::fold_ws): a table of per-(slice,
// token) scale exponents and bias sums, then the B tiles of every k-tile.
constexpr int kWsTableBytes = 2048;                 // int pexp[8][32] at 0, float cpart[8][32] at kWsCpart
constexpr int kWsCpart = 1024;
constexpr int kWsTileStride = 96 * 128;             // B tile bytes per k-tile at the widest N

struct SkLayer {
  const uint8_t* codes;
  const uint8_t* hi;   // 3-bit codes: the high-bit plane (2048 bytes per tile), else null
  const uint8_t* ws;   // fold workspace (B tiles at kWsTableBytes)
  uint16_t* y;         // bf16 [M][N]
  int N;
  int rb0;             // first grid.y row block of this layer
};

struct SkArgs {
  int M, KT;
  int kt_per_cta;
  int nlayers;
  int* err;
  SkLayer layer[kMaxGroup];
};

// The fold kernel is instantiated for DV, the largest vector length of the
// launch's layers: DV = 4 (d in {1, 2, 4}) keeps A in registers and the
// parameter block small; DV = 8 stages the 8 x 8 A in shared memory.
template <int DV>
struct FoldLayer {
  uint8_t* ws;
  int d;
  int odd_exp;         // exponent of the B columns of odd s: -2 (2-bit codes, bytes 4 z), 0 (3-bit, bytes z)
  float colnorm;       // max_c sum_r |A[r][c]|
  float A[DV * DV];    // row-major d x d (d <= DV)
  float B[DV];
};

template <int DV>
struct FoldArgs {
  const uint16_t* x;   // bf16 [M][K]
  int M, K, KT;
  int kt_per_cta;
  int ncol;            // B rows (16, 32, 48)
  int nlayers;
  // Fused input rotation of the inverse RHT (x -> (x S_V) H_K / sqrt(K)):
  // S_V as sign bytes [K] (1 = -1), or null for none.
  const uint8_t* rht_sv;
  int rht_m;                   // Paley order m of K = p2 m (1, 12, 20 or 28)
  float rht_scale;             // 1 / sqrt(K)
  uint32_t rht_neg[28];        // column masks of H_m (m > 1)
  FoldLayer<DV> layer[kMaxGroup];
};

// Geometry: T k-tiles per pipeline stage. T = 2: 256 TMEM columns (accumulator
// in [0, 64), three A slots of 64), two CTAs per SM; for N = 96 (up to 32
// tokens) 512 columns (accumulator in [0, 128)), one CTA per SM. T = 1: 128
// TMEM columns (accumulator in [0, 32), three A slots of 32), N <= 32, three
// CTAs per SM.
// (One-tile stages for N = 48 would leave room for two A slots only; measured
// slower than two-tile stages on every Llama shape.)
template <int NCOL, int T, int BITS = 2>
struct Cfg {
  static constexpr int kT = T;
  static constexpr int kMinBlocks = T == 1 ? 3 : (NCOL > 64 ? 1 : 2);
  static constexpr int kCodeBytes = T * kTileBytes;
  static constexpr int kHiBytes = BITS == 3 ? T * (kTileBytes / 2) : 0;   // the stage's high-bit plane
  static constexpr int kAColBase = T == 1 ? 32 : (NCOL > 64 ? 128 : 64);
  static constexpr int kASlots = 3;                              // TMEM A slots (one stage each)
  static constexpr int kASlotCols = 32 * T;
  static constexpr int kTmemCols = T == 1 ? 128 : (NCOL > 64 ? 512 : 256);
  static constexpr int kMaxTok = NCOL / 3;
  static constexpr int kStages = NCOL >= 48 ? 4 : 6;
  static constexpr int kBTile = NCOL * 128;                      // one k-tile of B (NCOL rows x 128 bytes)
  static constexpr int kBBytes = T * kBTile;
  static constexpr int kStageBytes = kCodeBytes + kHiBytes + kBBytes;   // [codes | high bits | B tiles]
  static constexpr int kOffBStage = kCodeBytes + kHiBytes;
  static constexpr int kOffRed = kStages * kStageBytes;
  static constexpr int kRedBytes = (kTileRows + 8) * kMaxTok * 4;
  static constexpr int kOffBars = kOffRed + (kRedBytes + 15) / 16 * 16;
  static constexpr int kNumBars = 4 * kStages + 2 * kASlots + 3;
  static constexpr int kOffTok = kOffBars + kNumBars * 8;        // pexp[32], cpart[32]
  static constexpr int kOffMisc = kOffTok + 256;                 // tmem ptr, abort flag
  static constexpr int kSmem = kOffMisc + 64 + 1024;             // + alignment slack
  // kind::f8f6f4: D f32, A and B e4m3, both K-major, N = NCOL, M = 128.
  static constexpr uint32_t kIdesc =
      (1u << 4) | (static_cast<uint32_t>(NCOL >> 3) << 17) | ((128u >> 4) << 24);
  static_assert(kStageBytes % 1024 == 0 && kBTile % 1024 == 0, "128B-swizzled B tiles need 1024-byte alignment");
  static_assert(kStages % (kConvWarps / 4) == 0, "a converter group revisits its own stages");
  static_assert(NCOL <= kAColBase, "accumulator columns");
  static_assert(kAColBase + kASlots * kASlotCols <= kTmemCols, "TMEM columns");
  static_assert(kConvWarps / 4 <= kASlots, "converter groups must not run two slot uses ahead");
};

// ---- tcgen05 wrappers ----------------------------------------------------------

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups 1024 bytes apart.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  return static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4) | (static_cast<uint64_t>(1) << 16) |
         (static_cast<uint64_t>(1024 >> 4) << 32) | (static_cast<uint64_t>(1) << 46) |
         (static_cast<uint64_t>(2) << 61);
}

__device__ __forceinline__ void mma_f8_tmem_a(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                              uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

// 16 lanes x 32 columns: thread 4g + t holds, for column group k (0..3),
// v[4k + 0 .. 1] = lane g, columns 8k + 2t + (0, 1) and
// v[4k + 2 .. 3] = lane g + 8, columns 8k + 2t + (0, 1).
__device__ __forceinline__ void tmem_st16x256b_x4(uint32_t taddr, const uint32_t (&v)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.16x256b.x4.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]),
      "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
      : "memory");
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t* r) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}

// The 16 A-slot words of one lane for one 16-row unit. c holds the words of rows
// g (c.x half 0, c.z half 1) and g + 8 (c.y, c.w) for column quarter t. Word
// (h, s) of row g goes to v[4k + e], of row g + 8 to v[4k + 2 + e], with
// k = 2h + s/2 and e = s % 2: TMEM column 16h + 8(s/2) + 2t + s%2 of the slot
// holds the four columns 64h + 16t + 4s + (0..3) (times 4 for odd s).
__device__ __forceinline__ void expand_unit(uint4 c, uint32_t (&v)[16]) {
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const uint32_t wg = h ? c.z : c.x, wg8 = h ? c.w : c.y;
    const uint32_t sg = wg >> 4, sg8 = wg8 >> 4;
    v[8 * h + 0] = wg & 0x03030303u;    // k = 2h,     e = 0: s = 0
    v[8 * h + 1] = wg & 0x0c0c0c0cu;    // k = 2h,     e = 1: s = 1
    v[8 * h + 2] = wg8 & 0x03030303u;
    v[8 * h + 3] = wg8 & 0x0c0c0c0cu;
    v[8 * h + 4] = sg & 0x03030303u;    // k = 2h + 1, e = 0: s = 2
    v[8 * h + 5] = sg & 0x0c0c0c0cu;    // k = 2h + 1, e = 1: s = 3
    v[8 * h + 6] = sg8 & 0x03030303u;
    v[8 * h + 7] = sg8 & 0x0c0c0c0cu;
  }
}

// 3-bit codes: the same slot placement with the whole code z = z_lo + 4 z_hi in
// every byte (e4m3 z * 2^-9, exact for z <= 7; odd s get no factor 4, so the
// fold leaves their B columns unscaled). hw holds the chunk's four high-bit
// halfwords (halfword i for word i; bit 4b + s is z_hi of byte b, shift s).
__device__ __forceinline__ uint32_t spread_nibbles(uint32_t h16) {   // nibble b -> byte b
  return (h16 & 0xFu) | ((h16 & 0xF0u) << 4) | ((h16 & 0xF00u) << 8) | ((h16 & 0xF000u) << 12);
}
__device__ __forceinline__ void expand_unit3(uint4 c, uint2 hw, uint32_t (&v)[16]) {
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const uint32_t wg = h ? c.z : c.x, wg8 = h ? c.w : c.y;
    const uint32_t hh = h ? hw.y : hw.x;   // halfwords 2h (row g) and 2h + 1 (row g + 8)
    const uint32_t Hg = spread_nibbles(hh & 0xFFFFu), Hg8 = spread_nibbles(hh >> 16);
#pragma unroll
    for (int sq = 0; sq < 4; ++sq) {
      const int k = 2 * h + (sq >> 1), e = sq & 1;
      // bit s of each nibble-byte to bit 2 of the byte
      const uint32_t hig = (sq <= 2 ? (Hg << (2 - sq)) : (Hg >> 1)) & 0x04040404u;
      const uint32_t hig8 = (sq <= 2 ? (Hg8 << (2 - sq)) : (Hg8 >> 1)) & 0x04040404u;
      v[4 * k + e] = ((wg >> (2 * sq)) & 0x03030303u) | hig;
      v[4 * k + 2 + e] = ((wg8 >> (2 * sq)) & 0x03030303u) | hig8;
    }
  }
}

// e4m3x2 <-> f16x2 (lower byte <-> lower half).
__device__ __forceinline__ uint16_t f16x2_to_e4m3x2(uint32_t v) {
  uint16_t r;
  asm("cvt.rn.satfinite.e4m3x2.f16x2 %0, %1;" : "=h"(r) : "r"(v));
  return r;
}
__device__ __forceinline__ uint32_t e4m3x2_to_f16x2(uint16_t v) {
  uint32_t r;
  asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(r) : "h"(v));
  return r;
}
__device__ __forceinline__ uint32_t hsub2(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

// Split an f16 pair into three e4m3 pairs h + m + l (each residual is exact in f16).
__device__ __forceinline__ void split3(uint32_t v, uint16_t& h, uint16_t& m, uint16_t& l) {
  h = f16x2_to_e4m3x2(v);
  const uint32_t r1 = hsub2(v, e4m3x2_to_f16x2(h));
  m = f16x2_to_e4m3x2(r1);
  const uint32_t r2 = hsub2(r1, e4m3x2_to_f16x2(m));
  l = f16x2_to_e4m3x2(r2);
}

// x'[k+c] for the d-vectors inside x[k .. k+3] (k % 4 == 0): row vector x_g A.
__device__ __forceinline__ void fold4(int d, const float (&A)[16], const float (&v)[4], float (&o)[4]) {
  if (d == 1) {
#pragma unroll
    for (int e = 0; e < 4; ++e) o[e] = v[e] * A[0];
  } else if (d == 2) {
    o[0] = fmaf(v[1], A[2], v[0] * A[0]);
    o[1] = fmaf(v[1], A[3], v[0] * A[1]);
    o[2] = fmaf(v[3], A[2], v[2] * A[0]);
    o[3] = fmaf(v[3], A[3], v[2] * A[1]);
  } else {
#pragma unroll
    for (int c = 0; c < 4; ++c)
      o[c] = fmaf(v[3], A[12 + c], fmaf(v[2], A[8 + c], fmaf(v[1], A[4 + c], v[0] * A[c])));
  }
}

// The rotated activations of slice s (positions [s L, (s + 1) L) of the
// row, L = K / KS with KS = gridDim.x slices) for the fused inverse RHT, into
// xs as bf16. With H_K = H_{2^a} (Sylvester) Kronecker H_m and KS dividing
// 2^a, Sylvester's matrix splits over the high and low bits of the block
// index, so the slice needs (1) the signed sum over the KS slices of the row,
// term h with sign (-1)^popcount(h & s), of S_V x; (2) H_m on each of its
// L / m blocks; (3) Sylvester's transform over those blocks; then the scale
// 1 / sqrt(K). r0, r1: two fp32 buffers of L values in shared memory.
template <int DV>
__device__ __forceinline__ void fold_rotate_slice(const FoldArgs<DV>& a, const uint16_t* row, int s, int L,
                                                  uint16_t* xs, float* r0, float* r1) {
  const int KS = static_cast<int>(gridDim.x);
  for (int j8 = threadIdx.x; j8 < L / 8; j8 += kFoldThreads) {
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    for (int h = 0; h < KS; ++h) {
      const int k = h * L + 8 * j8;
      const uint4 u = ldg_v4(row + k);
      const uint2 sb = __ldg(reinterpret_cast<const uint2*>(a.rht_sv + k));
      const uint32_t flip_h = (__popc(h & s) & 1) ? 0x80000000u : 0u;
      const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
      for (int t = 0; t < 8; ++t) {
        const float v = (t & 1) ? bf16_hi(w[t >> 1]) : bf16_lo(w[t >> 1]);
        const uint32_t sbyte = (((t >> 2) ? sb.y : sb.x) >> (8 * (t & 3))) & 0xffu;
        acc[t] += __uint_as_float(__float_as_uint(v) ^ flip_h ^ (sbyte ? 0x80000000u : 0u));
      }
    }
#pragma unroll
    for (int t = 0; t < 8; ++t) r0[8 * j8 + t] = acc[t];
  }
  __syncthreads();
  const int m = a.rht_m, nblk = L / m;
  float* buf = r0;
  if (m > 1) {
    if (m == 12) paley_blocks<kFoldThreads, 12>(r0, r1, nblk, a.rht_neg);
    else if (m == 20) paley_blocks<kFoldThreads, 20>(r0, r1, nblk, a.rht_neg);
    else paley_blocks<kFoldThreads, 28>(r0, r1, nblk, a.rht_neg);
    buf = r1;
    __syncthreads();
  }
  sylvester_all<kFoldThreads>(buf, nblk, m);
  for (int j = threadIdx.x; j < L; j += kFoldThreads) xs[j] = f32_to_bf16_rn(buf[j] * a.rht_scale);
  __syncthreads();
}

// Fold of one K slice for one token of one layer: the scale 2^P and the bias
// sum c over the slice, then the slice's B tiles (rows 3 tok .. 3 tok + 2) in
// the layer's workspace. Rows of absent tokens are never written: an MMA
// column depends on its own B row only, and the epilogue never reads those
// columns.
// kRht: the instance with the fused input rotation (its registers do not
// limit the residency of the plain instance).
template <int DV, bool kRht>
__global__ void __launch_bounds__(kFoldThreads) fold_kernel(const __grid_constant__ FoldArgs<DV> a) {
  extern __shared__ __align__(16) uint8_t fsm[];
  uint16_t* xs = reinterpret_cast<uint16_t*>(fsm);   // the token's x slice, zero past K
  __shared__ float wmx[kFoldThreads / 32], wcs[kFoldThreads / 32];
  __shared__ int sp;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int s = blockIdx.x, tok = blockIdx.y, li = blockIdx.z;
  // This CTA's layer, read with constant parameter offsets only. For DV = 4,
  // A and B go to registers; for DV = 8, A goes to shared memory and
  // Bv[i] = B[i mod d] (the 8 columns of a chunk) to registers.
  __shared__ float sA[DV == 8 ? 64 : 1];
  uint8_t* ws = a.layer[0].ws;
  int d = a.layer[0].d;
  float colnorm = a.layer[0].colnorm;
  int odd_exp = a.layer[0].odd_exp;
  float A4[16], Bv[DV == 8 ? 8 : 4];
  if constexpr (DV == 4) {
#pragma unroll
    for (int i = 0; i < 16; ++i) A4[i] = a.layer[0].A[i];
#pragma unroll
    for (int i = 0; i < 4; ++i) Bv[i] = a.layer[0].B[i];
  }
#pragma unroll
  for (int l = 1; l < kMaxGroup; ++l)
    if (l == li) {
      ws = a.layer[l].ws;
      d = a.layer[l].d;
      colnorm = a.layer[l].colnorm;
      odd_exp = a.layer[l].odd_exp;
      if constexpr (DV == 4) {
#pragma unroll
        for (int i = 0; i < 16; ++i) A4[i] = a.layer[l].A[i];
#pragma unroll
        for (int i = 0; i < 4; ++i) Bv[i] = a.layer[l].B[i];
      }
    }
  if constexpr (DV == 8) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      float v = a.layer[0].B[i & (a.layer[0].d - 1)];
#pragma unroll
      for (int l = 1; l < kMaxGroup; ++l)
        if (l == li) v = a.layer[l].B[i & (a.layer[l].d - 1)];
      Bv[i] = v;
    }
    if (tid < 64) {
      float v = a.layer[0].A[tid];
#pragma unroll
      for (int l = 1; l < kMaxGroup; ++l)
        if (l == li) v = a.layer[l].A[tid];
      sA[tid] = v;
    }
  }
  const int kt0 = s * a.kt_per_cta;
  const int n_kt = min(a.kt_per_cta, a.KT - kt0);
  pdl_launch_dependents();   // the decode kernel may start fetching codes
  if (n_kt <= 0 || tok >= a.M || li >= a.nlayers) return;
  // x is the previous kernel's output, and the previous launch on this handle
  // may still read the workspace: both wait for the previous kernel.
  pdl_wait();
  const int kbeg = kt0 * kTileCols;
  const int kend = min(a.K, (kt0 + n_kt) * kTileCols);
  const int span = n_kt * kTileCols;
  const bool vec8 = (a.K & 7) == 0;
  const uint16_t* row = a.x + static_cast<size_t>(tok) * a.K;
  float mx = 0.f, cs = 0.f;
  if constexpr (kRht) {   // the slice of the rotated row (every slice full: K = KS span)
    float* r0 = reinterpret_cast<float*>(fsm + static_cast<size_t>(span) * 2);
    fold_rotate_slice(a, row, s, span, xs, r0, r0 + span);
    for (int c = tid * 8; c < span; c += kFoldThreads * 8) {
      const uint4 u = *reinterpret_cast<const uint4*>(xs + c);
      const uint32_t w4[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
      for (int t = 0; t < 4; ++t) {   // c is a multiple of 8: (k + i) mod d = i mod d
        const float v0 = bf16_lo(w4[t]), v1 = bf16_hi(w4[t]);
        mx = fmaxf(mx, fmaxf(fabsf(v0), fabsf(v1)));
        if constexpr (DV == 8) {
          cs = fmaf(v0, Bv[2 * t], cs);
          cs = fmaf(v1, Bv[2 * t + 1], cs);
        } else {
          cs = fmaf(v0, Bv[(2 * t) & (d - 1)], cs);
          cs = fmaf(v1, Bv[(2 * t + 1) & (d - 1)], cs);
        }
      }
    }
  }
  for (int c0 = tid * 8; !kRht && c0 < span; c0 += kFoldThreads * 8 * 4) {
    uint4 u[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int k = kbeg + c0 + j * kFoldThreads * 8;
      if (vec8 && k + 7 < kend) {
        u[j] = ldg_v4(row + k);
      } else {
        uint32_t e[8];
#pragma unroll
        for (int t = 0; t < 8; ++t) e[t] = (k + t < kend) ? static_cast<uint32_t>(row[k + t]) : 0u;
        u[j] = make_uint4(e[0] | (e[1] << 16), e[2] | (e[3] << 16), e[4] | (e[5] << 16), e[6] | (e[7] << 16));
      }
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int c = c0 + j * kFoldThreads * 8;
      if (c >= span) break;
      *reinterpret_cast<uint4*>(xs + c) = u[j];
      const uint32_t w4[4] = {u[j].x, u[j].y, u[j].z, u[j].w};
#pragma unroll
      for (int t = 0; t < 4; ++t) {   // kbeg and c are multiples of 8: (k + i) mod d = i mod d
        const float v0 = bf16_lo(w4[t]), v1 = bf16_hi(w4[t]);
        mx = fmaxf(mx, fmaxf(fabsf(v0), fabsf(v1)));
        if constexpr (DV == 8) {
          cs = fmaf(v0, Bv[2 * t], cs);
          cs = fmaf(v1, Bv[2 * t + 1], cs);
        } else {
          cs = fmaf(v0, Bv[(2 * t) & (d - 1)], cs);
          cs = fmaf(v1, Bv[(2 * t + 1) & (d - 1)], cs);
        }
      }
    }
  }
#pragma unroll
  for (int off = 16; off; off >>= 1) {
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    cs += __shfl_xor_sync(0xffffffffu, cs, off);
  }
  if (lane == 0) {
    wmx[warp] = mx;
    wcs[warp] = cs;
  }
  __syncthreads();
  if (tid == 0) {
    float tmx = 0.f, tcs = 0.f;
    for (int w = 0; w < kFoldThreads / 32; ++w) {
      tmx = fmaxf(tmx, wmx[w]);
      tcs += wcs[w];
    }
    // 2^P puts the largest possible |x'| (<= max|x| * colnorm) below 2^8.
    const float bound = tmx * colnorm;
    int e2 = 0;
    if (bound > 0.f) frexpf(bound, &e2);
    const int P = bound > 0.f ? max(-100, min(100, 8 - e2)) : 0;
    sp = P;
    reinterpret_cast<int*>(ws)[s * kMaxTokPerLaunch + tok] = P;
    reinterpret_cast<float*>(ws + kWsCpart)[s * kMaxTokPerLaunch + tok] = tcs;
  }
  __syncthreads();
  const int P = sp;
  const int ncol = a.ncol;
  uint8_t* tiles = ws + kWsTableBytes + static_cast<size_t>(kt0) * ncol * 128;
  if constexpr (DV == 8) {   // A for d <= 4 layers of the launch, in registers for the item loop
#pragma unroll
    for (int i = 0; i < 16; ++i) A4[i] = sA[i];
  }
  // Item (k-tile kt, column group g): columns 4g .. 4g + 3 of the tile, i.e.
  // quarter t = (g/4) % 4, s = g % 4, half h = g / 16, which sit in A-slot
  // column ac = 16h + 8(s/2) + 2t + s%2 (expand_unit): bytes 4 ac .. 4 ac + 3
  // of the 128-byte B row; odd s carries the factor 1/4.
  for (int item = tid; item < n_kt * 32; item += kFoldThreads) {
    const int kt = item >> 5, g = item & 31;
    const uint32_t ac = 16 * (g >> 4) + 8 * ((g & 3) >> 1) + 2 * ((g >> 2) & 3) + (g & 1);
    const uint32_t cidx = (ac & 3) * 4, chunk = ac >> 2;
    float o[4];
    if (DV == 8 && d == 8) {
      // Columns 4g .. 4g+3 are coordinates 4(g%2) .. of the vector 8(g/2) ..
      const uint4 xv = *reinterpret_cast<const uint4*>(xs + kt * kTileCols + 8 * (g >> 1));
      const float v[8] = {bf16_lo(xv.x), bf16_hi(xv.x), bf16_lo(xv.y), bf16_hi(xv.y),
                          bf16_lo(xv.z), bf16_hi(xv.z), bf16_lo(xv.w), bf16_hi(xv.w)};
      const int c0 = 4 * (g & 1);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        float acc = 0.f;
#pragma unroll
        for (int r = 0; r < 8; ++r) acc = fmaf(v[r], sA[8 * r + c0 + j], acc);
        o[j] = acc;
      }
    } else {
      const uint2 xv = *reinterpret_cast<const uint2*>(xs + kt * kTileCols + 4 * g);
      const float v[4] = {bf16_lo(xv.x), bf16_hi(xv.x), bf16_lo(xv.y), bf16_hi(xv.y)};
      fold4(d, A4, v, o);
    }
    const float sc = exp2i(P + ((g & 1) ? odd_exp : 0));
    uint16_t h0, m0, l0, h1, m1, l1;
    split3(pack_half2(o[0] * sc, o[1] * sc), h0, m0, l0);
    split3(pack_half2(o[2] * sc, o[3] * sc), h1, m1, l1);
    uint8_t* bt = tiles + static_cast<size_t>(kt) * ncol * 128;
    const int r = 3 * tok;
    *reinterpret_cast<uint32_t*>(bt + r * 128 + ((chunk ^ (r & 7)) << 4) + cidx) = h0 | (static_cast<uint32_t>(h1) << 16);
    *reinterpret_cast<uint32_t*>(bt + (r + 1) * 128 + ((chunk ^ ((r + 1) & 7)) << 4) + cidx) =
        m0 | (static_cast<uint32_t>(m1) << 16);
    *reinterpret_cast<uint32_t*>(bt + (r + 2) * 128 + ((chunk ^ ((r + 2) & 7)) << 4) + cidx) =
        l0 | (static_cast<uint32_t>(l1) << 16);
  }
}

template <int NCOL, int T, int BITS>
__global__ void __launch_bounds__(kThreads, Cfg<NCOL, T, BITS>::kMinBlocks)
    decode_kernel(const __grid_constant__ SkArgs a) {
  using C = Cfg<NCOL, T, BITS>;
  constexpr int kStageTiles = C::kT;
  constexpr int kCodeBytes = C::kCodeBytes;
  constexpr int kAColBase = C::kAColBase;
  constexpr int kASlotCols = C::kASlotCols;
  constexpr int kTmemCols = C::kTmemCols;
  constexpr int kASlots = C::kASlots;
  constexpr int S = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024 - (raw & 1023)) & 1023);
  const uint32_t sbase = smem_u32(smem);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int KS = gridDim.x;
  const int kt0 = blockIdx.x * a.kt_per_cta;
  const int n_kt = min(a.kt_per_cta, a.KT - kt0);
  const int n_st = (n_kt + kStageTiles - 1) / kStageTiles;
  const int M = a.M;
  // This CTA's layer, read with constant parameter offsets only.
  int li = 0;
#pragma unroll
  for (int i = 1; i < kMaxGroup; ++i)
    if (i < a.nlayers && static_cast<int>(blockIdx.y) >= a.layer[i].rb0) li = i;
  const uint8_t* lcodes = a.layer[0].codes;
  const uint8_t* lhi = a.layer[0].hi;
  const uint8_t* lws = a.layer[0].ws;
  uint16_t* ly = a.layer[0].y;
  int lN = a.layer[0].N, lrb0 = a.layer[0].rb0;
#pragma unroll
  for (int i = 1; i < kMaxGroup; ++i)
    if (i == li) {
      lcodes = a.layer[i].codes;
      lhi = a.layer[i].hi;
      lws = a.layer[i].ws;
      ly = a.layer[i].y;
      lN = a.layer[i].N;
      lrb0 = a.layer[i].rb0;
    }
  const int rb = static_cast<int>(blockIdx.y) - lrb0;

  const uint32_t bar0 = sbase + C::kOffBars;
  auto cfull = [&](int s) { return bar0 + 8u * s; };
  auto bfull = [&](int s) { return bar0 + 8u * (S + s); };
  auto cempty = [&](int s) { return bar0 + 8u * (2 * S + s); };
  auto bempty = [&](int s) { return bar0 + 8u * (3 * S + s); };
  auto a_full = [&](int s) { return bar0 + 8u * (4 * S + s); };
  auto a_empty = [&](int s) { return bar0 + 8u * (4 * S + kASlots + s); };
  const uint32_t bar_tail = bar0 + 8u * (4 * S + 2 * kASlots);
  const uint32_t d_full = bar_tail, tmem_ready = bar_tail + 8, drain = bar_tail + 16;
  int* pexp = reinterpret_cast<int*>(smem + C::kOffTok);
  float* cpart = reinterpret_cast<float*>(smem + C::kOffTok + 128);
  uint32_t* tmem_ptr = reinterpret_cast<uint32_t*>(smem + C::kOffMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::kOffMisc + 8);
  float* red = reinterpret_cast<float*>(smem + C::kOffRed);

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(cfull(s), 1);
      mbar_init(bfull(s), 1);
      mbar_init(cempty(s), 4);
      mbar_init(bempty(s), 1);
    }
    for (int s = 0; s < kASlots; ++s) {
      mbar_init(a_full(s), 4);
      mbar_init(a_empty(s), 1);
    }
    mbar_init(d_full, 1);
    mbar_init(tmem_ready, 1);
    mbar_init(drain, 1);
    const bool bad = n_kt <= 0 || M < 1 || M > C::kMaxTok;
    *abort_flag = bad ? 1 : 0;
    if (bad) record_error(a.err, kErrBadLaunch);
    fence_mbar_init();
  }
  __syncthreads();
  if (KS > 1) cluster_arrive_relaxed();   // waited for before the first remote store
  pdl_launch_dependents();

  if (warp == 0) {
    // ---------------- producer: code and B stages -> shared ring ----------------
    if (lane == 0 && !*abort_flag) {
      const uint64_t pol = policy_evict_first();
      const uint8_t* csrc = lcodes + (static_cast<size_t>(rb) * a.KT + kt0) * kTileBytes;
      const uint8_t* hsrc = BITS == 3 ? lhi + (static_cast<size_t>(rb) * a.KT + kt0) * (kTileBytes / 2) : nullptr;
      const uint8_t* bsrc = lws + kWsTableBytes + static_cast<size_t>(kt0) * C::kBTile;
      const int pre = min(S, n_st);
      // Codes of the first stages do not depend on the previous kernels.
      for (int st = 0; st < pre; ++st) {
        const uint32_t nt = static_cast<uint32_t>(min(kStageTiles, n_kt - st * kStageTiles));
        mbar_arrive_expect_tx(cfull(st), nt * (kTileBytes + C::kHiBytes / kStageTiles));
        bulk_g2s(sbase + st * C::kStageBytes, csrc + static_cast<size_t>(st) * kCodeBytes, nt * kTileBytes,
                 cfull(st), pol);
        if constexpr (BITS == 3)
          bulk_g2s(sbase + st * C::kStageBytes + kCodeBytes, hsrc + static_cast<size_t>(st) * C::kHiBytes,
                   nt * (kTileBytes / 2), cfull(st), pol);
      }
      pdl_wait();   // the B tiles come from the fold kernel
      for (int st = 0; st < pre; ++st) {
        const uint32_t nt = static_cast<uint32_t>(min(kStageTiles, n_kt - st * kStageTiles));
        mbar_arrive_expect_tx(bfull(st), nt * C::kBTile);
        bulk_g2s(sbase + st * C::kStageBytes + C::kOffBStage, bsrc + static_cast<size_t>(st) * C::kBBytes,
                 nt * C::kBTile, bfull(st), pol);
      }
      int st = pre;
      for (; st < n_st; ++st) {
        const int s = st % S;
        const uint32_t par = ((st / S) - 1) & 1;
        if (!mbar_wait(cempty(s), par, a.err, kErrTimeoutEmpty) || !mbar_wait(bempty(s), par, a.err, kErrTimeoutEmpty)) {
          *abort_flag = 1;
          break;
        }
        if (*abort_flag) break;
        const uint32_t nt = static_cast<uint32_t>(min(kStageTiles, n_kt - st * kStageTiles));
        mbar_arrive_expect_tx(cfull(s), nt * (kTileBytes + C::kHiBytes / kStageTiles));
        bulk_g2s(sbase + s * C::kStageBytes, csrc + static_cast<size_t>(st) * kCodeBytes, nt * kTileBytes, cfull(s),
                 pol);
        if constexpr (BITS == 3)
          bulk_g2s(sbase + s * C::kStageBytes + kCodeBytes, hsrc + static_cast<size_t>(st) * C::kHiBytes,
                   nt * (kTileBytes / 2), cfull(s), pol);
        mbar_arrive_expect_tx(bfull(s), nt * C::kBTile);
        bulk_g2s(sbase + s * C::kStageBytes + C::kOffBStage, bsrc + static_cast<size_t>(st) * C::kBBytes,
                 nt * C::kBTile, bfull(s), pol);
      }
      if (*abort_flag)   // copies nobody consumed must land before exit
        for (int j = st - S > 0 ? st - S : 0; j < st; ++j) {
          mbar_wait(cfull(j % S), (j / S) & 1, a.err, kErrTimeoutFull);
          mbar_wait(bfull(j % S), (j / S) & 1, a.err, kErrTimeoutFull);
        }
    }
  } else if (warp == 1) {
    // ---------------- TMEM owner + MMA issuer ----------------
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     sbase + C::kOffMisc),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    tc_fence_before();
    __syncwarp();
    if (lane == 0) {
      mbar_arrive(tmem_ready);
      tc_fence_after();
      const uint32_t tbase = *tmem_ptr;
      bool ok = !*abort_flag;
      for (int st = 0; st < n_st && ok; ++st) {
        const int sa = st % kASlots, s = st % S;
        // The converters arrive on a_full only once the stage's B tiles have
        // landed too (they wait on bfull), so one wait covers both operands.
        ok = mbar_wait(a_full(sa), (st / kASlots) & 1, a.err, kErrTimeoutFull);
        if (!ok) break;
        tc_fence_after();
        const int nt = min(kStageTiles, n_kt - st * kStageTiles);
        const uint32_t acol = tbase + kAColBase + kASlotCols * sa;
        const uint32_t bst = sbase + s * C::kStageBytes + C::kOffBStage;
        for (int j = 0; j < nt; ++j) {
          const uint64_t bd = sw128_desc(bst + j * C::kBTile);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)   // K = 32 bytes per MMA inside the 128-byte swizzle row
            mma_f8_tmem_a(tbase, acol + 32 * j + 8 * kk, bd + 2 * kk, C::kIdesc, (st | j | kk) != 0 ? 1u : 0u);
        }
        mma_commit(a_empty(sa));
        mma_commit(bempty(s));
      }
      if (ok) mma_commit(d_full);
      else *abort_flag = 1;
      mma_commit(drain);   // everything issued must retire before TMEM is released
      mbar_wait(drain, 0, a.err, kErrTimeoutMma);
    }
  } else {
    // ---------------- converters: shared ring -> TMEM A slots ----------------
    // Warp w serves TMEM lane quarter q = w % 4, i.e. units 2q and 2q + 1
    // (rows 32q .. 32q + 31), for the stages of parity p.
    const int cw = warp - kConvWarp0;
    const int q = warp & 3, p = cw >> 2;
    constexpr int kStep = kConvWarps / 4;
    bool ok = !*abort_flag && mbar_wait(tmem_ready, 0, a.err, kErrTimeoutFull);
    tc_fence_after();
    const uint32_t tq = *tmem_ptr + (static_cast<uint32_t>(32 * q) << 16);
    for (int st = p; st < n_st; st += kStep) {
      const int s = st % S, sa = st % kASlots;
      if (ok) ok = !*abort_flag && mbar_wait(cfull(s), (st / S) & 1, a.err, kErrTimeoutFull);
      const int nt = min(kStageTiles, n_kt - st * kStageTiles);
      uint4 cu[kStageTiles][2];
      uint2 hu[kStageTiles][2];
#pragma unroll
      for (int j = 0; j < kStageTiles; ++j) {
        cu[j][0] = make_uint4(0, 0, 0, 0);
        cu[j][1] = cu[j][0];
        hu[j][0] = make_uint2(0, 0);
        hu[j][1] = hu[j][0];
        if (ok && j < nt) {
          const uint8_t* tile = smem + s * C::kStageBytes + j * kTileBytes + (2 * q) * kUnitBytes + lane * 16;
          cu[j][0] = *reinterpret_cast<const uint4*>(tile);
          cu[j][1] = *reinterpret_cast<const uint4*>(tile + kUnitBytes);
          if constexpr (BITS == 3) {   // unit u's halfwords at 256 u + 8 lane of the tile's 2 KB
            const uint8_t* ht = smem + s * C::kStageBytes + kCodeBytes + j * (kTileBytes / 2) + (2 * q) * 256 + lane * 8;
            hu[j][0] = *reinterpret_cast<const uint2*>(ht);
            hu[j][1] = *reinterpret_cast<const uint2*>(ht + 256);
          }
        }
      }
      __syncwarp();
      if (lane == 0 && ok) mbar_arrive(cempty(s));
      if (ok && st >= kASlots)
        ok = !*abort_flag && mbar_wait(a_empty(sa), ((st / kASlots) - 1) & 1, a.err, kErrTimeoutMma);
      if (ok) {
        tc_fence_after();
        const uint32_t col = kAColBase + kASlotCols * sa;
#pragma unroll
        for (int j = 0; j < kStageTiles; ++j) {
          if (j < nt) {
            uint32_t v[16];
            if constexpr (BITS == 3) expand_unit3(cu[j][0], hu[j][0], v);
            else expand_unit(cu[j][0], v);
            tmem_st16x256b_x4(tq + col + 32 * j, v);
            if constexpr (BITS == 3) expand_unit3(cu[j][1], hu[j][1], v);
            else expand_unit(cu[j][1], v);
            tmem_st16x256b_x4(tq + (16u << 16) + col + 32 * j, v);
          }
        }
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
        tc_fence_before();
      }
      if (ok) ok = mbar_wait(bfull(s), (st / S) & 1, a.err, kErrTimeoutFull);
      __syncwarp();
      if (lane == 0 && ok) mbar_arrive(a_full(sa));
      if (!ok) *abort_flag = 1;
    }

    if (p == 0) {
      // ---------------- epilogue: accumulator rows -> cluster reduction ----------------
      const int r = 32 * q + lane;               // accumulator row (TMEM lane) of this thread
      if (ok) ok = !*abort_flag && mbar_wait(d_full, 0, a.err, kErrTimeoutMma);
      if (!ok) *abort_flag = 1;
      pdl_wait();   // the scale table comes from the fold kernel
      if (q == 0 && lane < M) {
        pexp[lane] = reinterpret_cast<const int*>(lws)[blockIdx.x * kMaxTokPerLaunch + lane];
        cpart[lane] = reinterpret_cast<const float*>(lws + kWsCpart)[blockIdx.x * kMaxTokPerLaunch + lane];
      }
      named_barrier_sync(1, 4 * 32);
      const int rows_per = (kTileRows + KS - 1) / KS;
      const int owner = r / rows_per;
      const uint32_t slot_off =
          (static_cast<uint32_t>(blockIdx.x) * rows_per + (r - owner * rows_per)) * C::kMaxTok * 4u;
      const uint32_t red_addr = sbase + C::kOffRed;
      if (KS > 1) cluster_wait();
      tc_fence_after();
      uint32_t dv[NCOL];
#pragma unroll
      for (int c0 = 0; c0 < NCOL; c0 += 16) tmem_ld16(tq + c0, dv + c0);
      asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
      bool done_v4 = false;
      if constexpr (C::kMaxTok % 4 == 0) {
        if (KS > 1) {
          // 16-byte stores into the owner's slots (kMaxTok floats per row,
          // 16-byte aligned): a quarter of the cluster transactions of scalar
          // stores; slots past M get zeros the reduction never reads
          done_v4 = true;
          const uint32_t dst = map_shared_rank(red_addr + slot_off, owner);
#pragma unroll
          for (int t4 = 0; t4 < C::kMaxTok; t4 += 4) {
            if (ok && t4 < M) {
              float v[4];
#pragma unroll
              for (int j = 0; j < 4; ++j) {
                const int tok = t4 + j;
                const float acc = __uint_as_float(dv[3 * tok]) + __uint_as_float(dv[3 * tok + 1]) +
                                  __uint_as_float(dv[3 * tok + 2]);
                v[j] = tok < M ? fmaf(acc, exp2i(9 - pexp[tok]), cpart[tok]) : 0.f;
              }
              asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(dst + 4u * t4), "f"(v[0]),
                           "f"(v[1]), "f"(v[2]), "f"(v[3])
                           : "memory");
            }
          }
        }
      }
      if (!done_v4) {
#pragma unroll
        for (int tok = 0; tok < C::kMaxTok; ++tok) {
          if (ok && tok < M) {
            const float acc = __uint_as_float(dv[3 * tok]) + __uint_as_float(dv[3 * tok + 1]) +
                              __uint_as_float(dv[3 * tok + 2]);
            const float val = fmaf(acc, exp2i(9 - pexp[tok]), cpart[tok]);
            const uint32_t off = slot_off + tok * 4u;
            if (KS > 1) st_shared_cluster_f32(map_shared_rank(red_addr + off, owner), val);
            else red[off / 4] = val;
          }
        }
      }
      tc_fence_before();
    }
  }

  // ---------------- reduction over the K slices of the cluster ----------------
  __syncwarp();
  const bool epilogue_warp = warp >= kConvWarp0 && warp < kConvWarp0 + 4;
  if (KS > 1) {
    if (!epilogue_warp) cluster_wait();   // the epilogue warps waited before their stores
    cluster_sync();
  } else {
    __syncthreads();
  }
  {
    const int rows_per = (kTileRows + KS - 1) / KS;
    const int r0 = static_cast<int>(blockIdx.x) * rows_per;
    const int nrows = max(0, min(kTileRows, r0 + rows_per) - r0);
    for (int idx = tid; idx < nrows * M; idx += kThreads) {
      const int tok = idx / nrows;
      const int rl = idx - tok * nrows;
      const int n = rb * kTileRows + r0 + rl;
      float s = 0.f;
      for (int qq = 0; qq < KS; ++qq) s += red[(qq * rows_per + rl) * C::kMaxTok + tok];
      if (n < lN && !*abort_flag) ly[static_cast<size_t>(tok) * lN + n] = f32_to_bf16_rn(s);
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(*tmem_ptr), "r"(kTmemCols)
                 : "memory");
  }
}

int ncol_for(int M) { return M <= 5 ? 16 : (M <= 10 ? 32 : (M <= 16 ? 48 : 96)); }

template <int NCOL, int T, int BITS>
bool set_attrs(int dev) {
  static std::atomic<bool> done[64];
  if (dev < 0 || dev >= 64) return false;
  if (done[dev].load(std::memory_order_acquire)) return true;
  if (cudaFuncSetAttribute(decode_kernel<NCOL, T, BITS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           Cfg<NCOL, T, BITS>::kSmem) != cudaSuccess ||
      cudaFuncSetAttribute(decode_kernel<NCOL, T, BITS>, cudaFuncAttributePreferredSharedMemoryCarveout,
                           cudaSharedmemCarveoutMaxShared) != cudaSuccess)
    return false;
  done[dev].store(true, std::memory_order_release);
  return true;
}

constexpr int kFoldMaxSmem = 96 * 1024;   // x slice of one token: <= 384 k-tiles

bool set_fold_attrs(int dev) {
  static bool done[64] = {};
  if (dev < 0 || dev >= 64) return false;
  if (done[dev]) return true;
  if (cudaFuncSetAttribute(fold_kernel<4, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, kFoldMaxSmem) !=
          cudaSuccess ||
      cudaFuncSetAttribute(fold_kernel<8, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, kFoldMaxSmem) !=
          cudaSuccess ||
      cudaFuncSetAttribute(fold_kernel<4, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, kFoldMaxSmem) !=
          cudaSuccess ||
      cudaFuncSetAttribute(fold_kernel<8, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, kFoldMaxSmem) !=
          cudaSuccess)
    return false;
  done[dev] = true;
  return true;
}

template <int T, int BITS>
size_t smem_of_b(int ncol) {
  return ncol == 16 ? Cfg<16, T, BITS>::kSmem
                    : (ncol == 32 ? Cfg<32, T, BITS>::kSmem
                                  : (ncol == 48 ? Cfg<48, 2, BITS>::kSmem : Cfg<96, 2, BITS>::kSmem));
}
size_t smem_of(int ncol, int T, int bits) {
  if (bits == 3) return T == 1 ? smem_of_b<1, 3>(ncol) : smem_of_b<2, 3>(ncol);
  return T == 1 ? smem_of_b<1, 2>(ncol) : smem_of_b<2, 2>(ncol);
}

// Resident CTAs per SM: as many as the shared memory, the TMEM columns
// (512 / kTmemCols) and the registers of 320 threads allow (two for T = 2,
// one for the 96-column accumulator, three for T = 1). The occupancy query of the runtime reports one for this
// kernel although two or three run side by side (measured), so the count is
// derived here.
int resident_for(int ncol, int T, int bits) {
  const size_t smem = smem_of(ncol, T, bits);
  const int by_smem = static_cast<int>((static_cast<size_t>(228) * 1024) / (smem + 1024));
  const int by_tmem = T == 1 ? 4 : (ncol > 64 ? 1 : 2);
  const int by_regs = T == 1 ? 3 : (ncol > 64 ? 1 : 2);
  return max(1, min(by_smem, min(by_tmem, by_regs)));
}

// Largest K split (cluster size <= 8, >= 1 k-tile per CTA) whose grid fits in
// one wave of resident CTAs of geometry T; at least enough slices for the
// fold kernel's shared memory.
DecodePlan plan_with(int nb, int KT, int num_sms, int ncol, int T, int bits) {
  DecodePlan p{};
  p.nt = ncol;
  p.nb = nb;
  p.geom = T;
  const int slots = resident_for(ncol, T, bits) * num_sms;
  const int min_ks = (KT * kTileCols * 2 + kFoldMaxSmem - 1) / kFoldMaxSmem;
  int ks = 0;
  for (int c = kMaxSplit; c >= 1; --c)
    if (c <= KT && nb * c <= slots) {
      ks = c;
      break;
    }
  if (ks < min_ks) ks = min_ks;
  if (ks < 1) ks = 1;
  p.kt_per_cta = (KT + ks - 1) / ks;
  p.ks = (KT + p.kt_per_cta - 1) / p.kt_per_cta;
  p.smem = smem_of(ncol, T, bits);
  return p;
}

// Two-tile stages (two CTAs per SM) unless one-tile stages (three CTAs per
// SM, accumulator <= 32 columns) allow a larger K split: per byte the longer
// stages are cheaper, but more slices spread a launch over more CTAs
// (measured on GB300: 4096 x 11008 prefers two-tile stages at K split 8;
// 3 x 4096 x 4096 and 28672 x 8192 prefer one-tile stages).
DecodePlan plan_rows_split(int nb, int KT, int num_sms, int M, int bits = 2) {
  const int ncol = ncol_for(M);
  const DecodePlan p2 = plan_with(nb, KT, num_sms, ncol, 2, bits);
  if (ncol <= 32) {
    const DecodePlan p1 = plan_with(nb, KT, num_sms, ncol, 1, bits);
    if (p1.ks > p2.ks) return p1;
  }
  return p2;
}

// The plan of a launch whose fold kernel also rotates x (K = p2 m): the K
// split reduced to the largest power of 2 that divides both KT and p2, so
// every slice is full and a union of whole m-blocks.
DecodePlan plan_rht(int nb, int KT, int num_sms, int M, int p2) {
  DecodePlan p = plan_rows_split(nb, KT, num_sms, M);
  int ks = 1;
  while (ks * 2 <= p.ks && KT % (ks * 2) == 0 && p2 % (ks * 2) == 0) ks *= 2;
  p.ks = ks;
  p.kt_per_cta = KT / ks;
  return p;
}

cudaLaunchAttribute pdl_attr() {
  cudaLaunchAttribute at;
  at.id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at.val.programmaticStreamSerializationAllowed = 1;
  return at;
}

template <int NCOL, int T, int BITS>
unisvq_status launch_ncol(const SkArgs& a, const DecodePlan& p, int dev, cudaStream_t s) {
  if (!set_attrs<NCOL, T, BITS>(dev)) return UNISVQ_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.ks, p.nb, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = Cfg<NCOL, T, BITS>::kSmem;
  cfg.stream = s;
  cudaLaunchAttribute attrs[2];
  attrs[0].id = cudaLaunchAttributeClusterDimension;
  attrs[0].val.clusterDim.x = p.ks;
  attrs[0].val.clusterDim.y = 1;
  attrs[0].val.clusterDim.z = 1;
  attrs[1] = pdl_attr();
  cfg.attrs = attrs;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, decode_kernel<NCOL, T, BITS>, a) == cudaSuccess ? UNISVQ_OK : UNISVQ_ERR_CUDA;
}

}  // namespace

size_t fold_workspace_bytes(int KT) { return kWsTableBytes + static_cast<size_t>(KT) * kWsTileStride; }

// Fold workspace a launch of at most max_tok tokens writes (B tiles of the
// launch's N only).
static size_t fold_workspace_bytes_for(int KT, int max_tok) {
  return kWsTableBytes + static_cast<size_t>(KT) * ncol_for(max_tok) * 128;
}

// Tokens per launch pair: 32 (the 96-column accumulator, one CTA per SM)
// where that takes fewer waves of row blocks than two 16-token launches (two
// CTAs per SM), else 16. Measured on GB300 at M = 32: Llama-2-7B q/k/v (96
// row blocks: 1 wave against 2) 19.1 us in one launch, 24.6 in two; the
// gate/up pair (172: 2 against 2) 35.5 against 32.3; the Llama-2-70B gate/up
// pair (448: 3 against 4) is faster in one launch.
int skinny_tokens_per_launch(const unisvq_layer* const* Ls, int n) {
  int nb = 0;
  for (int i = 0; i < n; ++i) nb += Ls[i]->Np / kTileRows;
  const int sms = Ls[0]->num_sms > 0 ? Ls[0]->num_sms : 1;
  const int waves32 = (nb + sms - 1) / sms, waves16 = 2 * ((nb + 2 * sms - 1) / (2 * sms));
  return waves32 < waves16 ? kMaxTokPerLaunch : 16;
}

DecodePlan plan_skinny(const unisvq_layer* const* Ls, int n, int M) {
  int nb = 0;
  for (int i = 0; i < n; ++i) nb += Ls[i]->Np / kTileRows;
  const int per = skinny_tokens_per_launch(Ls, n);
  return plan_rows_split(nb, Ls[0]->KT, Ls[0]->num_sms, M > per ? per : M, Ls[0]->bits);
}

namespace {

// The fold of tokens m0 .. m0 + mc - 1 for plan p (fold_kernel<DV, rht_sv != null>).
template <int DV>
unisvq_status launch_fold(const unisvq_layer* const* Ls, int n, const void* x, int m0, int mc, const DecodePlan& p,
                          cudaStream_t s, uint8_t* const* ws, const uint8_t* rht_sv) {
  const unisvq_layer* L0 = Ls[0];
  FoldArgs<DV> f{};
  f.x = static_cast<const uint16_t*>(x) + static_cast<size_t>(m0) * L0->K;
  f.M = mc;
  f.K = L0->K;
  f.KT = L0->KT;
  f.kt_per_cta = p.kt_per_cta;
  f.ncol = p.nt;
  f.nlayers = n;
  size_t smem = static_cast<size_t>(p.kt_per_cta) * kTileCols * 2;
  if (rht_sv) {   // fused input rotation: two fp32 copies of the slice besides the bf16 one
    int p2 = 0, m = 0;
    if (!rht_factor(L0->K, &p2, &m) || m > 28) return UNISVQ_ERR_UNSUPPORTED;
    f.rht_sv = rht_sv;
    f.rht_m = m;
    f.rht_scale = static_cast<float>(1.0 / std::sqrt(static_cast<double>(L0->K)));
    if (m > 1) std::memcpy(f.rht_neg, rht_paley_masks(m), sizeof(f.rht_neg));
    smem *= 5;
  }
  for (int i = 0; i < n; ++i) {
    const unisvq_layer* L = Ls[i];
    FoldLayer<DV>& fl = f.layer[i];
    fl.ws = ws[i];
    fl.d = L->d;
    fl.colnorm = L->colnorm;
    fl.odd_exp = L->bits == 3 ? 0 : -2;
    for (int j = 0; j < DV * DV; ++j) fl.A[j] = L->A[j];
    for (int j = 0; j < DV; ++j) fl.B[j] = L->B[j];
  }
  cudaLaunchConfig_t fc = {};
  fc.gridDim = dim3(p.ks, mc, n);
  fc.blockDim = dim3(kFoldThreads, 1, 1);
  fc.dynamicSmemBytes = smem;
  fc.stream = s;
  cudaLaunchAttribute fat[1] = {pdl_attr()};
  fc.attrs = fat;
  fc.numAttrs = 1;
  const cudaError_t e = rht_sv ? cudaLaunchKernelEx(&fc, fold_kernel<DV, true>, f)
                               : cudaLaunchKernelEx(&fc, fold_kernel<DV, false>, f);
  return e == cudaSuccess ? UNISVQ_OK : UNISVQ_ERR_CUDA;
}

// Fold and stream, the fold workspace of layer i at ws[i], at most max_tok
// tokens per launch.
unisvq_status launch_skinny_ws(const unisvq_layer* const* Ls, int n, const void* x, void* const* ys, int M,
                               cudaStream_t s, uint8_t* const* ws, int max_tok = kMaxTokPerLaunch,
                               const uint8_t* rht_sv = nullptr) {
  if (n < 1 || n > kMaxGroup) return UNISVQ_ERR_INVALID_ARG;
  const unisvq_layer* L0 = Ls[0];
  if (!set_fold_attrs(L0->device)) return UNISVQ_ERR_CUDA;
  int nb = 0;
  bool d8 = false;
  for (int i = 0; i < n; ++i) {
    nb += Ls[i]->Np / kTileRows;
    d8 = d8 || Ls[i]->d == 8;
    // one code width per launch (the kernel instance); 3-bit codes have d <= 4
    if (Ls[i]->bits != L0->bits || Ls[i]->grouped || (Ls[i]->bits == 3 && Ls[i]->d > 4))
      return UNISVQ_ERR_UNSUPPORTED;
  }
  int rht_p2 = 0, rht_m = 0;
  if (rht_sv && (L0->bits != 2 || !rht_factor(L0->K, &rht_p2, &rht_m))) return UNISVQ_ERR_UNSUPPORTED;
  for (int m0 = 0; m0 < M; m0 += max_tok) {
    const int mc = M - m0 < max_tok ? M - m0 : max_tok;
    const DecodePlan p = rht_sv ? plan_rht(nb, L0->KT, L0->num_sms, mc, rht_p2)
                                : plan_rows_split(nb, L0->KT, L0->num_sms, mc, L0->bits);
    if (p.ks > kMaxSplit) return UNISVQ_ERR_UNSUPPORTED;
    SkArgs a{};
    a.M = mc;
    a.KT = L0->KT;
    a.kt_per_cta = p.kt_per_cta;
    a.nlayers = n;
    a.err = device_error_word();
    int rb0 = 0;
    for (int i = 0; i < n; ++i) {
      const unisvq_layer* L = Ls[i];
      SkLayer& l = a.layer[i];
      l.codes = L->codes;
      l.hi = L->bits == 3 ? L->hi : nullptr;
      l.ws = ws[i];
      l.y = static_cast<uint16_t*>(ys[i]) + static_cast<size_t>(m0) * L->N;
      l.N = L->N;
      l.rb0 = rb0;
      rb0 += L->Np / kTileRows;
    }
    unisvq_status st = d8 ? launch_fold<8>(Ls, n, x, m0, mc, p, s, ws, rht_sv)
                          : launch_fold<4>(Ls, n, x, m0, mc, p, s, ws, rht_sv);
    if (st != UNISVQ_OK) return st;
    if (L0->bits == 3) {
      if (p.nt == 16) st = p.geom == 1 ? launch_ncol<16, 1, 3>(a, p, L0->device, s) : launch_ncol<16, 2, 3>(a, p, L0->device, s);
      else if (p.nt == 32) st = p.geom == 1 ? launch_ncol<32, 1, 3>(a, p, L0->device, s) : launch_ncol<32, 2, 3>(a, p, L0->device, s);
      else if (p.nt == 48) st = launch_ncol<48, 2, 3>(a, p, L0->device, s);
      else st = launch_ncol<96, 2, 3>(a, p, L0->device, s);
    } else {
      if (p.nt == 16) st = p.geom == 1 ? launch_ncol<16, 1, 2>(a, p, L0->device, s) : launch_ncol<16, 2, 2>(a, p, L0->device, s);
      else if (p.nt == 32) st = p.geom == 1 ? launch_ncol<32, 1, 2>(a, p, L0->device, s) : launch_ncol<32, 2, 2>(a, p, L0->device, s);
      else if (p.nt == 48) st = launch_ncol<48, 2, 2>(a, p, L0->device, s);
      else st = launch_ncol<96, 2, 2>(a, p, L0->device, s);
    }
    if (st != UNISVQ_OK) return st;
  }
  return UNISVQ_OK;
}

}  // namespace

unisvq_status launch_skinny_group(const unisvq_layer* const* Ls, int n, const void* x, void* const* ys, int M,
                                  cudaStream_t s) {
  if (n < 1 || n > kMaxGroup) return UNISVQ_ERR_INVALID_ARG;
  uint8_t* ws[kMaxGroup];
  for (int i = 0; i < n; ++i) ws[i] = Ls[i]->fold_ws;
  return launch_skinny_ws(Ls, n, x, ys, M, s, ws, skinny_tokens_per_launch(Ls, n));
}

unisvq_status launch_skinny(const unisvq_layer* L, const void* x, void* y, int M, cudaStream_t s) {
  void* ys[1] = {y};
  return launch_skinny_group(&L, 1, x, ys, M, s);
}

bool skinny_rht_foldable(const unisvq_layer* const* Ls, int n, int M) {
  if (n < 1 || n > kMaxGroup || M < 1) return false;
  const unisvq_layer* L0 = Ls[0];
  int p2 = 0, m = 0;
  if (!rht_factor(L0->K, &p2, &m) || m > 28 || L0->K != L0->KT * kTileCols) return false;
  int nb = 0;
  for (int i = 0; i < n; ++i) nb += Ls[i]->Np / kTileRows;
  // every launch size of the call: full launches and the remainder
  const int per = skinny_tokens_per_launch(Ls, n);
  const int sizes[2] = {M < per ? M : per, M > per ? M % per : 0};
  for (const int mc : sizes) {
    if (mc == 0) continue;
    // a K split of 1 would leave one CTA per token and layer to transform the
    // whole row: measured slower than the separate rotation kernel (cluster
    // of CTAs) whose latency the decode kernel's code prefetch hides
    const DecodePlan p = plan_rht(nb, L0->KT, L0->num_sms, mc, p2);
    if (p.ks < 2 || p.ks * p.kt_per_cta != L0->KT || p2 % p.ks != 0) return false;
    if (static_cast<size_t>(p.kt_per_cta) * kTileCols * 10 > static_cast<size_t>(kFoldMaxSmem)) return false;
  }
  return true;
}

unisvq_status launch_skinny_group_rht(const unisvq_layer* const* Ls, int n, const void* x, void* const* ys, int M,
                                      const uint8_t* rht_sv, cudaStream_t s) {
  if (n < 1 || n > kMaxGroup || !rht_sv) return UNISVQ_ERR_INVALID_ARG;
  if (!skinny_rht_foldable(Ls, n, M)) return UNISVQ_ERR_UNSUPPORTED;
  uint8_t* ws[kMaxGroup];
  for (int i = 0; i < n; ++i) ws[i] = Ls[i]->fold_ws;
  return launch_skinny_ws(Ls, n, x, ys, M, s, ws, skinny_tokens_per_launch(Ls, n), rht_sv);
}

// ---- allocation-free variant (unisvq_linear_noalloc) -------------------------
// The same fold and streaming kernels with the fold workspace taken from a
// file-scope device array that exists from module load, for callers that may
// not allocate on the call path. One array per device: calls of this entry
// point that overlap on the GPU race on it. Nothing in it has to start at
// zero (the fold kernel writes every table entry and B row the streaming
// kernel reads).
constexpr size_t kStaticWsBytes = static_cast<size_t>(2) << 20;   // 2 MiB: Kp <= 43648
__device__ __align__(256) uint8_t g_static_fold_ws[kStaticWsBytes];

size_t static_fold_workspace_bytes() { return kStaticWsBytes; }

unisvq_status launch_skinny_static(const unisvq_layer* L, const void* x, void* y, int M, cudaStream_t s) {
  // unisvq_linear's tokens per launch where their B tiles fit the array, else 16
  const int per = skinny_tokens_per_launch(&L, 1);
  const int max_tok = fold_workspace_bytes_for(L->KT, per) <= kStaticWsBytes ? per : 16;
  if (fold_workspace_bytes_for(L->KT, max_tok) > kStaticWsBytes) return UNISVQ_ERR_UNSUPPORTED;
  // In host code g_static_fold_ws only names the symbol; its device address
  // is looked up once per device (the device of L is current here) and kept
  // in an atomic slot, so concurrent first calls store the same value. A
  // cudaDeviceReset unloads the module: the library must then be reloaded.
  static std::atomic<uint8_t*> dev_ptr[64] = {};
  if (L->device < 0 || L->device >= 64) return UNISVQ_ERR_INVALID_ARG;
  uint8_t* wsp = dev_ptr[L->device].load(std::memory_order_acquire);
  if (!wsp) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_static_fold_ws) != cudaSuccess || !p) return UNISVQ_ERR_CUDA;
    wsp = static_cast<uint8_t*>(p);
    dev_ptr[L->device].store(wsp, std::memory_order_release);
  }
  uint8_t* ws[1] = {wsp};
  void* ys[1] = {y};
  return launch_skinny_ws(&L, 1, x, ys, M, s, ws, max_tok);
}

}  // namespace unisvq
