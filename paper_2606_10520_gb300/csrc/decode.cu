// Skinny GEMM for decode batches (M <= 64 tokens per launch): tcgen05 tensor cores
// with the 2-bit codes as an 8-bit operand resident in tensor memory.
//
// Computes y = x W_hat^T through the fold of Eq. (col:matmul):
//   y[m, n] = sum_k x'[m, k] z[n, k] + c[m],
//   x'[m, g d + c] = sum_r x[m, g d + r] A[r][c]      (the row vectors X_i A)
//   c[m]          = sum_g x[m, g d .. g d + d - 1] . B  (the X_i B terms)
// so the codes are never turned into weights. Each code z becomes the byte z,
// which is exactly the e4m3 subnormal z * 2^-9; one shift and one AND expand
// four codes (layout.h) and tcgen05.st writes them as the A operand of
// tcgen05.mma.kind::f8f6f4 (128 rows in TMEM lanes). The folded activations,
// scaled per token by 2^P so that |x' 2^P| < 256, are split into three e4m3
// terms h + m + l (about 12 significant bits, the precision of fp16) that
// form three B operands in 128B-swizzled shared memory and accumulate into the
// same fp32 TMEM accumulator; the epilogue multiplies by 2^(9 - P).
//
// CTA = 128 output rows x one K slice; the KS CTAs sharing the rows form a
// thread-block cluster and add their partial sums through distributed shared
// memory. Warp roles (10 warps):
//   0      producer: 4 KB code tiles -> shared-memory ring (cp.async.bulk)
//   1      TMEM owner; one thread issues the MMAs
//   2..5   converters: shared ring -> TMEM A slots (two units of 16 rows per
//          warp), then the epilogue (tcgen05.ld of their 32 accumulator rows)
//   6..9   fold: x -> per-token scale, x' = x_g A, three e4m3 B terms
// Producer and converters never touch x, so they run before the programmatic-
// launch wait: while the previous kernel finishes, this layer's codes already
// stream into shared memory and TMEM.
#include "common.cuh"
#include "internal.h"

namespace unisvq {
namespace {

constexpr int kThreads = 10 * 32;
constexpr int kFoldWarp0 = 6;
constexpr int kTmemCols = 256;
constexpr int kAColBase = 64;        // A slots start here; the accumulator uses [0, NTOK)
constexpr int kASlots = (kTmemCols - kAColBase) / 32;
constexpr int kMaxTokPerLaunch = 64;

struct DecodeArgs {
  const uint8_t* codes;
  const uint16_t* x;   // bf16 [M][K]
  uint16_t* y;         // bf16 [M][N]
  int M, N, K, KT, d;
  int kt_per_cta;
  float A[16];
  float B[4];
  float colnorm;       // max_c sum_r |A[r][c]|
  int* err;
};

template <int NTOK>
struct Cfg {
  static constexpr int kCodeStages = NTOK == 64 ? 4 : 8;
  static constexpr int kBStages = NTOK == 16 ? 4 : 2;
  static constexpr int kTermBytes = NTOK * 128;                  // one e4m3 B tile (128 columns)
  static constexpr int kBStageBytes = 3 * kTermBytes;
  static constexpr int kOffCode = 0;
  static constexpr int kOffB = kOffCode + kCodeStages * kTileBytes;
  static constexpr int kOffX = kOffB + kBStages * kBStageBytes;
  static constexpr int kXBytes = NTOK == 64 ? 8192 : 32768;      // staged x slice (bf16)
  static constexpr int kOffRed = kOffX + kXBytes;
  static constexpr int kRedBytes = (kTileRows + 8) * NTOK * 4;
  static constexpr int kOffBars = kOffRed + kRedBytes;
  static constexpr int kNumBars = 2 * kCodeStages + 2 * kASlots + 2 * kBStages + 4;
  static constexpr int kOffTok = kOffBars + kNumBars * 8;        // pexp[64], cpart[64]
  static constexpr int kOffMisc = kOffTok + 512;                 // tmem ptr, abort flag
  static constexpr int kSmem = kOffMisc + 64 + 1024;             // + alignment slack
  static constexpr uint32_t kIdesc =
      (1u << 4) | (0u << 7) | (0u << 10) | (static_cast<uint32_t>(NTOK >> 3) << 17) | ((128u >> 4) << 24);
};

// ---- tcgen05 wrappers ----------------------------------------------------------

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

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
__device__ __forceinline__ void fold4(const DecodeArgs& a, const float (&v)[4], float (&o)[4]) {
  if (a.d == 1) {
#pragma unroll
    for (int e = 0; e < 4; ++e) o[e] = v[e] * a.A[0];
  } else if (a.d == 2) {
    o[0] = fmaf(v[1], a.A[2], v[0] * a.A[0]);
    o[1] = fmaf(v[1], a.A[3], v[0] * a.A[1]);
    o[2] = fmaf(v[3], a.A[2], v[2] * a.A[0]);
    o[3] = fmaf(v[3], a.A[3], v[2] * a.A[1]);
  } else {
#pragma unroll
    for (int c = 0; c < 4; ++c)
      o[c] = fmaf(v[3], a.A[12 + c], fmaf(v[2], a.A[8 + c], fmaf(v[1], a.A[4 + c], v[0] * a.A[c])));
  }
}

// Activations x[k .. k+3] of one token as packed bf16 (zero at or past kend).
__device__ __forceinline__ uint2 load_x4(const uint16_t* row, int k, int kend, bool vec) {
  if (vec && k + 3 < kend) return ldg_v2(row + k);
  uint32_t e[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) e[j] = (k + j < kend) ? static_cast<uint32_t>(row[k + j]) : 0u;
  return make_uint2(e[0] | (e[1] << 16), e[2] | (e[3] << 16));
}

template <int NTOK>
__global__ void __launch_bounds__(kThreads, 2) decode_kernel(const __grid_constant__ DecodeArgs a) {
  using C = Cfg<NTOK>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024 - (raw & 1023)) & 1023);
  const uint32_t sbase = smem_u32(smem);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int KS = gridDim.x;
  const int kt0 = blockIdx.x * a.kt_per_cta;
  const int n_kt = min(a.kt_per_cta, a.KT - kt0);
  const int rb = blockIdx.y;

  const uint32_t bar0 = sbase + C::kOffBars;
  auto code_full = [&](int s) { return bar0 + 8u * s; };
  auto code_empty = [&](int s) { return bar0 + 8u * (C::kCodeStages + s); };
  auto a_full = [&](int s) { return bar0 + 8u * (2 * C::kCodeStages + s); };
  auto a_empty = [&](int s) { return bar0 + 8u * (2 * C::kCodeStages + kASlots + s); };
  auto b_full = [&](int s) { return bar0 + 8u * (2 * C::kCodeStages + 2 * kASlots + s); };
  auto b_empty = [&](int s) { return bar0 + 8u * (2 * C::kCodeStages + 2 * kASlots + C::kBStages + s); };
  const uint32_t bar_tail = bar0 + 8u * (2 * C::kCodeStages + 2 * kASlots + 2 * C::kBStages);
  const uint32_t d_full = bar_tail, tmem_ready = bar_tail + 8, fold_done = bar_tail + 16, drain = bar_tail + 24;
  int* pexp = reinterpret_cast<int*>(smem + C::kOffTok);
  float* cpart = reinterpret_cast<float*>(smem + C::kOffTok + 256);
  uint32_t* tmem_ptr = reinterpret_cast<uint32_t*>(smem + C::kOffMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::kOffMisc + 8);
  float* red = reinterpret_cast<float*>(smem + C::kOffRed);

  if (tid == 0) {
    for (int s = 0; s < C::kCodeStages; ++s) {
      mbar_init(code_full(s), 1);
      mbar_init(code_empty(s), 4);
    }
    for (int s = 0; s < kASlots; ++s) {
      mbar_init(a_full(s), 4);
      mbar_init(a_empty(s), 1);
    }
    for (int s = 0; s < C::kBStages; ++s) {
      mbar_init(b_full(s), 1);
      mbar_init(b_empty(s), 1);
    }
    mbar_init(d_full, 1);
    mbar_init(tmem_ready, 1);
    mbar_init(fold_done, 4);
    mbar_init(drain, 1);
    *abort_flag = n_kt <= 0 ? 1 : 0;
    if (n_kt <= 0) record_error(a.err, kErrBadLaunch);
    fence_mbar_init();
  }
  __syncthreads();
  if (KS > 1) cluster_arrive_relaxed();   // waited for before the first remote store
  pdl_launch_dependents();

  if (warp == 0) {
    // ---------------- producer: code tiles -> shared ring ----------------
    if (lane == 0 && !*abort_flag) {
      const uint64_t pol = policy_evict_first();
      const uint8_t* src = a.codes + (static_cast<size_t>(rb) * a.KT + kt0) * kTileBytes;
      int kt = 0;
      for (; kt < n_kt; ++kt) {
        const int s = kt % C::kCodeStages;
        if (kt >= C::kCodeStages &&
            !mbar_wait(code_empty(s), ((kt / C::kCodeStages) - 1) & 1, a.err, kErrTimeoutEmpty)) {
          *abort_flag = 1;
          break;
        }
        if (*abort_flag) break;
        mbar_arrive_expect_tx(code_full(s), kTileBytes);
        bulk_g2s(sbase + C::kOffCode + s * kTileBytes, src + static_cast<size_t>(kt) * kTileBytes, kTileBytes,
                 code_full(s), pol);
      }
      if (*abort_flag)   // copies nobody consumed must land before exit
        for (int j = kt - C::kCodeStages > 0 ? kt - C::kCodeStages : 0; j < kt; ++j)
          mbar_wait(code_full(j % C::kCodeStages), (j / C::kCodeStages) & 1, a.err, kErrTimeoutFull);
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
      for (int kt = 0; kt < n_kt && ok; ++kt) {
        const int sa = kt % kASlots, sb = kt % C::kBStages;
        ok = !*abort_flag && mbar_wait(a_full(sa), (kt / kASlots) & 1, a.err, kErrTimeoutFull) &&
             mbar_wait(b_full(sb), (kt / C::kBStages) & 1, a.err, kErrTimeoutFull);
        if (!ok) break;
        tc_fence_after();
        const uint32_t acol = tbase + kAColBase + 32 * sa;
        const uint32_t bst = sbase + C::kOffB + sb * C::kBStageBytes;
#pragma unroll
        for (int term = 0; term < 3; ++term) {
          const uint64_t bd = sw128_desc(bst + term * C::kTermBytes);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)   // K = 32 bytes per MMA inside the 128-byte swizzle row
            mma_f8_tmem_a(tbase, acol + 8 * kk, bd + 2 * kk, C::kIdesc, (kt | term | kk) != 0 ? 1u : 0u);
        }
        mma_commit(a_empty(sa));
        mma_commit(b_empty(sb));
      }
      if (ok) mma_commit(d_full);
      else *abort_flag = 1;
      mma_commit(drain);   // everything issued must retire before TMEM is released
      mbar_wait(drain, 0, a.err, kErrTimeoutMma);
    }
  } else if (warp < kFoldWarp0) {
    // ---------------- converters: shared ring -> TMEM A slots ----------------
    // Warp of TMEM lane quarter Q covers units 2Q and 2Q+1 (rows 32Q .. 32Q+31).
    // Lane 4g + t reads the words of rows g and g + 8 of a unit for column
    // quarter t (one 16-byte load, layout.h) and stores them as TMEM columns
    // 8k + 2t + e of lanes g and g + 8, k = 2h + s/2, e = s % 2: the K order
    // of the A slot is therefore a fixed permutation of the 128 columns, which
    // the fold applies to the B operand as well (a_slot_col below).
    const int q = warp & 3;                    // TMEM lane quarter
    bool ok = !*abort_flag && mbar_wait(tmem_ready, 0, a.err, kErrTimeoutFull);
    tc_fence_after();
    const uint32_t tbase = *tmem_ptr;
    const uint32_t tq = tbase + (static_cast<uint32_t>(32 * q) << 16);
    for (int kt = 0; kt < n_kt; ++kt) {
      const int s = kt % C::kCodeStages, sa = kt % kASlots;
      if (ok) ok = !*abort_flag && mbar_wait(code_full(s), (kt / C::kCodeStages) & 1, a.err, kErrTimeoutFull);
      uint4 c0 = make_uint4(0, 0, 0, 0), c1 = c0;
      if (ok) {
        const uint8_t* tile = smem + C::kOffCode + s * kTileBytes + (2 * q) * kUnitBytes + lane * 16;
        c0 = *reinterpret_cast<const uint4*>(tile);
        c1 = *reinterpret_cast<const uint4*>(tile + kUnitBytes);
      }
      __syncwarp();
      if (lane == 0 && ok) mbar_arrive(code_empty(s));
      uint32_t v0[16], v1[16];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int h = k >> 1, s0 = 2 * (k & 1);
        const uint32_t a0 = h ? c0.z : c0.x, a1 = h ? c0.w : c0.y;   // unit 2Q: rows g, g + 8
        const uint32_t b0 = h ? c1.z : c1.x, b1 = h ? c1.w : c1.y;   // unit 2Q+1
        v0[4 * k + 0] = extract4(a0, s0);
        v0[4 * k + 1] = extract4(a0, s0 + 1);
        v0[4 * k + 2] = extract4(a1, s0);
        v0[4 * k + 3] = extract4(a1, s0 + 1);
        v1[4 * k + 0] = extract4(b0, s0);
        v1[4 * k + 1] = extract4(b0, s0 + 1);
        v1[4 * k + 2] = extract4(b1, s0);
        v1[4 * k + 3] = extract4(b1, s0 + 1);
      }
      if (ok && kt >= kASlots) ok = !*abort_flag && mbar_wait(a_empty(sa), ((kt / kASlots) - 1) & 1, a.err, kErrTimeoutMma);
      if (ok) {
        tc_fence_after();
        tmem_st16x256b_x4(tq + kAColBase + 32 * sa, v0);
        tmem_st16x256b_x4(tq + (16u << 16) + kAColBase + 32 * sa, v1);
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
        tc_fence_before();
      }
      __syncwarp();
      if (lane == 0 && ok) mbar_arrive(a_full(sa));
      if (!ok) *abort_flag = 1;
    }

    // ---------------- epilogue: accumulator rows -> cluster reduction ----------------
    const int r = 32 * q + lane;               // accumulator row (TMEM lane) of this thread
    const uint32_t trow = tq;
    if (ok) ok = !*abort_flag && mbar_wait(d_full, 0, a.err, kErrTimeoutMma);
    if (ok) ok = mbar_wait(fold_done, 0, a.err, kErrTimeoutFull);
    if (!ok) *abort_flag = 1;
    const int rows_per = (kTileRows + KS - 1) / KS;
    const int owner = r / rows_per;
    const uint32_t slot_off =
        (static_cast<uint32_t>(blockIdx.x) * rows_per + (r - owner * rows_per)) * NTOK * 4u;
    const uint32_t red_addr = sbase + C::kOffRed;
    if (KS > 1) cluster_wait();
    tc_fence_after();
#pragma unroll
    for (int c0 = 0; c0 < NTOK; c0 += 16) {
      uint32_t dv[16];
      tmem_ld16(trow + c0, dv);
      asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int tok = c0 + j;
        if (ok && tok < a.M) {
          const float val = fmaf(__uint_as_float(dv[j]), exp2i(9 - pexp[tok]), cpart[tok]);
          const uint32_t off = slot_off + tok * 4u;
          if (KS > 1) st_shared_cluster_f32(map_shared_rank(red_addr + off, owner), val);
          else red[off / 4] = val;
        }
      }
    }
    tc_fence_before();
  } else {
    // ---------------- fold: x -> scaled three-term e4m3 B tiles ----------------
    const int fw = warp - kFoldWarp0;
    // Fold warp fw < kBStages owns B stage fw (k-tiles kt = fw mod kBStages),
    // so each stage has one writer and every wait on it is one phase behind.
    // The owner zeroes the rows of tokens >= M once (those rows stay zero).
    if (fw < C::kBStages)
      for (int tok = a.M; tok < NTOK; ++tok)
        for (int term = 0; term < 3; ++term)
          reinterpret_cast<uint32_t*>(smem + C::kOffB + fw * C::kBStageBytes + term * C::kTermBytes + tok * 128)[lane] = 0u;
    pdl_wait();   // x may be the previous kernel's output
    const int kbeg = kt0 * kTileCols;
    const int kend = min(a.K, (kt0 + n_kt) * kTileCols);
    const int kspan = n_kt * kTileCols;                       // staged row length (bf16)
    const bool vec8 = (a.K & 7) == 0;
    const bool staged = a.M * kspan * 2 <= C::kXBytes;
    uint16_t* xs = reinterpret_cast<uint16_t*>(smem + C::kOffX);
    // Pass 1: per-token max |x| (scale) and sum_k x[k] B[k mod d] over the
    // slice; warp fw owns tokens fw, fw+4, ...; 8 columns per lane per load,
    // 8 loads in flight. The slice is kept in shared memory when it fits.
    for (int tok = fw; tok < a.M; tok += 4) {
      const uint16_t* row = a.x + static_cast<size_t>(tok) * a.K;
      float mx = 0.f, cs = 0.f;
      for (int k0 = kbeg + 8 * lane; k0 < kbeg + kspan; k0 += 8 * 32 * 8) {
        uint4 u[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int k = k0 + 256 * j;
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
        for (int j = 0; j < 8; ++j) {
          const int k = k0 + 256 * j;
          if (k >= kbeg + kspan) break;
          if (staged) *reinterpret_cast<uint4*>(xs + tok * kspan + (k - kbeg)) = u[j];
          const uint32_t w4[4] = {u[j].x, u[j].y, u[j].z, u[j].w};
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            const float v0 = bf16_lo(w4[t]), v1 = bf16_hi(w4[t]);
            mx = fmaxf(mx, fmaxf(fabsf(v0), fabsf(v1)));
            cs = fmaf(v0, a.B[(2 * t) & (a.d - 1)], cs);
            cs = fmaf(v1, a.B[(2 * t + 1) & (a.d - 1)], cs);
          }
        }
      }
#pragma unroll
      for (int off = 16; off; off >>= 1) {
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
        cs += __shfl_xor_sync(0xffffffffu, cs, off);
      }
      if (lane == 0) {
        // 2^P puts the largest possible |x'| (<= max|x| * colnorm) below 2^8.
        const float bound = mx * a.colnorm;
        int e2 = 0;
        if (bound > 0.f) frexpf(bound, &e2);
        pexp[tok] = bound > 0.f ? max(-100, min(100, 8 - e2)) : 0;
        cpart[tok] = cs;
      }
    }
    // All fold warps need every token's scale (and staged x) from here on.
    named_barrier_sync(1, 4 * 32);
    if (lane == 0) mbar_arrive(fold_done);

    // Pass 2: warp fw folds k-tiles fw, fw + kBStages, ... (its own stage) for
    // all tokens; lane covers columns 4 lane .. 4 lane + 3 of the k-tile.
    bool ok = !*abort_flag;
    // Columns 4 lane .. 4 lane + 3 = 64h + 16t + 4s + (0..3) sit in A-slot
    // column 16h + 8(s/2) + 2t + s%2 (converter mapping), i.e. at bytes
    // 4 * that column of each 128-byte B row.
    const uint32_t a_slot_col = 16 * (lane >> 4) + 8 * ((lane & 3) >> 1) + 2 * ((lane >> 2) & 3) + (lane & 1);
    const uint32_t cidx = (a_slot_col & 3) * 4;
    const uint32_t chunk = a_slot_col >> 2;
    for (int kt = fw; fw < C::kBStages && kt < n_kt; kt += C::kBStages) {
      const int sb = fw;
      const int use = kt / C::kBStages;      // how many times stage sb was filled before
      if (ok && use > 0)
        ok = !*abort_flag && mbar_wait(b_empty(sb), (use - 1) & 1, a.err, kErrTimeoutMma);
      if (ok) {
        uint8_t* bst = smem + C::kOffB + sb * C::kBStageBytes;
        const int k = (kt0 + kt) * kTileCols + 4 * lane;
        for (int tok = 0; tok < a.M; ++tok) {
          uint2 xv;
          if (staged) {
            xv = *reinterpret_cast<const uint2*>(xs + tok * kspan + kt * kTileCols + 4 * lane);
          } else {
            xv = load_x4(a.x + static_cast<size_t>(tok) * a.K, k, kend, (a.K & 3) == 0);
          }
          const float v[4] = {bf16_lo(xv.x), bf16_hi(xv.x), bf16_lo(xv.y), bf16_hi(xv.y)};
          float o[4];
          fold4(a, v, o);
          const float sc = exp2i(pexp[tok]);
          uint16_t h0, m0, l0, h1, m1, l1;
          split3(pack_half2(o[0] * sc, o[1] * sc), h0, m0, l0);
          split3(pack_half2(o[2] * sc, o[3] * sc), h1, m1, l1);
          const uint32_t off = tok * 128 + ((chunk ^ (tok & 7)) << 4) + cidx;
          *reinterpret_cast<uint32_t*>(bst + off) = h0 | (static_cast<uint32_t>(h1) << 16);
          *reinterpret_cast<uint32_t*>(bst + C::kTermBytes + off) = m0 | (static_cast<uint32_t>(m1) << 16);
          *reinterpret_cast<uint32_t*>(bst + 2 * C::kTermBytes + off) = l0 | (static_cast<uint32_t>(l1) << 16);
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      }
      __syncwarp();
      if (lane == 0 && ok) mbar_arrive(b_full(sb));
      if (!ok) *abort_flag = 1;
    }
  }

  // ---------------- reduction over the K slices of the cluster ----------------
  __syncwarp();
  if (KS > 1) {
    if (warp < 2 || warp >= kFoldWarp0) cluster_wait();   // converters waited before their stores
    cluster_sync();
  } else {
    __syncthreads();
  }
  {
    const int rows_per = (kTileRows + KS - 1) / KS;
    const int r0 = static_cast<int>(blockIdx.x) * rows_per;
    const int nrows = max(0, min(kTileRows, r0 + rows_per) - r0);
    for (int idx = tid; idx < nrows * a.M; idx += kThreads) {
      const int tok = idx / nrows;
      const int rl = idx - tok * nrows;
      const int n = rb * kTileRows + r0 + rl;
      float s = 0.f;
      for (int qq = 0; qq < KS; ++qq) s += red[(qq * rows_per + rl) * NTOK + tok];
      if (n < a.N) a.y[static_cast<size_t>(tok) * a.N + n] = f32_to_bf16_rn(s);
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(*tmem_ptr), "r"(kTmemCols)
                 : "memory");
  }
}

template <int NTOK>
int resident_ctas_per_sm() {
  static int n = 0;
  if (!n) {
    cudaFuncSetAttribute(decode_kernel<NTOK>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<NTOK>::kSmem);
    cudaFuncSetAttribute(decode_kernel<NTOK>, cudaFuncAttributePreferredSharedMemoryCarveout,
                         cudaSharedmemCarveoutMaxShared);
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, decode_kernel<NTOK>, kThreads, Cfg<NTOK>::kSmem) !=
            cudaSuccess ||
        n < 1)
      n = 1;
    // Each resident CTA holds kTmemCols of the 512 TMEM columns.
    n = min(n, 512 / kTmemCols);
  }
  return n;
}

template <int NTOK>
unisvq_status launch_ntok(const unisvq_layer* L, const DecodePlan& p, const void* x, void* y, int M,
                          cudaStream_t s) {
  using C = Cfg<NTOK>;
  static bool attr_set[64] = {};
  const int dev = L->device;
  if (dev < 0 || dev >= 64) return UNISVQ_ERR_CUDA;
  if (!attr_set[dev]) {
    if (cudaFuncSetAttribute(decode_kernel<NTOK>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem) !=
            cudaSuccess ||
        cudaFuncSetAttribute(decode_kernel<NTOK>, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared) != cudaSuccess)
      return UNISVQ_ERR_CUDA;
    attr_set[dev] = true;
  }
  DecodeArgs a{};
  a.codes = L->codes;
  a.x = static_cast<const uint16_t*>(x);
  a.y = static_cast<uint16_t*>(y);
  a.M = M;
  a.N = L->N;
  a.K = L->K;
  a.KT = L->KT;
  a.d = L->d;
  a.kt_per_cta = p.kt_per_cta;
  for (int i = 0; i < 16; ++i) a.A[i] = L->A[i];
  for (int i = 0; i < 4; ++i) a.B[i] = L->B[i];
  a.colnorm = L->colnorm;
  a.err = device_error_word();

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.ks, p.nb, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = C::kSmem;
  cfg.stream = s;
  cudaLaunchAttribute attrs[2];
  attrs[0].id = cudaLaunchAttributeClusterDimension;
  attrs[0].val.clusterDim.x = p.ks;
  attrs[0].val.clusterDim.y = 1;
  attrs[0].val.clusterDim.z = 1;
  attrs[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attrs[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attrs;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, decode_kernel<NTOK>, a) == cudaSuccess ? UNISVQ_OK : UNISVQ_ERR_CUDA;
}

}  // namespace

DecodePlan plan_skinny(const unisvq_layer* L, int M) {
  DecodePlan p{};
  p.nt = M <= 16 ? 16 : (M <= 32 ? 32 : 64);
  p.nb = L->Np / kTileRows;
  const int occ = p.nt == 16 ? resident_ctas_per_sm<16>() : (p.nt == 32 ? resident_ctas_per_sm<32>()
                                                                         : resident_ctas_per_sm<64>());
  // Largest K split (cluster size <= 8, >= 1 k-tile per CTA) whose grid fits
  // in one wave of resident CTAs.
  const int slots = occ * L->num_sms;
  int ks = 1;
  for (int c = 8; c >= 1; --c)
    if (c <= L->KT && p.nb * c <= slots) {
      ks = c;
      break;
    }
  p.kt_per_cta = (L->KT + ks - 1) / ks;
  p.ks = (L->KT + p.kt_per_cta - 1) / p.kt_per_cta;
  p.smem = p.nt == 16 ? Cfg<16>::kSmem : (p.nt == 32 ? Cfg<32>::kSmem : Cfg<64>::kSmem);
  return p;
}

unisvq_status launch_skinny(const unisvq_layer* L, const void* x, void* y, int M, cudaStream_t s) {
  for (int m0 = 0; m0 < M; m0 += kMaxTokPerLaunch) {
    const int mc = M - m0 < kMaxTokPerLaunch ? M - m0 : kMaxTokPerLaunch;
    const DecodePlan p = plan_skinny(L, mc);
    const void* xs = static_cast<const uint16_t*>(x) + static_cast<size_t>(m0) * L->K;
    void* ys = static_cast<uint16_t*>(y) + static_cast<size_t>(m0) * L->N;
    unisvq_status st;
    if (p.nt == 16) st = launch_ntok<16>(L, p, xs, ys, mc, s);
    else if (p.nt == 32) st = launch_ntok<32>(L, p, xs, ys, mc, s);
    else st = launch_ntok<64>(L, p, xs, ys, mc, s);
    if (st != UNISVQ_OK) return st;
  }
  return UNISVQ_OK;
}

}  // namespace unisvq
