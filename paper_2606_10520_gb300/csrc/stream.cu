// Streaming decode GEMV: one launch per call, no thread-block cluster, one CTA
// per SM, M <= 8 tokens per launch.
//
// Computes y = x W_hat^T through the fold of Eq. (col:matmul):
//   y[m, n] = sum_k x'[m, k] z[n, k] + c[m],  x' = x_g A,  c = sum_g x_g . B,
// with the codes as fp16 subnormal A registers of m16n8k16 MMAs (the operand
// trick of gemv.cu: (w >> 8k) & (0x00030003 << 2j) is the fp16 pair
// z * 4^j * 2^-24) and the folded activations as fp16 B fragments
// x' * 2^P * 4^-j.
//
// Why this shape. A decode step is a chain of dependent calls, each moving a
// few MB of codes. The codes never depend on the previous kernel, so every
// CTA copies its slice of codes into shared memory (cp.async.bulk) before
// griddepcontrol.wait, while the previous call still runs. The grid has one
// CTA per SM and a CTA uses at most half of an SM (registers, shared memory),
// so the next call's CTAs fit beside it; the next call is released only once
// this one has passed its wait, so at most two calls share the SMs. After the
// wait a call folds x and runs its MMAs out of shared memory. Each CTA owns
// whole output rows over the whole of K, so no partial sum leaves the CTA: no
// cluster and no second kernel, both of which cost a call about a
// microsecond of dependent latency.
//
// CTA = a run of consecutive 16-row units of one layer (the layers of a
// grouped call get CTAs in proportion to their rows) x all k-tiles. Eight
// warps form a grid of WU unit groups x WK k-groups: warp (wu, wk) runs units
// wu, wu + WU, ... of the CTA over the k-tiles wk, wk + WK, ...; the WK partial
// sums of a row are added in shared memory at the end, in a fixed order.
//
// Fold, in chunks of CK k-tiles (double-buffered, one block barrier per
// chunk): an item is (k-tile, token); its 32 lanes load four columns each,
// take max |x| over the 128 columns (one scale 2^P per token and k-tile,
// |x' 2^P| < 2^15) and write the fp16 B pairs of their columns, from where
// lane 4g + t of an MMA warp reads the fragments of token g. The loads of
// chunk c + 1 are in flight while the MMAs of chunk c run. The accumulators of
// a token carry the scale of the last k-tile: before a k-tile's MMAs they are
// multiplied by 2^(P_new - P_old), exact powers of two.
//
// Codes: stage s of a CTA is its units' 512-byte pieces of k-tiles
// s SK .. s SK + SK - 1, fetched by one 4-D tensor copy per unit (the tile
// layout seen as [row block][k-tile][unit][512 bytes]; one copy moves SK x 512
// bytes, small copies being what limits a copy engine). A stage lives in slot
// s mod nslots; when the slice does not fit (nslots < stages), every warp
// releases a stage once it has read its k-tiles there and the last warp to do
// so refills the slot with stage s + nslots. Every wait is bounded.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "mma_sync.cuh"
#include "internal.h"

namespace unisvq {
namespace {

constexpr int kSWarps = 8;
constexpr int kSThreads = kSWarps * 32;
constexpr int kSItems = 8;                      // fold items per warp and chunk
constexpr int kSMaxGroup = UNISVQ_MAX_GROUP;
constexpr size_t kSSmemLimit = 112 * 1024;      // two CTAs (of this or another call) per SM
constexpr size_t kSFoldBudget = 32 * 1024;      // both chunk buffers of B fragments

struct StLayer {
  CUtensorMap tmap;   // the codes as uint64 [NB][KT][8][64], box 64 x 1 x SK x 1
  const uint8_t* codes;
  uint16_t* y;   // bf16 [M][N]
  int N;
  int units;     // Np / 16
  int cta0;      // first CTA of the layer
  int nctas;     // CTAs of the layer
  int d;
  float colnorm;
  float A[16];   // row-major d x d, d <= 4
  float B[4];
};

struct StArgs {
  const uint16_t* x;   // bf16 [M][K]
  int M, K, KT;
  int ucta;            // most units of any CTA
  int WU, WK;
  int CK;              // k-tiles per fold chunk (a multiple of WK)
  int SK;              // k-tiles per code stage (a multiple of WK, a power of two)
  int sk_log2;
  int nslots;
  int stage_bytes;     // ucta * SK * 512
  int off_b, off_ptab, off_bars, off_tok;
  int nlayers;
  int* err;
  StLayer layer[kSMaxGroup];
};

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
  return v;
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap* map, int c0, int c1, int c2, int c3,
                                            uint32_t bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint "
      "[%0], [%1, {%2, %3, %4, %5}], [%6], %7;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(bar), "l"(policy)
      : "memory");
}

// Non-blocking test of an mbarrier phase. Polling it a few times before the
// bounded (suspending) wait makes a wait on data that has already landed cost
// a few cycles instead of hundreds.
__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool wait_stage(uint32_t bar, uint32_t parity, int* err) {
#pragma unroll 1
  for (int i = 0; i < 32; ++i)
    if (mbar_test(bar, parity)) return true;
  return mbar_wait(bar, parity, err, kErrTimeoutFull);
}

// x'[c .. c+3] for the d-vectors inside x[c .. c+3] (c % 4 == 0): row vector x_g A
// (A row-major d x d in shared memory).
__device__ __forceinline__ void sfold4(int d, const float* A, const float (&v)[4], float (&o)[4]) {
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

// 2^e for e in [-252, 254] as a product of two exact powers of two.
__device__ __forceinline__ float exp2i_wide(int e) {
  const int h = e / 2;
  return exp2i(h) * exp2i(e - h);
}

template <int MT, int UW>
__global__ void __launch_bounds__(kSThreads, 2) stream_kernel(const __grid_constant__ StArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  const uint32_t sbase = smem_u32(smem);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int cta = static_cast<int>(blockIdx.x);
  const int M = a.M, KT = a.KT, K = a.K;

  // This CTA's layer, read with constant parameter offsets only.
  int li = 0;
#pragma unroll
  for (int i = 1; i < kSMaxGroup; ++i)
    if (i < a.nlayers && cta >= a.layer[i].cta0) li = i;
  const CUtensorMap* tmap = &a.layer[0].tmap;
  uint16_t* yout = nullptr;
  int N = 0, units = 0, cta0 = 0, nctas = 1, d = 1;
  float colnorm = 0.f, Bv[4];
  __shared__ float sA[16];
#pragma unroll
  for (int i = 0; i < kSMaxGroup; ++i)
    if (i == li) {
      tmap = &a.layer[i].tmap;
      yout = a.layer[i].y;
      N = a.layer[i].N;
      units = a.layer[i].units;
      cta0 = a.layer[i].cta0;
      nctas = a.layer[i].nctas;
      d = a.layer[i].d;
      colnorm = a.layer[i].colnorm;
#pragma unroll
      for (int e = 0; e < 4; ++e) Bv[e] = a.layer[i].B[e];
      if (tid < 16) sA[tid] = a.layer[i].A[tid];
    }
  const int lc = cta - cta0;
  const int u0 = static_cast<int>(static_cast<long long>(lc) * units / nctas);
  const int U = static_cast<int>(static_cast<long long>(lc + 1) * units / nctas) - u0;
  const int nslots = a.nslots, SK = a.SK;
  const int nstages = (KT + SK - 1) / SK;

  const uint32_t bars = sbase + a.off_bars;
  auto full = [&](int s) { return bars + 8u * s; };
  float* cpart = reinterpret_cast<float*>(smem + a.off_tok);             // [MT][8 warps]
  int* flags = reinterpret_cast<int*>(smem + a.off_tok + MT * kSWarps * 4);   // [0] abort, [1 + s] fills of slot s
  int* releases = flags + 1 + nslots;                                           // [s] warps done with slot s
  int* ptab = reinterpret_cast<int*>(smem + a.off_ptab);                 // [2][CK][MT] scale exponents

  if (tid == 0) {
    for (int s = 0; s < nslots; ++s) mbar_init(full(s), 1);
    fence_mbar_init();
  }
  for (int i = tid; i < 1 + 2 * nslots; i += kSThreads) flags[i] = 0;
  __syncthreads();
  if (tid == 0 && (U < 1 || U > a.ucta || M < 1 || M > MT)) {
    flags[0] = 1;
    record_error(a.err, kErrBadLaunch);
  }
  __syncthreads();
  const bool bad = flags[0] != 0;

  const uint64_t pol = policy_evict_first();
  // Stage st: k-tiles st SK .. st SK + SK - 1 of units u0 .. u0 + U - 1 into slot
  // st mod nslots, unit u at (u - u0) SK 512 (k-tiles past KT read as zero).
  auto issue_stage = [&](int st, int s) {
    const uint32_t dst = sbase + static_cast<uint32_t>(s) * a.stage_bytes;
    mbar_arrive_expect_tx(full(s), static_cast<uint32_t>(U * SK) * kUnitBytes);
    for (int u = 0; u < U; ++u)
      tma_load_4d(dst + static_cast<uint32_t>(u * SK) * kUnitBytes, tmap, 0, (u0 + u) & 7, st * SK, (u0 + u) >> 3,
                  full(s), pol);
    atomicAdd(&flags[1 + s], 1);
  };
  // Codes never depend on the previous kernel: fetch the first stages now.
  if (warp == 0 && !bad)
    for (int st = lane; st < nslots; st += 32) issue_stage(st, st);

  pdl_wait();                // x may be the previous kernel's output
  pdl_launch_dependents();   // the next call may now start fetching its codes

  const int WU = a.WU, WK = a.WK, CK = a.CK;
  const int wk = warp % WK, wu = warp / WK;
  const int g = lane >> 2, t = lane & 3;
  // fold role of a lane: columns 4 lane .. 4 lane + 3 of a k-tile = 64 h + 16 tq + 4 j + (0..3)
  const int fh = lane >> 4, ftq = (lane >> 2) & 3, fj = lane & 3;
  float Bcol[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) Bcol[e] = d == 1 ? Bv[0] : (d == 2 ? Bv[e & 1] : Bv[e]);
  constexpr uint32_t kKtBytes = MT * 256;   // B fragments of one k-tile
  const uint32_t wr_off = static_cast<uint32_t>(((fh * 2 + (fj >> 1)) * MT) * 64 + ftq * 16 + (fj & 1) * 8);
  const bool vec4 = (K & 3) == 0;
  // fold items per chunk: (k-tile it / MT, token it % MT), tokens past M skipped
  // (MT is a power of two: no integer division in the loops)

  float cs[MT];
#pragma unroll
  for (int m = 0; m < MT; ++m) cs[m] = 0.f;
  uint2 xl[kSItems];
  // All loads of a chunk go out before any of them is used (a select on a
  // loaded value right after each load would serialise them).
  auto load_chunk = [&](int c) {
#pragma unroll
    for (int j = 0; j < kSItems; ++j) xl[j] = make_uint2(0u, 0u);
#pragma unroll
    for (int j = 0; j < kSItems; ++j) {
      const int it = warp + kSWarps * j;
      const int kt = c * CK + it / MT, m = it % MT;
      const int k = kt * kTileCols + 4 * lane;
      if (it < CK * MT && m < M && kt < KT) {
        const uint16_t* row = a.x + static_cast<size_t>(m) * K;
        if (vec4 && k + 3 < K) {
          xl[j] = ldg_v2(row + k);
        } else {
          uint32_t e[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) e[q] = (k + q < K) ? static_cast<uint32_t>(row[k + q]) : 0u;
          xl[j] = make_uint2(e[0] | (e[1] << 16), e[2] | (e[3] << 16));
        }
      }
    }
  };
  auto fold_chunk = [&](int c) {
    const int buf = c & 1;
    float mx[kSItems];
#pragma unroll
    for (int j = 0; j < kSItems; ++j)
      mx[j] = fmaxf(fmaxf(fabsf(bf16_lo(xl[j].x)), fabsf(bf16_hi(xl[j].x))),
                    fmaxf(fabsf(bf16_lo(xl[j].y)), fabsf(bf16_hi(xl[j].y))));
#pragma unroll
    for (int off = 16; off; off >>= 1)
#pragma unroll
      for (int j = 0; j < kSItems; ++j) mx[j] = fmaxf(mx[j], __shfl_xor_sync(0xffffffffu, mx[j], off));
#pragma unroll
    for (int j = 0; j < kSItems; ++j) {
      const int it = warp + kSWarps * j;
      const int kl = it / MT, m = it % MT;
      if (it < CK * MT && m < M && c * CK + kl < KT) {
        const float v[4] = {bf16_lo(xl[j].x), bf16_hi(xl[j].x), bf16_lo(xl[j].y), bf16_hi(xl[j].y)};
        const int P = token_scale_exp(mx[j] * colnorm);
        const float cv = fmaf(v[0], Bcol[0], fmaf(v[1], Bcol[1], fmaf(v[2], Bcol[2], v[3] * Bcol[3])));
#pragma unroll
        for (int q = 0; q < MT; ++q)
          if (q == m) cs[q] += cv;
        float o[4];
        sfold4(d, sA, v, o);
        const float sc = exp2i(P - 2 * fj);
        uint2* dst = reinterpret_cast<uint2*>(smem + a.off_b + (buf * CK + kl) * kKtBytes + wr_off + m * 64);
        *dst = make_uint2(pack_half2(o[0] * sc, o[2] * sc), pack_half2(o[1] * sc, o[3] * sc));
        if (lane == 0) ptab[(buf * CK + kl) * MT + m] = P;
      }
    }
  };

  // acc[q]: unit wu + q WU (at most UW per warp); the first kDual units keep
  // the second half of every k-tile in acc2 (two independent MMA chains each).
  constexpr int kDual = 2;
  float acc[UW][4], acc2[kDual][4];
#pragma unroll
  for (int q = 0; q < UW; ++q)
#pragma unroll
    for (int e = 0; e < 4; ++e) acc[q][e] = 0.f;
#pragma unroll
  for (int q = 0; q < kDual; ++q)
#pragma unroll
    for (int e = 0; e < 4; ++e) acc2[q][e] = 0.f;
  int po0 = 0, po1 = 0;   // scale exponents of tokens 2t, 2t + 1 carried by acc
  bool ok = !bad;
  int cur_st = -1, slot = 0;
  uint32_t phase = 0;
  if (ok) {
    load_chunk(0);
    fold_chunk(0);
  }
  __syncthreads();
  const int nchunks = (KT + CK - 1) / CK;
  for (int c = 0; c < nchunks; ++c) {
    const bool more = c + 1 < nchunks;
    if (more && ok) load_chunk(c + 1);   // in flight during this chunk's MMAs
    const int buf = c & 1;
    for (int kl = wk; kl < CK && ok; kl += WK) {
      const int i = c * CK + kl;
      if (i >= KT) break;
      // ---- B fragments and scales of k-tile i ----
      const uint32_t bk = sbase + a.off_b + static_cast<uint32_t>(buf * CK + kl) * kKtBytes;
      uint4 bf[2][2];
#pragma unroll
      for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int jp = 0; jp < 2; ++jp)
          bf[h][jp] = g < M ? lds128(bk + static_cast<uint32_t>(((h * 2 + jp) * MT + g) * 64 + t * 16))
                            : make_uint4(0u, 0u, 0u, 0u);
      const int* pk = ptab + (buf * CK + kl) * MT;
      const int pn0 = 2 * t < M ? pk[2 * t] : 0;
      const int pn1 = 2 * t + 1 < M ? pk[2 * t + 1] : 0;
      if (pn0 != po0 || pn1 != po1) {   // accumulators to this k-tile's scale
        const float f0 = exp2i_wide(pn0 - po0), f1 = exp2i_wide(pn1 - po1);
#pragma unroll
        for (int q = 0; q < UW; ++q) {
          acc[q][0] *= f0;
          acc[q][1] *= f1;
          acc[q][2] *= f0;
          acc[q][3] *= f1;
        }
#pragma unroll
        for (int q = 0; q < kDual; ++q) {
          acc2[q][0] *= f0;
          acc2[q][1] *= f1;
          acc2[q][2] *= f0;
          acc2[q][3] *= f1;
        }
        po0 = pn0;
        po1 = pn1;
      }
      // ---- codes of k-tile i: stage st in slot st mod nslots (tracked, the
      // warp's k-tiles visit the stages in order) ----
      const int st = i >> a.sk_log2;
      if (st != cur_st) {
        if (cur_st >= 0 && ++slot == nslots) {
          slot = 0;
          phase ^= 1u;
        }
        cur_st = st;
        ok = wait_stage(full(slot), phase, a.err);
        if (!ok) break;
      }
      const uint32_t sl = sbase + static_cast<uint32_t>(slot) * a.stage_bytes +
                          static_cast<uint32_t>(i & (SK - 1)) * kUnitBytes + lane * 16;
#pragma unroll
      for (int q = 0; q < UW; ++q) {
        const int ul = wu + q * WU;
        if (ul < U) {
          const uint4 cw = lds128(sl + static_cast<uint32_t>(ul * SK) * kUnitBytes);
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const uint32_t wa = h ? cw.z : cw.x, wb = h ? cw.w : cw.y;   // rows g, g + 8
            const uint32_t was = wa >> 8, wbs = wb >> 8;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const uint32_t msk = 0x00030003u << (2 * j);
              const uint4 b4 = bf[h][j >> 1];
              const uint2 b = (j & 1) ? make_uint2(b4.z, b4.w) : make_uint2(b4.x, b4.y);
              if (q < kDual && h == 1)
                mma_16816(acc2[q < kDual ? q : 0], wa & msk, wb & msk, was & msk, wbs & msk, b);
              else
                mma_16816(acc[q], wa & msk, wb & msk, was & msk, wbs & msk, b);
            }
          }
        }
      }
      // ---- after this warp's last k-tile of the stage: release; the last warp refills ----
      if (st + nslots < nstages && i + WK >= (st + 1) * SK) {
        __syncwarp();
        if (lane == 0) {
          __threadfence_block();
          if (atomicAdd(&releases[slot], 1) == kSWarps - 1) {
            releases[slot] = 0;
            __threadfence_block();
            fence_proxy_async_smem();
            issue_stage(st + nslots, slot);
          }
        }
      }
    }
    if (more && ok) fold_chunk(c + 1);
    if (!ok) flags[0] = 1;
    __syncthreads();   // chunk c's fragments are read, chunk c + 1's written
  }

  // ---- c sums: each warp's share of every token ----
#pragma unroll
  for (int m = 0; m < MT; ++m) {
    float cv = cs[m];
#pragma unroll
    for (int off = 16; off; off >>= 1) cv += __shfl_xor_sync(0xffffffffu, cv, off);
    if (lane == 0) cpart[m * kSWarps + warp] = cv;
  }
  __syncthreads();   // every stage consumed: the ring becomes the reduction buffer
  if (flags[0] != 0) {
    // copies that nobody consumed must land before the CTA exits
    for (int s = tid; s < nslots; s += kSThreads) {
      const int f = flags[1 + s];
      if (f > 0) mbar_wait(full(s), static_cast<uint32_t>((f - 1) & 1), a.err, kErrTimeoutFull);
    }
    return;
  }
#pragma unroll
  for (int q = 0; q < kDual; ++q)
#pragma unroll
    for (int e = 0; e < 4; ++e) acc[q][e] += acc2[q][e];
  float* red = reinterpret_cast<float*>(smem);   // [ucta * 16 rows][MT tokens][WK]
  {
    const float s0 = exp2i(24 - po0), s1 = exp2i(24 - po1);
#pragma unroll
    for (int q = 0; q < UW; ++q) {
      const int ul = wu + q * WU;
      if (ul < U) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int row = ul * 16 + g + ((e & 2) ? 8 : 0);
          const int tok = 2 * t + (e & 1);
          if (tok < M) red[(row * MT + tok) * WK + wk] = acc[q][e] * ((e & 1) ? s1 : s0);
        }
      }
    }
  }
  __syncthreads();
  const int rows = U * 16;
  for (int tok = 0; tok < M; ++tok)
  for (int r = tid; r < rows; r += kSThreads) {
    const float* pr = red + (r * MT + tok) * WK;
    float sum = 0.f;
    for (int q = 0; q < WK; ++q) sum += pr[q];
    float cv = 0.f;
#pragma unroll
    for (int w = 0; w < kSWarps; ++w) cv += cpart[tok * kSWarps + w];
    const int n = u0 * 16 + r;
    if (n < N) yout[static_cast<size_t>(tok) * N + n] = f32_to_bf16_rn(sum + cv);
  }
}

template <int MT, int UW>
bool stream_set_attrs(int dev) {
  static bool done[64] = {};
  if (dev < 0 || dev >= 64) return false;
  if (!done[dev]) {
    if (cudaFuncSetAttribute(stream_kernel<MT, UW>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(kSSmemLimit)) != cudaSuccess ||
        cudaFuncSetAttribute(stream_kernel<MT, UW>, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared) != cudaSuccess)
      return false;
    done[dev] = true;
  }
  return true;
}

template <int MT, int UW>
cudaError_t launch_mt_uw(const cudaLaunchConfig_t& cfg, const StArgs& a, int dev) {
  if (!stream_set_attrs<MT, UW>(dev)) return cudaErrorUnknown;
  return cudaLaunchKernelEx(&cfg, stream_kernel<MT, UW>, a);
}

template <int MT>
cudaError_t launch_mt(const cudaLaunchConfig_t& cfg, const StArgs& a, int dev, int uw) {
  return uw == 2 ? launch_mt_uw<MT, 2>(cfg, a, dev) : (uw == 4 ? launch_mt_uw<MT, 4>(cfg, a, dev)
                                                                : launch_mt_uw<MT, 8>(cfg, a, dev));
}

}  // namespace

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  }
  return fn;
}

// CTAs of each layer of a streaming launch: one per SM in all (or one per
// unit if there are fewer units), in proportion to the layers' rows so that
// the largest run of units per CTA is as short as possible.
static void stream_split(const unisvq_layer* const* Ls, int n, int num_sms, int* nctas) {
  int units[kSMaxGroup], total = 0;
  for (int i = 0; i < n; ++i) {
    units[i] = Ls[i]->Np / kUnitRows;
    total += units[i];
  }
  const int budget = total < num_sms ? total : num_sms;
  int used = 0;
  for (int i = 0; i < n; ++i) {
    nctas[i] = static_cast<int>(static_cast<long long>(budget) * units[i] / total);
    if (nctas[i] < 1) nctas[i] = 1;
    used += nctas[i];
  }
  while (used < budget) {   // one more CTA to the layer with the longest runs
    int best = -1, worst = 0;
    for (int i = 0; i < n; ++i) {
      const int run = (units[i] + nctas[i] - 1) / nctas[i];
      if (nctas[i] < units[i] && run > worst) {
        worst = run;
        best = i;
      }
    }
    if (best < 0) break;
    ++nctas[best];
    ++used;
  }
}

StreamPlan plan_stream(const unisvq_layer* const* Ls, int n, int M) {
  StreamPlan p{};
  if (n < 1 || n > kSMaxGroup || M < 1 || M > kStreamMaxTok) return p;
  const int KT = Ls[0]->KT;
  int nctas[kSMaxGroup];
  stream_split(Ls, n, Ls[0]->num_sms, nctas);
  int U = 0, ctas = 0;
  for (int i = 0; i < n; ++i) {
    const int units = Ls[i]->Np / kUnitRows;
    const int run = (units + nctas[i] - 1) / nctas[i];
    U = run > U ? run : U;
    ctas += nctas[i];
  }
  p.ctas = ctas;
  p.ucta = U;
  p.WU = 1;
  while ((U + p.WU - 1) / p.WU > 8) p.WU *= 2;
  if (p.WU > kSWarps) return StreamPlan{};
  p.WK = kSWarps / p.WU;
  const int uw = (U + p.WU - 1) / p.WU;
  p.uw = uw <= 2 ? 2 : (uw <= 4 ? 4 : 8);
  p.mt = M <= 1 ? 1 : (M <= 2 ? 2 : (M <= 4 ? 4 : 8));
  // fold chunk: kSItems items per warp (CK * M <= 64) and both buffers in kSFoldBudget
  int ck = kSItems * kSWarps / p.mt;   // items = ck * mt
  const int ck_fit = static_cast<int>(kSFoldBudget / (2 * static_cast<size_t>(p.mt) * 256));
  ck = ck < ck_fit ? ck : ck_fit;
  const int kt_up = (KT + p.WK - 1) / p.WK * p.WK;
  ck = ck < kt_up ? ck : kt_up;
  ck = ck / p.WK * p.WK;
  if (ck < p.WK) return StreamPlan{};
  p.ck = ck;
  // Shared memory: [code ring | reduction buffer (aliased)] [B fragments of
  // two chunks] [their scale exponents] [mbarriers] [c sums, flags]; the ring
  // takes what the rest leaves. Code stages of SK k-tiles (8, or fewer when
  // the ring would otherwise hold fewer than three stages of a long slice).
  const size_t bfrag = (ck < KT ? 2 : 1) * static_cast<size_t>(ck) * p.mt * 256;   // one buffer if one chunk
  const size_t ptab = (ck < KT ? 2 : 1) * static_cast<size_t>(ck) * p.mt * 4;
  const size_t fixed = bfrag + ptab + 256 + static_cast<size_t>(p.mt) * kSWarps * 4 + 64;
  if (fixed >= kSSmemLimit) return StreamPlan{};
  int sk = 8, ns = 0;
  for (;; sk /= 2) {
    const size_t per_slot = static_cast<size_t>(U) * sk * kUnitBytes + 8 + 8;
    const int nst = (KT + sk - 1) / sk;
    ns = static_cast<int>((kSSmemLimit - fixed) / per_slot);
    if (ns > nst) ns = nst;
    const int want = nst < 3 ? nst : 3;
    if (ns >= want || sk / 2 < p.WK) break;
  }
  if (ns < 1) return StreamPlan{};
  p.sk = sk;
  p.stage_bytes = U * sk * kUnitBytes;
  p.nslots = ns;
  const size_t ring = static_cast<size_t>(ns) * p.stage_bytes;
  const size_t red = static_cast<size_t>(U) * 16 * p.mt * p.WK * 4;
  size_t off = ring > red ? ring : red;
  off = (off + 127) / 128 * 128;
  p.off_b = static_cast<int>(off);
  off += bfrag;
  p.off_ptab = static_cast<int>(off);
  off += ptab;
  off = (off + 15) / 16 * 16;
  p.off_bars = static_cast<int>(off);
  off += static_cast<size_t>(ns) * 8;
  off = (off + 15) / 16 * 16;
  p.off_tok = static_cast<int>(off);
  off += static_cast<size_t>(p.mt) * kSWarps * 4 + static_cast<size_t>(1 + 2 * ns) * 4;
  p.smem = (off + 127) / 128 * 128;
  if (p.smem > kSSmemLimit) return StreamPlan{};
  p.ok = true;
  return p;
}

bool stream_supported(const unisvq_layer* const* Ls, int n, int M) {
  if (n < 1 || n > kSMaxGroup) return false;
  for (int i = 0; i < n; ++i)
    if (Ls[i]->bits != 2 || Ls[i]->grouped || Ls[i]->d > 4 || Ls[i]->K != Ls[0]->K) return false;
  for (int m = 1; m <= kStreamMaxTok && m <= M; ++m)   // every chunk size a launch of M tokens uses
    if (!plan_stream(Ls, n, m).ok) return false;
  return true;
}

unisvq_status launch_stream_group(const unisvq_layer* const* Ls, int n, const void* x, void* const* ys, int M,
                                  cudaStream_t s) {
  if (!stream_supported(Ls, n, M)) return UNISVQ_ERR_UNSUPPORTED;
  int nctas[kSMaxGroup];
  stream_split(Ls, n, Ls[0]->num_sms, nctas);
  const PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
  if (!enc) return UNISVQ_ERR_CUDA;
  for (int m0 = 0; m0 < M; m0 += kStreamMaxTok) {
    const int mc = M - m0 < kStreamMaxTok ? M - m0 : kStreamMaxTok;
    const StreamPlan p = plan_stream(Ls, n, mc);
    if (!p.ok) return UNISVQ_ERR_UNSUPPORTED;
    StArgs a{};
    a.x = static_cast<const uint16_t*>(x) + static_cast<size_t>(m0) * Ls[0]->K;
    a.M = mc;
    a.K = Ls[0]->K;
    a.KT = Ls[0]->KT;
    a.ucta = p.ucta;
    a.WU = p.WU;
    a.WK = p.WK;
    a.CK = p.ck;
    a.SK = p.sk;
    a.sk_log2 = p.sk == 1 ? 0 : (p.sk == 2 ? 1 : (p.sk == 4 ? 2 : (p.sk == 8 ? 3 : 4)));
    a.nslots = p.nslots;
    a.stage_bytes = p.stage_bytes;
    a.off_b = p.off_b;
    a.off_ptab = p.off_ptab;
    a.off_bars = p.off_bars;
    a.off_tok = p.off_tok;
    a.nlayers = n;
    a.err = device_error_word();
    int cta0 = 0;
    for (int i = 0; i < n; ++i) {
      const unisvq_layer* L = Ls[i];
      StLayer& l = a.layer[i];
      // the codes as uint64 [Np/128][KT][8 units][64], one box = one unit x SK k-tiles
      const cuuint64_t dims[4] = {64, 8, static_cast<cuuint64_t>(L->KT), static_cast<cuuint64_t>(L->Np / kTileRows)};
      const cuuint64_t strides[3] = {kUnitBytes, kTileBytes, static_cast<cuuint64_t>(L->KT) * kTileBytes};
      const cuuint32_t box[4] = {64, 1, static_cast<cuuint32_t>(p.sk), 1};
      const cuuint32_t estr[4] = {1, 1, 1, 1};
      if (enc(&l.tmap, CU_TENSOR_MAP_DATA_TYPE_UINT64, 4, L->codes, dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return UNISVQ_ERR_CUDA;
      l.codes = L->codes;
      l.y = static_cast<uint16_t*>(ys[i]) + static_cast<size_t>(m0) * L->N;
      l.N = L->N;
      l.units = L->Np / kUnitRows;
      l.cta0 = cta0;
      l.nctas = nctas[i];
      l.d = L->d;
      l.colnorm = L->colnorm;
      for (int e = 0; e < 16; ++e) l.A[e] = e < L->d * L->d ? L->A[e] : 0.f;
      for (int e = 0; e < 4; ++e) l.B[e] = e < L->d ? L->B[e] : 0.f;
      cta0 += nctas[i];
    }
    if (cta0 != p.ctas) return UNISVQ_ERR_UNSUPPORTED;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(p.ctas, 1, 1);
    cfg.blockDim = dim3(kSThreads, 1, 1);
    cfg.dynamicSmemBytes = p.smem;
    cfg.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    const int dev = Ls[0]->device;
    const cudaError_t e = p.mt == 1   ? launch_mt<1>(cfg, a, dev, p.uw)
                          : p.mt == 2 ? launch_mt<2>(cfg, a, dev, p.uw)
                          : p.mt == 4 ? launch_mt<4>(cfg, a, dev, p.uw)
                                      : launch_mt<8>(cfg, a, dev, p.uw);
    if (e != cudaSuccess) return UNISVQ_ERR_CUDA;
  }
  return UNISVQ_OK;
}

}  // namespace unisvq
