// Decode GEMV / skinny GEMM for M <= 32 tokens (HBM-bound path).
//
// Computes y = x W_hat^T through the fold of Eq. (col:matmul):
//   y[m, n] = sum_k x'[m, k] z[n, k] + c[m],
//   x'[m, g d + c] = sum_r x[m, g d + r] A[r][c]   (the row vectors X_i A),
//   c[m]          = sum_g x[m, g d .. g d + d - 1] . B  (the X_i B terms),
// so the 2-bit codes are never turned into weights: they go from the code
// stream straight into tensor-core A-operand registers.
//
// Per CTA: 128 output rows (8 consumer warps x 16 rows) times a slice of K;
// the KS CTAs that share the rows form a cluster and add their partial sums
// through distributed shared memory. A producer warp streams the slice's code
// tiles into a shared-memory ring with 1-D bulk copies before waiting on the
// previous kernel (codes never depend on it), so under programmatic dependent
// launch the code stream of this layer overlaps the tail of the last one.
//
// Code -> MMA operand: one AND per fp16x2 register (layout.h). The extracted
// halves are fp16 subnormals z * 4^s * 2^-24; the folded activations are
// stored as fp16 x' * 2^P * 4^-s (P per token, chosen so the largest |x'| in
// the CTA's slice stays below 2^15), so every product is x' z 2^(P-24) and the
// fp32 accumulator is rescaled by 2^(24-P) once at the end.
#include "common.cuh"
#include "internal.h"

namespace unisvq {
namespace {

constexpr int kDecWarps = 8;
constexpr int kDecThreads = (kDecWarps + 1) * 32;
constexpr int kDecRows = kDecWarps * kTileRows;   // 128 rows per CTA
constexpr int kKB = 2;                            // k-tiles per ring stage
constexpr int kStages = 4;
constexpr int kMaxTok = 32;
constexpr int kConsumerThreads = kDecWarps * 32;
constexpr uint32_t kFoldBarrier = 1;

struct DecodeArgs {
  const uint8_t* codes;
  const uint16_t* x;   // bf16 [M][K]
  uint16_t* y;         // bf16 [M][N]
  int M, N, K, KT, d;
  int kt_per_cta;
  float A[16];
  float B[4];
  float colnorm;
  int* err;
};

template <int NT>
struct DecCfg {
  static constexpr int CH = NT == 1 ? 8 : (NT == 2 ? 4 : 2);   // k-tiles per fold chunk
  static constexpr int MP = 8 * NT;                              // padded tokens
  static constexpr int kStageBytes = kDecWarps * kKB * kTileBytes;
  static constexpr int kXfragBytes = NT * CH * 8 * 32 * 8;       // one fold buffer
  static constexpr int kOffBars = 0;
  static constexpr int kOffTok = 128;
  static constexpr int kOffRing = 1024;
  static constexpr int kOffXfrag = kOffRing + kStages * kStageBytes;
  static constexpr int kOffRed = kOffXfrag + 2 * kXfragBytes;
  static constexpr int kSmem = kOffRed + kDecRows * MP * 4;
};

__device__ __forceinline__ void mma_f16_16816(float (&d)[4], uint32_t a0, uint32_t a1,
                                              uint32_t a2, uint32_t a3, uint32_t b0,
                                              uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Four consecutive activations x[k .. k+3] of one token (zero past K).
__device__ __forceinline__ void load4(const uint16_t* xr, int k, int K, float (&v)[4]) {
  if ((K & 3) == 0 && k + 3 < K) {
    const uint2 u = __ldg(reinterpret_cast<const uint2*>(xr + k));
    v[0] = bf16_lo(u.x);
    v[1] = bf16_hi(u.x);
    v[2] = bf16_lo(u.y);
    v[3] = bf16_hi(u.y);
  } else {
#pragma unroll
    for (int e = 0; e < 4; ++e)
      v[e] = (k + e < K) ? __uint_as_float(static_cast<uint32_t>(xr[k + e]) << 16) : 0.f;
  }
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

template <int NT>
__global__ void __launch_bounds__(kDecThreads, 2) decode_kernel(const __grid_constant__ DecodeArgs a) {
  using C = DecCfg<NT>;
  extern __shared__ __align__(1024) uint8_t smem[];
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const int KS = gridDim.x;
  const int kt0 = blockIdx.x * a.kt_per_cta;
  const int n_kt = min(a.kt_per_cta, a.KT - kt0);
  const int n_st = (n_kt + kKB - 1) / kKB;
  const int rt0 = blockIdx.y * kDecWarps;

  const uint32_t bar0 = smem_u32(smem + C::kOffBars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (kStages + s); };
  float* xmax = reinterpret_cast<float*>(smem + C::kOffTok);
  float* cpart = reinterpret_cast<float*>(smem + C::kOffTok + 128);
  int* pexp = reinterpret_cast<int*>(smem + C::kOffTok + 256);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::kOffTok + 384);
  float* red = reinterpret_cast<float*>(smem + C::kOffRed);

  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), kDecWarps);
    }
    *abort_flag = (n_kt <= 0) ? 1 : 0;
    if (n_kt <= 0) record_error(a.err, kErrBadLaunch);
    fence_mbar_init();
  }
  if (tid < kMaxTok) {
    xmax[tid] = 0.f;
    cpart[tid] = 0.f;
    pexp[tid] = 0;
  }
  {  // zero both fold buffers: tokens >= M stay zero for the whole kernel
    uint4* xf = reinterpret_cast<uint4*>(smem + C::kOffXfrag);
    for (int i = tid; i < 2 * C::kXfragBytes / 16; i += kDecThreads) xf[i] = make_uint4(0, 0, 0, 0);
  }
  __syncthreads();
  pdl_launch_dependents();

  int issued = 0;
  if (warp == kDecWarps) {
    // ---------------- producer: code tiles -> shared-memory ring ----------------
    if (lane == 0 && !*abort_flag) {
      const uint64_t pol = policy_evict_first();
      for (int st = 0; st < n_st; ++st) {
        const int slot = st % kStages;
        if (st >= kStages &&
            !mbar_wait(empty_bar(slot), ((st / kStages) - 1) & 1, a.err, kErrTimeoutEmpty)) {
          *abort_flag = 1;
          break;
        }
        if (*abort_flag) break;
        const int nk = min(kKB, n_kt - st * kKB);
        mbar_arrive_expect_tx(full_bar(slot), kDecWarps * nk * kTileBytes);
        const uint32_t dst = smem_u32(smem + C::kOffRing + slot * C::kStageBytes);
        for (int r = 0; r < kDecWarps; ++r) {
          const uint8_t* src =
              a.codes + (static_cast<size_t>(rt0 + r) * a.KT + kt0 + st * kKB) * kTileBytes;
          bulk_g2s(dst + r * kKB * kTileBytes, src, nk * kTileBytes, full_bar(slot), pol);
        }
        issued = st + 1;
      }
    }
  } else {
    // ---------------- consumers ----------------
    pdl_wait();   // x may be the previous kernel's output
    const int kend = min(a.K, (kt0 + n_kt) * kTileCols);
    const int kbeg = kt0 * kTileCols;

    // Per-token max |x| and partial sum_g x_g . B over this CTA's K slice.
    for (int tok = warp; tok < a.M; tok += kDecWarps) {
      const uint16_t* xr = a.x + static_cast<size_t>(tok) * a.K;
      float mx = 0.f, cp = 0.f;
      for (int k = kbeg + 4 * lane; k < kend; k += 128) {
        float v[4];
        load4(xr, k, a.K, v);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          mx = fmaxf(mx, fabsf(v[e]));
          cp = fmaf(v[e], a.B[e & (a.d - 1)], cp);
        }
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) {
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        cp += __shfl_xor_sync(0xffffffffu, cp, o);
      }
      if (lane == 0) {
        xmax[tok] = mx;
        cpart[tok] = cp;
      }
    }
    named_barrier_sync(kFoldBarrier, kConsumerThreads);
    if (tid < a.M) {
      // 2^P scales the largest possible |x'| (<= max|x| * colnorm) below 2^15.
      const float bound = xmax[tid] * a.colnorm;
      int e = 0;
      if (bound > 0.f) frexpf(bound, &e);   // bound < 2^e
      pexp[tid] = bound > 0.f ? max(-100, min(100, 15 - e)) : 0;
    }
    named_barrier_sync(kFoldBarrier, kConsumerThreads);

    auto fold = [&](int c) {
      uint2* xf = reinterpret_cast<uint2*>(smem + C::kOffXfrag + (c & 1) * C::kXfragBytes);
      const int ck0 = (kt0 + c * C::CH) * kTileCols;
      constexpr int units = C::CH * 32;   // 4-column units per token per chunk
      for (int u = tid; u < a.M * units; u += kConsumerThreads) {
        const int tok = u / units;
        const int j = u - tok * units;
        const int k = ck0 + 4 * j;
        uint32_t lo = 0, hi = 0;
        if (k < kend) {
          float v[4], o[4];
          load4(a.x + static_cast<size_t>(tok) * a.K, k, a.K, v);
          fold4(a, v, o);
          const int i = (k & 63) >> 4;
          const float sc0 = exp2i(pexp[tok] - 2 * pos_scale_class(2 * i));
          const float sc1 = exp2i(pexp[tok] - 2 * pos_scale_class(2 * i + 1));
          lo = pack_half2(o[0] * sc0, o[1] * sc0);
          hi = pack_half2(o[2] * sc1, o[3] * sc1);
        }
        xf[((tok >> 3) * C::CH * 8 + (j >> 2)) * 32 + (tok & 7) * 4 + (j & 3)] = make_uint2(lo, hi);
      }
    };

    const int n_ch = (n_kt + C::CH - 1) / C::CH;
    fold(0);
    float acc[NT][4];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[nt][e] = 0.f;

    bool ok = !*abort_flag;
    for (int kk = 0; kk < n_kt; ++kk) {
      const int st = kk / kKB;
      const int kb = kk - st * kKB;
      const int slot = st % kStages;
      if (kk % C::CH == 0) {
        named_barrier_sync(kFoldBarrier, kConsumerThreads);
        const int c = kk / C::CH;
        if (c + 1 < n_ch) fold(c + 1);
      }
      if (ok && kb == 0) {
        ok = !*abort_flag && mbar_wait(full_bar(slot), (st / kStages) & 1, a.err, kErrTimeoutFull);
        if (!ok) *abort_flag = 1;
      }
      if (ok) {
        const uint4 wv = *reinterpret_cast<const uint4*>(
            smem + C::kOffRing + slot * C::kStageBytes + (warp * kKB + kb) * kTileBytes + lane * 16);
        const uint2* xf = reinterpret_cast<const uint2*>(
            smem + C::kOffXfrag + ((kk / C::CH) & 1) * C::kXfragBytes);
        const int kl = kk % C::CH;
#pragma unroll
        for (int grp = 0; grp < 2; ++grp) {
          const uint32_t wg = grp ? wv.z : wv.x;    // row g
          const uint32_t wg8 = grp ? wv.w : wv.y;   // row g + 8
          const uint32_t wgs = wg >> 10, wg8s = wg8 >> 10;
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const uint32_t a0 = extract_pos(wg, wgs, 2 * i);
            const uint32_t a1 = extract_pos(wg8, wg8s, 2 * i);
            const uint32_t a2 = extract_pos(wg, wgs, 2 * i + 1);
            const uint32_t a3 = extract_pos(wg8, wg8s, 2 * i + 1);
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
              const uint2 b = xf[(nt * C::CH * 8 + kl * 8 + grp * 4 + i) * 32 + lane];
              mma_f16_16816(acc[nt], a0, a1, a2, a3, b.x, b.y);
            }
          }
        }
      }
      if (kb == kKB - 1 || kk == n_kt - 1) {
        __syncwarp();
        if (lane == 0 && ok) mbar_arrive(empty_bar(slot));
      }
    }

    // Partial outputs of this K slice: acc * 2^(24 - P) + partial c.
    const int g = lane >> 2, t = lane & 3;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int row = warp * 16 + g + ((e & 2) ? 8 : 0);
        const int tok = nt * 8 + 2 * t + (e & 1);
        if (tok < a.M) red[row * C::MP + tok] = fmaf(acc[nt][e], exp2i(24 - pexp[tok]), cpart[tok]);
      }
  }

  // ---------------- reduction over the K slices of the cluster ----------------
  __syncwarp();
  if (KS > 1) cluster_sync(); else __syncthreads();
  const int rank = static_cast<int>(blockIdx.x);
  const int rows_per = (kDecRows + KS - 1) / KS;
  const int r0 = rank * rows_per;
  const int nrows = max(0, min(kDecRows, r0 + rows_per) - r0);
  const uint32_t red_addr = smem_u32(red);
  for (int idx = tid; idx < nrows * a.M; idx += kDecThreads) {
    const int tok = idx / nrows;
    const int row = r0 + (idx - tok * nrows);
    const int n = blockIdx.y * kDecRows + row;
    float s = 0.f;
    if (KS > 1) {
      for (int q = 0; q < KS; ++q)
        s += ld_shared_cluster_f32(map_shared_rank(red_addr + (row * C::MP + tok) * 4u, q));
    } else {
      s = red[row * C::MP + tok];
    }
    if (n < a.N) a.y[static_cast<size_t>(tok) * a.N + n] = f32_to_bf16_rn(s);
  }
  // Copies still in flight after an abort must land before the CTA exits.
  if (warp == kDecWarps && lane == 0 && *abort_flag) {
    for (int st = max(0, issued - kStages); st < issued; ++st)
      mbar_wait(full_bar(st % kStages), (st / kStages) & 1, a.err, kErrTimeoutFull);
  }
  __syncwarp();
  if (KS > 1) cluster_sync();
}

template <int NT>
unisvq_status launch_nt(const unisvq_layer* L, const DecodePlan& p, const void* x, void* y, int M,
                        cudaStream_t s) {
  using C = DecCfg<NT>;
  static bool attr_set[64] = {};
  const int dev = L->device;
  if (dev < 0 || dev >= 64) return UNISVQ_ERR_CUDA;
  if (!attr_set[dev]) {
    if (cudaFuncSetAttribute(decode_kernel<NT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             C::kSmem) != cudaSuccess)
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
  cfg.blockDim = dim3(kDecThreads, 1, 1);
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
  return cudaLaunchKernelEx(&cfg, decode_kernel<NT>, a) == cudaSuccess ? UNISVQ_OK
                                                                       : UNISVQ_ERR_CUDA;
}

}  // namespace

DecodePlan plan_decode(const unisvq_layer* L, int M) {
  DecodePlan p{};
  p.nt = M <= 8 ? 1 : (M <= 16 ? 2 : 4);
  p.nb = L->Np / kDecRows;
  const int target = 2 * L->num_sms;
  int ks = 1;
  while (ks < 8 && p.nb * ks < target && ks * 2 <= L->KT) ks *= 2;
  p.kt_per_cta = (L->KT + ks - 1) / ks;
  p.ks = (L->KT + p.kt_per_cta - 1) / p.kt_per_cta;
  p.smem = p.nt == 1 ? DecCfg<1>::kSmem : (p.nt == 2 ? DecCfg<2>::kSmem : DecCfg<4>::kSmem);
  return p;
}

unisvq_status launch_decode(const unisvq_layer* L, const void* x, void* y, int M, cudaStream_t s) {
  // Token groups of at most 32 (one launch each) keep every M on this path.
  for (int m0 = 0; m0 < M; m0 += kMaxTok) {
    const int mc = M - m0 < kMaxTok ? M - m0 : kMaxTok;
    const DecodePlan p = plan_decode(L, mc);
    const void* xs = static_cast<const uint16_t*>(x) + static_cast<size_t>(m0) * L->K;
    void* ys = static_cast<uint16_t*>(y) + static_cast<size_t>(m0) * L->N;
    unisvq_status st;
    if (p.nt == 1) st = launch_nt<1>(L, p, xs, ys, mc, s);
    else if (p.nt == 2) st = launch_nt<2>(L, p, xs, ys, mc, s);
    else st = launch_nt<4>(L, p, xs, ys, mc, s);
    if (st != UNISVQ_OK) return st;
  }
  return UNISVQ_OK;
}

}  // namespace unisvq
