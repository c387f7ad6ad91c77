// GEMV for M <= 16 tokens per launch: register-operand tensor-core MMAs.
//
// Computes y = x W_hat^T through the fold of Eq. (col:matmul):
//   y[m, n] = sum_k x'[m, k] z[n, k] + c[m],  x' = x_g A,  c = sum_g x_g . B.
// For one or a few tokens the contraction is tiny, so the limit is the work
// per weight. Each code goes straight from a word of the packed layout into
// an m16n8k16 A-operand register: with w a code word of row n (columns
// 16 t + 4 s + b at bits 8b + 2s, layout.h),
//   w        & (0x00030003 << 2s)  = fp16 pair (z[4s], z[4s+2]) * 4^s * 2^-24,
//   (w >> 8) & (0x00030003 << 2s)  = fp16 pair (z[4s+1], z[4s+3]) * 4^s * 2^-24,
// fp16 subnormals (exact in the tensor core): one shift and eight ANDs turn 16
// codes into 8 registers. In MMA j of a 64-column half, thread t (of row
// group g) supplies word t of its two rows with s = j, so the MMA covers the
// 16 columns 16 t + 4 j + b; the folded activations are stored in the same
// order as fp16 x' * 2^P * 4^-j. Products are x' z 2^(P-24); the fp32 sums
// are rescaled by 2^(24-P) at the end.
//
// CTA = 128 output rows x one K slice, 8 warps of 16 rows. Each thread keeps
// 8 k-tiles of its code words in flight with plain coalesced loads (the first
// ones issued before the programmatic-launch wait, since codes never depend on
// the previous kernel); the K slices of a row block form a cluster and add
// their partial sums through distributed shared memory.
#include "common.cuh"
#include "internal.h"

namespace unisvq {
namespace {

constexpr int kGWarps = 8;                     // warps; warp w owns rows 16w .. 16w+15
constexpr int kGThreads = kGWarps * 32;
constexpr int kGDepth = 8;                     // k-tiles of codes in flight per thread
constexpr int kGMaxTok = 16;

struct GemvArgs {
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
struct GCfg {
  static constexpr int CHB = kGDepth;                            // k-tiles per fold chunk
  static constexpr int kFragTile = 8 * 32 * 8 * NT;              // B fragments of one k-tile
  static constexpr int kOffX = 0;
  static constexpr int kXBytes = NT == 1 ? 16384 : 32768;        // staged x slice (bf16)
  static constexpr int kOffF = kOffX + kXBytes;
  static constexpr int kFBytes = CHB * kFragTile;                // one fold buffer
  static constexpr int kOffRed = kOffF + 2 * kFBytes;
  static constexpr int kRedBytes = (kTileRows + 8) * 8 * NT * 4;
  static constexpr int kOffTok = kOffRed + kRedBytes;            // pexp[32], cpart[32]
  static constexpr int kOffMisc = kOffTok + 256;
  static constexpr int kSmem = kOffMisc + 64;
};

__device__ __forceinline__ void mma_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                          uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// x'[c .. c+3] for the d-vectors inside x[c .. c+3] (c % 4 == 0): row vector x_g A.
__device__ __forceinline__ void gfold4(const GemvArgs& a, const float (&v)[4], float (&o)[4]) {
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
__global__ void __launch_bounds__(kGThreads, 2) gemv_kernel(const __grid_constant__ GemvArgs a) {
  using C = GCfg<NT>;
  extern __shared__ __align__(128) uint8_t smem[];
  const uint32_t sbase = smem_u32(smem);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int KS = gridDim.x;
  const int kt0 = blockIdx.x * a.kt_per_cta;
  const int n_kt = min(a.kt_per_cta, a.KT - kt0);
  const int rb = blockIdx.y;

  int* pexp = reinterpret_cast<int*>(smem + C::kOffTok);
  float* cpart = reinterpret_cast<float*>(smem + C::kOffTok + 128);
  float* red = reinterpret_cast<float*>(smem + C::kOffRed);
  // A valid plan gives every CTA at least one k-tile; otherwise flag the error
  // and fall through with empty loops so the cluster barrier is still reached.
  if (n_kt <= 0 && tid == 0) record_error(a.err, kErrBadLaunch);
  {  // fold buffers start at zero: fragments of tokens >= M stay zero
    uint4* f = reinterpret_cast<uint4*>(smem + C::kOffF);
    for (int i = tid; i < 2 * C::kFBytes / 16; i += kGThreads) f[i] = make_uint4(0, 0, 0, 0);
  }

  // Codes: warp w reads, for each k-tile, word t (lane % 4) of rows r0 = 16w + g
  // and r0 + 8 in both 64-column halves (4 x 4 bytes; each warp load instruction
  // covers 128 contiguous bytes). kGDepth k-tiles are kept in flight; the first
  // ones are requested before the programmatic-launch wait (codes never depend
  // on the previous kernel).
  const int g = lane >> 2, t = lane & 3;
  const int r0 = 16 * warp + g;
  const uint8_t* cbase = a.codes + (static_cast<size_t>(rb) * a.KT + kt0) * kTileBytes + 4 * t;
  auto load_codes = [&](int kt, uint32_t (&w)[4]) {
    if (kt < n_kt) {
      const uint8_t* tb = cbase + static_cast<size_t>(kt) * kTileBytes;
      w[0] = __ldg(reinterpret_cast<const uint32_t*>(tb + tile_row_offset(r0, 0)));
      w[1] = __ldg(reinterpret_cast<const uint32_t*>(tb + tile_row_offset(r0 + 8, 0)));
      w[2] = __ldg(reinterpret_cast<const uint32_t*>(tb + tile_row_offset(r0, 1)));
      w[3] = __ldg(reinterpret_cast<const uint32_t*>(tb + tile_row_offset(r0 + 8, 1)));
    }
  };
  uint32_t cw[kGDepth][4];
#pragma unroll
  for (int i = 0; i < kGDepth; ++i) load_codes(i, cw[i]);
  __syncthreads();
  pdl_launch_dependents();

  pdl_wait();   // x may be the previous kernel's output
  const int kbeg = kt0 * kTileCols;
  const int kend = min(a.K, (kt0 + n_kt) * kTileCols);
  const int kspan = n_kt * kTileCols;
  const bool vec8 = (a.K & 7) == 0;
  const bool staged = a.M * kspan * 2 <= C::kXBytes;
  uint16_t* xs = reinterpret_cast<uint16_t*>(smem + C::kOffX);
  // Pass 1: per-token max |x| and sum_k x[k] B[k mod d] over the slice;
  // warp w owns tokens w, w + 8; 8 columns per lane per load, 8 in flight.
  for (int tok = warp; tok < a.M; tok += kGWarps) {
    const uint16_t* row = a.x + static_cast<size_t>(tok) * a.K;
    float mx = 0.f, cs = 0.f;
    for (int k0 = kbeg + 8 * lane; k0 < kbeg + kspan; k0 += 8 * 32 * 8) {
      uint4 u[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int k = k0 + 256 * j;
        if (vec8 && k + 7 < kend) {
          u[j] = __ldg(reinterpret_cast<const uint4*>(row + k));
        } else {
          uint32_t e[8];
#pragma unroll
          for (int q = 0; q < 8; ++q) e[q] = (k + q < kend) ? static_cast<uint32_t>(row[k + q]) : 0u;
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
        for (int q = 0; q < 4; ++q) {
          const float v0 = bf16_lo(w4[q]), v1 = bf16_hi(w4[q]);
          mx = fmaxf(mx, fmaxf(fabsf(v0), fabsf(v1)));
          cs = fmaf(v0, a.B[(2 * q) & (a.d - 1)], cs);
          cs = fmaf(v1, a.B[(2 * q + 1) & (a.d - 1)], cs);
        }
      }
    }
#pragma unroll
    for (int off = 16; off; off >>= 1) {
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
      cs += __shfl_xor_sync(0xffffffffu, cs, off);
    }
    if (lane == 0) {
      // 2^P puts the largest possible |x'| (<= max|x| * colnorm) below 2^15 (fp16).
      const float bound = mx * a.colnorm;
      int e2 = 0;
      if (bound > 0.f) frexpf(bound, &e2);
      pexp[tok] = bound > 0.f ? max(-100, min(100, 15 - e2)) : 0;
      cpart[tok] = cs;
    }
  }
  __syncthreads();

  // Fold chunk ch (CHB k-tiles) into B fragments: unit = (token, k-tile, half,
  // thread t, MMA j) -> 8 bytes (x'[c], x'[c+2]), (x'[c+1], x'[c+3]) * 2^P * 4^-j,
  // c = 64 h + 16 t + 4 j.
  auto fold = [&](int ch) {
    uint2* fb = reinterpret_cast<uint2*>(smem + C::kOffF + (ch & 1) * C::kFBytes);
    const int kt_a = ch * C::CHB;
    const int nkt = min(C::CHB, n_kt - kt_a);
    const int units = a.M * nkt * 32;   // 32 four-column units per k-tile
    for (int u = tid; u < units; u += kGThreads) {
      const int tok = u / (nkt * 32);
      const int r = u - tok * (nkt * 32);
      const int ktl = r >> 5;
      const int h = (r >> 4) & 1, tt = (r >> 2) & 3, j = r & 3;
      const int koff = (kt_a + ktl) * kTileCols + 64 * h + 16 * tt + 4 * j;   // column within the slice
      uint2 xv;
      if (staged) {
        xv = *reinterpret_cast<const uint2*>(xs + tok * kspan + koff);
      } else {
        const int k = kbeg + koff;
        const uint16_t* row = a.x + static_cast<size_t>(tok) * a.K;
        uint32_t e[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) e[q] = (k + q < kend) ? static_cast<uint32_t>(row[k + q]) : 0u;
        xv = make_uint2(e[0] | (e[1] << 16), e[2] | (e[3] << 16));
      }
      const float v[4] = {bf16_lo(xv.x), bf16_hi(xv.x), bf16_lo(xv.y), bf16_hi(xv.y)};
      float o[4];
      gfold4(a, v, o);
      const float sc = exp2i(pexp[tok] - 2 * j);
      const uint32_t lo = pack_half2(o[0] * sc, o[2] * sc);
      const uint32_t hi = pack_half2(o[1] * sc, o[3] * sc);
      fb[(((tok >> 3) * C::CHB + ktl) * 8 + h * 4 + j) * 32 + (tok & 7) * 4 + tt] = make_uint2(lo, hi);
    }
  };

  fold(0);
  float acc[2][NT][4];
#pragma unroll
  for (int h = 0; h < 2; ++h)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[h][nt][e] = 0.f;

  // One chunk of kGDepth k-tiles per step; the code registers of k-tile kt are
  // refilled with k-tile kt + kGDepth as soon as they have been used.
  for (int ch = 0; ch * C::CHB < n_kt; ++ch) {
    __syncthreads();                          // fold of chunk ch complete
    if ((ch + 1) * C::CHB < n_kt) fold(ch + 1);   // other buffer; its last readers passed the barrier
    const uint2* fb = reinterpret_cast<const uint2*>(smem + C::kOffF + (ch & 1) * C::kFBytes);
#pragma unroll
    for (int i = 0; i < kGDepth; ++i) {
      const int kt = ch * C::CHB + i;
      if (kt < n_kt) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const uint32_t w = cw[i][2 * h], w8 = cw[i][2 * h + 1];
          const uint32_t ws = w >> 8, ws8 = w8 >> 8;
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const uint32_t m = 0x00030003u << (2 * j);
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
              const uint2 b = fb[((nt * C::CHB + i) * 8 + h * 4 + j) * 32 + lane];
              mma_16816(acc[h][nt], w & m, w8 & m, ws & m, ws8 & m, b.x, b.y);
            }
          }
        }
        load_codes(kt + kGDepth, cw[i]);
      }
    }
  }

  // Partial outputs of this K slice go into the shared memory of the cluster
  // CTA that owns the row: slot [source rank][row - owner base].
  {
    const int rows_per = (kTileRows + KS - 1) / KS;
    const uint32_t red_addr = sbase + C::kOffRed;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int row = r0 + ((e & 2) ? 8 : 0);
        const int tok = nt * 8 + 2 * t + (e & 1);
        if (tok < a.M) {
          const float val = fmaf(acc[0][nt][e] + acc[1][nt][e], exp2i(24 - pexp[tok]), cpart[tok]);
          const int owner = row / rows_per;
          const uint32_t off =
              ((static_cast<uint32_t>(blockIdx.x) * rows_per + (row - owner * rows_per)) * 8 * NT + tok) * 4u;
          if (KS > 1) st_shared_cluster_f32(map_shared_rank(red_addr + off, owner), val);
          else red[off / 4] = val;
        }
      }
  }

  // ---------------- reduction over the K slices of the cluster ----------------
  __syncwarp();
  if (KS > 1) cluster_sync(); else __syncthreads();
  {
    const int rows_per = (kTileRows + KS - 1) / KS;
    const int r0 = static_cast<int>(blockIdx.x) * rows_per;
    const int nrows = max(0, min(kTileRows, r0 + rows_per) - r0);
    for (int idx = tid; idx < nrows * a.M; idx += kGThreads) {
      const int tok = idx / nrows;
      const int rl = idx - tok * nrows;
      const int n = rb * kTileRows + r0 + rl;
      float s = 0.f;
      for (int q = 0; q < KS; ++q) s += red[(q * rows_per + rl) * 8 * NT + tok];
      if (n < a.N) a.y[static_cast<size_t>(tok) * a.N + n] = f32_to_bf16_rn(s);
    }
  }
}

template <int NT>
int gemv_resident_ctas() {
  static int n = 0;
  if (!n) {
    cudaFuncSetAttribute(gemv_kernel<NT>, cudaFuncAttributeMaxDynamicSharedMemorySize, GCfg<NT>::kSmem);
    cudaFuncSetAttribute(gemv_kernel<NT>, cudaFuncAttributePreferredSharedMemoryCarveout,
                         cudaSharedmemCarveoutMaxShared);
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, gemv_kernel<NT>, kGThreads, GCfg<NT>::kSmem) !=
            cudaSuccess ||
        n < 1)
      n = 1;
  }
  return n;
}

template <int NT>
unisvq_status gemv_launch_nt(const unisvq_layer* L, const DecodePlan& p, const void* x, void* y, int M,
                             cudaStream_t s) {
  using C = GCfg<NT>;
  static bool attr_set[64] = {};
  const int dev = L->device;
  if (dev < 0 || dev >= 64) return UNISVQ_ERR_CUDA;
  if (!attr_set[dev]) {
    if (cudaFuncSetAttribute(gemv_kernel<NT>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem) !=
            cudaSuccess ||
        cudaFuncSetAttribute(gemv_kernel<NT>, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared) != cudaSuccess)
      return UNISVQ_ERR_CUDA;
    attr_set[dev] = true;
  }
  GemvArgs a{};
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
  cfg.blockDim = dim3(kGThreads, 1, 1);
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
  return cudaLaunchKernelEx(&cfg, gemv_kernel<NT>, a) == cudaSuccess ? UNISVQ_OK : UNISVQ_ERR_CUDA;
}

}  // namespace

DecodePlan plan_gemv(const unisvq_layer* L, int M) {
  DecodePlan p{};
  p.nt = M <= 8 ? 1 : 2;
  p.nb = L->Np / kTileRows;
  const int occ = p.nt == 1 ? gemv_resident_ctas<1>() : gemv_resident_ctas<2>();
  const int slots = occ * L->num_sms;
  int ks = 1;
  for (int c = 8; c >= 1; --c)
    if (c <= L->KT && p.nb * c <= slots) {
      ks = c;
      break;
    }
  p.kt_per_cta = (L->KT + ks - 1) / ks;
  p.ks = (L->KT + p.kt_per_cta - 1) / p.kt_per_cta;
  p.smem = p.nt == 1 ? GCfg<1>::kSmem : GCfg<2>::kSmem;
  return p;
}

unisvq_status launch_gemv(const unisvq_layer* L, const void* x, void* y, int M, cudaStream_t s) {
  for (int m0 = 0; m0 < M; m0 += kGMaxTok) {
    const int mc = M - m0 < kGMaxTok ? M - m0 : kGMaxTok;
    const DecodePlan p = plan_gemv(L, mc);
    const void* xs = static_cast<const uint16_t*>(x) + static_cast<size_t>(m0) * L->K;
    void* ys = static_cast<uint16_t*>(y) + static_cast<size_t>(m0) * L->N;
    const unisvq_status st = p.nt == 1 ? gemv_launch_nt<1>(L, p, xs, ys, mc, s) : gemv_launch_nt<2>(L, p, xs, ys, mc, s);
    if (st != UNISVQ_OK) return st;
  }
  return UNISVQ_OK;
}

}  // namespace unisvq
