// GEMV for M <= 32 tokens per launch: register-operand tensor-core MMAs.
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
// codes into 8 registers. In MMA (h, j) of a k-tile, lane 4g + t supplies the
// quarter-t words of rows g and g + 8 of half h with s = j, so the MMA covers
// the 16 columns 64h + 16t + 4j + b; the B operand holds the folded
// activations of those columns as fp16 x' * 2^P * 4^-j. Products are
// x' z 2^(P-24); the fp32 sums are rescaled by 2^(24-P) at the end.
//
// CTA = 128 output rows x one K slice, 8 warps: warp w owns unit w (16 rows)
// for every k-tile of the slice. Each lane streams its codes with one 16-byte
// load per k-tile (512 contiguous bytes per warp), kGDepth k-tiles deep, and
// the first loads are issued before the programmatic-launch wait: codes never
// depend on the previous kernel. Warp w also folds tokens w and w + 8 of the
// slice into shared memory by itself (per-token scale from a warp reduction),
// so one block barrier separates the fold from a main loop that has none. The
// K slices of a row block form a thread-block cluster; each CTA adds up the
// partial sums of the rows it owns, which the other CTAs deliver with st.async
// stores counted on an mbarrier.
#include "common.cuh"
#include "mma_sync.cuh"
#include "internal.h"

namespace unisvq {
namespace {

constexpr int kGWarps = 8;
constexpr int kGThreads = kGWarps * 32;
constexpr int kGDepth = 8;          // k-tiles of codes in flight per warp (16 bytes per lane each)
constexpr int kMaxSplit = 8;        // K slices per row block (cluster size)
constexpr int kGMaxTok = 32;
constexpr int kMaxGroup = UNISVQ_MAX_GROUP;   // layers per launch
constexpr int kXLoads = 4;          // 16-byte activation loads in flight per lane (fold)
constexpr int kXPad = 4;            // fp16 elements of padding per token row (bank spread)
constexpr int kTokBytes = 272;      // pexp[32], cpart[32], reduction mbarrier
constexpr size_t kSmemPerSm = 228 * 1024;
constexpr size_t kSmemPerCtaReserved = 1024;

// Kernels are instantiated for DV, the largest vector length of the launch's
// layers: DV = 4 (d in {1, 2, 4}) keeps A in registers and the parameter block
// small; DV = 8 adds the 8 x 8 fold, with A staged in shared memory.
template <int DV>
constexpr size_t static_smem() { return DV == 8 ? 64 * sizeof(float) : 0; }
template <int DV>
constexpr size_t dyn_smem_max() { return kSmemPerSm - kSmemPerCtaReserved - static_smem<DV>(); }

// One layer of a launch. A launch covers one layer, or several layers that
// read the same x (same K): their row blocks are stacked along grid.y.
template <int DV>
struct GemvLayer {
  const uint8_t* codes;
  const uint8_t* hi;   // high-bit plane of 3-bit codes (layout in internal.h), else null
  uint16_t* y;         // bf16 [M][N]
  int N, d;
  int rb0;             // first grid.y row block of this layer
  float colnorm;
  float A[DV * DV];    // row-major d x d (d <= DV)
  float B[DV];
};

template <int DV>
struct GemvArgs {
  const uint16_t* x;   // bf16 [M][K]
  int M, K, KT;
  int kt_per_cta;
  int xstride;         // fp16 elements per token row of the folded slice
  int off_red, off_tok;
  int nlayers;
  int* err;
  GemvLayer<DV> layer[kMaxGroup];
};

// x'[c .. c+3] for the d-vectors inside x[c .. c+3] (c % 4 == 0): row vector x_g A.
// A is a register copy of the kernel parameter (reading the parameter through a
// reference inside a lambda turns every access into a slow generic load).
__device__ __forceinline__ void gfold4(int d, const float (&A)[16], const float (&v)[4], float (&o)[4]) {
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

struct Vec8 {
  float v[8];
};

// x' = x_g A for one vector of d = 8 (A row-major in shared memory). Kept out
// of line: it runs in the fold only and would otherwise crowd the registers
// of the main loop.
__device__ __noinline__ Vec8 fold_vec8(const float* sA8, Vec8 x) {
  Vec8 o;
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    float acc = 0.f;
#pragma unroll
    for (int r = 0; r < 8; ++r) acc = fmaf(x.v[r], sA8[8 * r + c], acc);
    o.v[c] = acc;
  }
  return o;
}

// Columns 8ci .. 8ci+7 of a token's slice (packed bf16 xv) -> their B fragments:
// four-column groups j0 = 2ci mod 4 and j0 + 1, scaled by 2^(pe - 2j). For
// d = 8 the eight columns are one vector and A comes from shared memory (sA8,
// row-major 8 x 8); otherwise from the register copy A.
template <int DV>
__device__ __forceinline__ uint4 fold8(int ci, uint4 xv, int pe, int d, const float (&A)[16], const float* sA8) {
  const int j0 = (2 * ci) & 3;
  const float v0[4] = {bf16_lo(xv.x), bf16_hi(xv.x), bf16_lo(xv.y), bf16_hi(xv.y)};
  const float v1[4] = {bf16_lo(xv.z), bf16_hi(xv.z), bf16_lo(xv.w), bf16_hi(xv.w)};
  float o0[4], o1[4];
  if (DV == 8 && d == 8) {
    const Vec8 o = fold_vec8(sA8, Vec8{{v0[0], v0[1], v0[2], v0[3], v1[0], v1[1], v1[2], v1[3]}});
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      o0[c] = o.v[c];
      o1[c] = o.v[4 + c];
    }
  } else {
    gfold4(d, A, v0, o0);
    gfold4(d, A, v1, o1);
  }
  const float s0 = exp2i(pe - 2 * j0), s1 = exp2i(pe - 2 * j0 - 2);
  return make_uint4(pack_half2(o0[0] * s0, o0[2] * s0), pack_half2(o0[1] * s0, o0[3] * s0),
                    pack_half2(o1[0] * s1, o1[2] * s1), pack_half2(o1[1] * s1, o1[3] * s1));
}

// Bit j of x -> bit 2j (x < 2^16).
__device__ __forceinline__ uint32_t spread16(uint32_t x) {
  x = (x | (x << 8)) & 0x00FF00FFu;
  x = (x | (x << 4)) & 0x0F0F0F0Fu;
  x = (x | (x << 2)) & 0x33333333u;
  return (x | (x << 1)) & 0x55555555u;
}

// BITS = 3: codes z = z_lo + 4 z_hi; z_lo from the packed words as for 2-bit
// codes, z_hi from the layer's bit plane, spread so that the high bit of the
// code at bits [8b + 2s + 1 : 8b + 2s] lands on bit 8b + 2s + 2: the A
// registers become (w & m) | (h & m') = z 4^s 2^-24, z <= 7, the same
// subnormal scale as 2-bit codes, so the B fragments do not change.
template <int NT, int DV, int BITS>
__global__ void __launch_bounds__(kGThreads, 2) gemv_kernel(const __grid_constant__ GemvArgs<DV> a) {
  extern __shared__ __align__(16) uint8_t smem[];
  const uint32_t sbase = smem_u32(smem);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int KS = gridDim.x;
  const int kt0 = blockIdx.x * a.kt_per_cta;
  const int n_kt = min(a.kt_per_cta, a.KT - kt0);
  const int M = a.M;
  // This CTA's layer, read with constant parameter offsets only.
  int li = 0;
#pragma unroll
  for (int i = 1; i < kMaxGroup; ++i)
    if (i < a.nlayers && static_cast<int>(blockIdx.y) >= a.layer[i].rb0) li = i;
  const uint8_t* codes = nullptr;
  const uint8_t* hiplane = nullptr;
  uint16_t* yout = nullptr;
  int N = 0, d = 1, rb = 0;
  float colnorm = 0.f, Areg[16], Bq[DV];
#pragma unroll
  for (int i = 0; i < kMaxGroup; ++i) {
    if (i == li) {
      codes = a.layer[i].codes;
      if constexpr (BITS == 3) hiplane = a.layer[i].hi;
      yout = a.layer[i].y;
      N = a.layer[i].N;
      d = a.layer[i].d;
      rb = static_cast<int>(blockIdx.y) - a.layer[i].rb0;
      colnorm = a.layer[i].colnorm;
#pragma unroll
      for (int e = 0; e < 16; ++e) Areg[e] = a.layer[i].A[e];
#pragma unroll
      for (int e = 0; e < DV; ++e) Bq[e] = a.layer[i].B[e];
    }
  }
  float Bcol[8];   // B[e mod d] for column e of an 8-column chunk
#pragma unroll
  for (int e = 0; e < 8; ++e) Bcol[e] = d == 1 ? Bq[0] : (d == 2 ? Bq[e & 1] : (DV == 4 || d == 4 ? Bq[e & 3] : Bq[e & (DV - 1)]));
  __shared__ float sA8[DV == 8 ? 64 : 1];   // A for d = 8 (the fold reads it from here)
  if constexpr (DV == 8) {
    if (d == 8) {
      if (tid < 64) {
        float v = a.layer[0].A[tid];
#pragma unroll
        for (int i = 1; i < kMaxGroup; ++i)
          if (i == li) v = a.layer[i].A[tid];
        sA8[tid] = v;
      }
      __syncthreads();
    }
  }
  // Rows whose K-slice partial sums this CTA adds up (it "owns" them).
  const int rows_per = (kTileRows + KS - 1) / KS;
  const int own0 = static_cast<int>(blockIdx.x) * rows_per;
  const int nown = max(0, min(kTileRows, own0 + rows_per) - own0);

  int* pexp = reinterpret_cast<int*>(smem + a.off_tok);
  float* cpart = reinterpret_cast<float*>(smem + a.off_tok + 128);
  float* red = reinterpret_cast<float*>(smem + a.off_red);
  const uint32_t red_bar = sbase + a.off_tok + 256;

  // Reduction barrier: one arrival here plus the bytes the other CTAs of the
  // cluster store into this CTA's slots (st.async counts them).
  if (KS > 1) {
    if (tid == 0) {
      mbar_init(red_bar, 1);
      fence_mbar_init();
      mbar_arrive_expect_tx(red_bar, static_cast<uint32_t>((KS - 1) * nown * M * 4));
    }
    cluster_arrive_relaxed();
  }
  // A valid plan gives every CTA at least one k-tile; otherwise flag the error
  // and fall through with empty loops so that every partial is still sent.
  if (n_kt <= 0 && tid == 0) record_error(a.err, kErrBadLaunch);

  // ---- codes: unit `warp` (rows 16 warp .. +15) of every k-tile of the slice ----
  const int g = lane >> 2, t = lane & 3;
  const uint8_t* cbase =
      codes + (static_cast<size_t>(rb) * a.KT + kt0) * kTileBytes + warp * kUnitBytes + lane * 16;
  uint4 cw[kGDepth];
#pragma unroll
  for (int s = 0; s < kGDepth; ++s)
    if (s < n_kt) cw[s] = ldg_stream_v4(cbase + static_cast<size_t>(s) * kTileBytes);
  constexpr int kHiDepth = BITS == 3 ? kGDepth : 1;
  uint2 hw[kHiDepth];   // high bits of the four words of cw (halfword per word)
  const uint8_t* hbase = nullptr;
  if constexpr (BITS == 3) {
    hbase = hiplane + (static_cast<size_t>(rb) * a.KT + kt0) * (kTileBytes / 2) + warp * (kUnitBytes / 2) + lane * 8;
#pragma unroll
    for (int s = 0; s < kGDepth; ++s)
      if (s < n_kt) hw[s] = ldg_v2(hbase + static_cast<size_t>(s) * (kTileBytes / 2));
  }
  pdl_launch_dependents();

  pdl_wait();   // x may be the previous kernel's output

  // ---- fold: warp w prepares tokens w and w + 8 on its own (no block barrier) ----
  // Pass A stages the slice and finds max |x| and sum_k x[k] B[k mod d]; 2^P puts
  // the largest possible |x'| (<= max|x| * colnorm) below 2^15 (fp16). Pass B
  // folds in place: columns c .. c+3 (c = 16t' + 4j inside a 64-column half)
  // become the B fragment (x'[c], x'[c+2]), (x'[c+1], x'[c+3]) * 2^P * 4^-j.
  const int kbeg = kt0 * kTileCols;
  const int kend = min(a.K, (kt0 + n_kt) * kTileCols);
  const int nch = n_kt * (kTileCols / 8);   // 8-column chunks of the slice
  const bool vec8 = (a.K & 7) == 0;
  const uint32_t xrow_bytes = static_cast<uint32_t>(a.xstride) * 2u;
  if (nch <= 32 * kXLoads) {
    // Whole slice in registers: the loads of both of this warp's tokens go
    // out together, then each token is reduced, folded and stored.
    constexpr int kPair = NT < 2 ? NT : 2;   // tokens whose loads are in flight together
#pragma unroll 1
    for (int p0 = 0; p0 < NT; p0 += kPair) {
    uint4 u[kPair][kXLoads];
#pragma unroll
    for (int p = 0; p < kPair; ++p) {
      const int tk = warp + kGWarps * (p0 + p);
#pragma unroll
      for (int j = 0; j < kXLoads; ++j) {
        const int ci = lane + 32 * j;
        u[p][j] = (tk < M && ci < nch) ? load_x8(a.x + static_cast<size_t>(tk) * a.K, kbeg + 8 * ci, kend, vec8)
                                       : make_uint4(0, 0, 0, 0);
      }
    }
#pragma unroll
    for (int p = 0; p < kPair; ++p) {
      const int tk = warp + kGWarps * (p0 + p);
      if (tk < M) {
        float mx = 0.f, cs = 0.f;
#pragma unroll
        for (int j = 0; j < kXLoads; ++j) {
          const uint32_t w4[4] = {u[p][j].x, u[p][j].y, u[p][j].z, u[p][j].w};
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const float v0 = bf16_lo(w4[q]), v1 = bf16_hi(w4[q]);
            mx = fmaxf(mx, fmaxf(fabsf(v0), fabsf(v1)));
            cs = fmaf(v0, Bcol[2 * q], cs);
            cs = fmaf(v1, Bcol[2 * q + 1], cs);
          }
        }
#pragma unroll
        for (int off = 16; off; off >>= 1) {
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
          cs += __shfl_xor_sync(0xffffffffu, cs, off);
        }
        const int pe = token_scale_exp(mx * colnorm);
        if (lane == 0) {
          pexp[tk] = pe;
          cpart[tk] = cs;
        }
        uint8_t* xrow = smem + tk * xrow_bytes;
        uint4 f[kXLoads];
#pragma unroll
        for (int j = 0; j < kXLoads; ++j) f[j] = fold8<DV>(lane + 32 * j, u[p][j], pe, d, Areg, sA8);
#pragma unroll
        for (int j = 0; j < kXLoads; ++j) {
          const int ci = lane + 32 * j;
          if (ci < nch) {
            *reinterpret_cast<uint2*>(xrow + 16u * ci) = make_uint2(f[j].x, f[j].y);
            *reinterpret_cast<uint2*>(xrow + 16u * ci + 8) = make_uint2(f[j].z, f[j].w);
          }
        }
      }
    }
    }
  } else {
    for (int tk = warp; tk < M; tk += kGWarps) {
      const uint16_t* row = a.x + static_cast<size_t>(tk) * a.K;
      uint8_t* xrow = smem + tk * xrow_bytes;
      float mx = 0.f, cs = 0.f;
      uint4 u[kXLoads];
      // pass A: stage the chunks, max and c-sum
      for (int c0 = lane; c0 < nch; c0 += 32 * kXLoads) {
#pragma unroll
        for (int j = 0; j < kXLoads; ++j) {
          const int ci = c0 + 32 * j;
          u[j] = ci < nch ? load_x8(row, kbeg + 8 * ci, kend, vec8) : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int j = 0; j < kXLoads; ++j) {
          const int ci = c0 + 32 * j;
          if (ci < nch) {
            *reinterpret_cast<uint2*>(xrow + 16u * ci) = make_uint2(u[j].x, u[j].y);
            *reinterpret_cast<uint2*>(xrow + 16u * ci + 8) = make_uint2(u[j].z, u[j].w);
            const uint32_t w4[4] = {u[j].x, u[j].y, u[j].z, u[j].w};
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const float v0 = bf16_lo(w4[q]), v1 = bf16_hi(w4[q]);
              mx = fmaxf(mx, fmaxf(fabsf(v0), fabsf(v1)));
              cs = fmaf(v0, Bcol[2 * q], cs);
              cs = fmaf(v1, Bcol[2 * q + 1], cs);
            }
          }
        }
      }
#pragma unroll
      for (int off = 16; off; off >>= 1) {
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
        cs += __shfl_xor_sync(0xffffffffu, cs, off);
      }
      const int pe = token_scale_exp(mx * colnorm);
      if (lane == 0) {
        pexp[tk] = pe;
        cpart[tk] = cs;
      }
      // pass B: every lane re-reads only the chunks it staged itself
      for (int c0 = lane; c0 < nch; c0 += 32 * kXLoads) {
#pragma unroll
        for (int j = 0; j < kXLoads; ++j) {
          const int ci = c0 + 32 * j;
          if (ci < nch) {
            const uint2 lo = *reinterpret_cast<const uint2*>(xrow + 16u * ci);
            const uint2 hi = *reinterpret_cast<const uint2*>(xrow + 16u * ci + 8);
            u[j] = fold8<DV>(ci, make_uint4(lo.x, lo.y, hi.x, hi.y), pe, d, Areg, sA8);
          }
        }
#pragma unroll
        for (int j = 0; j < kXLoads; ++j) {
          const int ci = c0 + 32 * j;
          if (ci < nch) {
            *reinterpret_cast<uint2*>(xrow + 16u * ci) = make_uint2(u[j].x, u[j].y);
            *reinterpret_cast<uint2*>(xrow + 16u * ci + 8) = make_uint2(u[j].z, u[j].w);
          }
        }
      }
    }
  }
  __syncthreads();

  // ---- main loop: no block-wide barrier ----
  float acc[NT][4];   // both halves of a k-tile accumulate into one chain per token octet
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
#pragma unroll
    for (int e = 0; e < 4; ++e) acc[nt][e] = 0.f;
  bool act[NT];
  const uint8_t* xl[NT];   // this lane's B fragments: token 8nt + g, quarter t
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    const int tk = 8 * nt + g;
    act[nt] = tk < M;
    xl[nt] = smem + (act[nt] ? tk : 0) * xrow_bytes + 32u * t;
  }
  for (int i0 = 0; i0 < n_kt; i0 += kGDepth) {
#pragma unroll
    for (int s = 0; s < kGDepth; ++s) {
      const int i = i0 + s;
      if (i < n_kt) {
        const uint32_t koff = 256u * i;   // 256 bytes of B fragments per k-tile
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const uint32_t wa = h ? cw[s].z : cw[s].x, wb = h ? cw[s].w : cw[s].y;   // rows g, g + 8
          const uint32_t was = wa >> 8, wbs = wb >> 8;
          uint32_t ha = 0, hb = 0, has = 0, hbs = 0;
          if constexpr (BITS == 3) {
            const uint32_t hwd = h ? hw[s].y : hw[s].x;   // words 2h (row g) and 2h + 1 (row g + 8)
            const uint32_t sa = spread16(hwd & 0xFFFFu), sb = spread16(hwd >> 16);
            ha = sa << 2;   // bytes 0 and 2 (bit 32 of byte 3 falls off; a0, a1 do not use it)
            hb = sb << 2;
            has = sa >> 6;  // bytes 1 and 3, moved down one byte as w >> 8
            hbs = sb >> 6;
          }
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const uint32_t m = 0x00030003u << (2 * j);
            uint32_t a0 = wa & m, a1 = wb & m, a2 = was & m, a3 = wbs & m;
            if constexpr (BITS == 3) {
              const uint32_t mh = 0x00040004u << (2 * j);
              a0 |= ha & mh;
              a1 |= hb & mh;
              a2 |= has & mh;
              a3 |= hbs & mh;
            }
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
              const uint2 b = act[nt] ? *reinterpret_cast<const uint2*>(xl[nt] + koff + 128u * h + 8u * j)
                                      : make_uint2(0u, 0u);
              mma_16816(acc[nt], a0, a1, a2, a3, b);
            }
          }
        }
        if (i + kGDepth < n_kt) {
          cw[s] = ldg_stream_v4(cbase + static_cast<size_t>(i + kGDepth) * kTileBytes);
          if constexpr (BITS == 3) hw[s] = ldg_v2(hbase + static_cast<size_t>(i + kGDepth) * (kTileBytes / 2));
        }
      }
    }
  }

  // ---- partial sums -> owner CTA of the row: slot [rank][row - owner base][token] ----
  // Remote slots are written with st.async, which counts their bytes on the
  // owner's mbarrier; the owner waits for exactly that many bytes, so no
  // cluster-wide barrier is needed and no CTA's shared memory is written
  // after it has stopped waiting.
  constexpr int MP = 8 * NT;
  const uint32_t red_addr = sbase + a.off_red;
  if (KS > 1) cluster_wait();   // every CTA of the cluster has initialised its barrier
  float pv[NT][2][2];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    const int tok = 8 * nt + 2 * t;   // this lane holds tokens tok and tok + 1
    const float sc0 = tok < M ? exp2i(24 - pexp[tok]) : 0.f, c0v = tok < M ? cpart[tok] : 0.f;
    const float sc1 = tok + 1 < M ? exp2i(24 - pexp[tok + 1]) : 0.f, c1v = tok + 1 < M ? cpart[tok + 1] : 0.f;
#pragma unroll
    for (int rh = 0; rh < 2; ++rh) {
      pv[nt][rh][0] = fmaf(acc[nt][2 * rh], sc0, c0v);
      pv[nt][rh][1] = fmaf(acc[nt][2 * rh + 1], sc1, c1v);
    }
  }
#pragma unroll
  for (int rh = 0; rh < 2; ++rh) {
    const int row = 16 * warp + g + 8 * rh;
    const int owner = row / rows_per;
    const uint32_t row_off = (static_cast<uint32_t>(blockIdx.x) * rows_per + (row - owner * rows_per)) * MP;
    const bool local = owner == static_cast<int>(blockIdx.x);
    const uint32_t rbar = local ? 0u : map_shared_rank(red_bar, owner);
    const uint32_t rslot = local ? 0u : map_shared_rank(red_addr + row_off * 4u, owner);
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const int tok = 8 * nt + 2 * t;
      if (tok < M) {
        if (local) {
          red[row_off + tok] = pv[nt][rh][0];
          if (tok + 1 < M) red[row_off + tok + 1] = pv[nt][rh][1];
        } else if (tok + 1 < M) {
          st_async_v2f32(rslot + tok * 4u, pv[nt][rh][0], pv[nt][rh][1], rbar);
        } else {
          st_async_f32(rslot + tok * 4u, pv[nt][rh][0], rbar);
        }
      }
    }
  }

  // ---- reduction over the K slices of the row block ----
  __syncthreads();   // this CTA's own slots
  if (KS > 1 && nown > 0 && !mbar_wait_cluster(red_bar, 0, a.err, kErrTimeoutReduce)) return;
  for (int idx = tid; idx < nown * M; idx += kGThreads) {
    const int tok = idx / nown;
    const int rl = idx - tok * nown;
    const int n = rb * kTileRows + own0 + rl;
    float v[kMaxSplit];
#pragma unroll
    for (int q = 0; q < kMaxSplit; ++q) v[q] = q < KS ? red[(q * rows_per + rl) * MP + tok] : 0.f;
    float sum = 0.f;
#pragma unroll
    for (int q = 0; q < kMaxSplit; ++q) sum += v[q];
    if (n < N) yout[static_cast<size_t>(tok) * N + n] = f32_to_bf16_rn(sum);
  }
}

// ---------------------------------------------------------------------------
// Row-slice GEMV for M <= kRMaxTok: CTA = 32 rows (units 2c and 2c+1 of the
// layer) x the whole K, so no K-slice partial sums leave the CTA. Warp w owns
// the contiguous k-tiles [w kpw, (w+1) kpw) of both units and folds exactly
// those columns into its own shared-memory region with its own per-token
// scale: no block barrier precedes its MMAs. The eight partial sums per
// output are added in shared memory at the end. Each CTA folds all of x
// (M x K), which is cheap next to the codes for a few tokens.
// ---------------------------------------------------------------------------
constexpr int kRMaxTok = 4;
constexpr int kRDepth = 4;    // k-tiles of codes in flight per warp (2 x 16 bytes per lane each)
constexpr int kRItems = 4;    // activation loads in flight per lane in the fold

template <int DV>
__global__ void __launch_bounds__(kGThreads, 2) gemv_rows_kernel(const __grid_constant__ GemvArgs<DV> a) {
  extern __shared__ __align__(16) uint8_t smem[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int M = a.M;
  int li = 0;
#pragma unroll
  for (int i = 1; i < kMaxGroup; ++i)
    if (i < a.nlayers && static_cast<int>(blockIdx.x) >= a.layer[i].rb0) li = i;
  const uint8_t* codes = nullptr;
  uint16_t* yout = nullptr;
  int N = 0, d = 1, pr = 0;
  float colnorm = 0.f, Areg[16], Bq[DV];
#pragma unroll
  for (int i = 0; i < kMaxGroup; ++i) {
    if (i == li) {
      codes = a.layer[i].codes;
      yout = a.layer[i].y;
      N = a.layer[i].N;
      d = a.layer[i].d;
      pr = static_cast<int>(blockIdx.x) - a.layer[i].rb0;   // pair of units within the layer
      colnorm = a.layer[i].colnorm;
#pragma unroll
      for (int e = 0; e < 16; ++e) Areg[e] = a.layer[i].A[e];
#pragma unroll
      for (int e = 0; e < DV; ++e) Bq[e] = a.layer[i].B[e];
    }
  }
  float Bcol[8];   // B[e mod d] for column e of an 8-column chunk
#pragma unroll
  for (int e = 0; e < 8; ++e) Bcol[e] = d == 1 ? Bq[0] : (d == 2 ? Bq[e & 1] : (DV == 4 || d == 4 ? Bq[e & 3] : Bq[e & (DV - 1)]));
  __shared__ float sA8[DV == 8 ? 64 : 1];   // A for d = 8 (the fold reads it from here)
  if constexpr (DV == 8) {
    if (d == 8) {
      if (threadIdx.x < 64) {
        float v = a.layer[0].A[threadIdx.x];
#pragma unroll
        for (int i = 1; i < kMaxGroup; ++i)
          if (i == li) v = a.layer[i].A[threadIdx.x];
        sA8[threadIdx.x] = v;
      }
      __syncthreads();
    }
  }

  const int kpw = a.kt_per_cta;
  const int kw0 = warp * kpw;
  const int nkw = max(0, min(kpw, a.KT - kw0));
  const uint32_t wstride = static_cast<uint32_t>(a.xstride) * 2u;   // bytes per token row of a warp region
  uint8_t* wreg = smem + warp * M * wstride;
  float* red = reinterpret_cast<float*>(smem + a.off_red);         // [warp][32 rows][8 tokens]

  // ---- codes: units 2 pr and 2 pr + 1 (512 contiguous bytes each per k-tile) ----
  const int g = lane >> 2, t = lane & 3;
  const int u0 = 2 * pr;
  const uint8_t* cbase = codes + (static_cast<size_t>(u0 >> 3) * a.KT + kw0) * kTileBytes + (u0 & 7) * kUnitBytes +
                         lane * 16;
  uint4 cw[kRDepth][2];
#pragma unroll
  for (int s = 0; s < kRDepth; ++s)
    if (s < nkw) {
      cw[s][0] = ldg_stream_v4(cbase + static_cast<size_t>(s) * kTileBytes);
      cw[s][1] = ldg_stream_v4(cbase + static_cast<size_t>(s) * kTileBytes + kUnitBytes);
    }
  pdl_launch_dependents();

  pdl_wait();   // x may be the previous kernel's output

  // ---- fold of this warp's columns for every token (private, no block barrier) ----
  const int kbeg = kw0 * kTileCols;
  const int kend = min(a.K, (kw0 + nkw) * kTileCols);
  const int ncw = nkw * (kTileCols / 8);          // chunks per token
  const int jt = (ncw + 31) / 32;                 // loads per lane per token
  const int items = M * jt;
  const bool vec8 = (a.K & 7) == 0;
  float mx[kRMaxTok], cs[kRMaxTok];
#pragma unroll
  for (int q = 0; q < kRMaxTok; ++q) mx[q] = cs[q] = 0.f;
  for (int b0 = 0; b0 < items; b0 += kRItems) {
    uint4 u[kRItems];
#pragma unroll
    for (int r = 0; r < kRItems; ++r) {
      const int it = b0 + r;
      const int tk = it / jt, ci = lane + 32 * (it - tk * jt);
      u[r] = (it < items && ci < ncw)
                 ? load_x8(a.x + static_cast<size_t>(tk) * a.K, kbeg + 8 * ci, kend, vec8)
                 : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int r = 0; r < kRItems; ++r) {
      const int it = b0 + r;
      const int tk = it / jt, ci = lane + 32 * (it - tk * jt);
      if (it < items && ci < ncw) {
        uint8_t* dst = wreg + tk * wstride + 16u * ci;
        *reinterpret_cast<uint2*>(dst) = make_uint2(u[r].x, u[r].y);
        *reinterpret_cast<uint2*>(dst + 8) = make_uint2(u[r].z, u[r].w);
      }
      float m8 = 0.f, c8 = 0.f;
      const uint32_t w4[4] = {u[r].x, u[r].y, u[r].z, u[r].w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float v0 = bf16_lo(w4[q]), v1 = bf16_hi(w4[q]);
        m8 = fmaxf(m8, fmaxf(fabsf(v0), fabsf(v1)));
        c8 = fmaf(v0, Bcol[2 * q], c8);
        c8 = fmaf(v1, Bcol[2 * q + 1], c8);
      }
#pragma unroll
      for (int q = 0; q < kRMaxTok; ++q)
        if (q == tk) {
          mx[q] = fmaxf(mx[q], m8);
          cs[q] += c8;
        }
    }
  }
  int pe[kRMaxTok];
#pragma unroll
  for (int q = 0; q < kRMaxTok; ++q) {
#pragma unroll
    for (int off = 16; off; off >>= 1) {
      mx[q] = fmaxf(mx[q], __shfl_xor_sync(0xffffffffu, mx[q], off));
      cs[q] += __shfl_xor_sync(0xffffffffu, cs[q], off);
    }
    pe[q] = token_scale_exp(mx[q] * colnorm);
  }
  for (int b0 = 0; b0 < items; b0 += kRItems) {
    uint4 f[kRItems];
#pragma unroll
    for (int r = 0; r < kRItems; ++r) {
      const int it = b0 + r;
      const int tk = it / jt, ci = lane + 32 * (it - tk * jt);
      if (it < items && ci < ncw) {
        int pt = 0;
#pragma unroll
        for (int q = 0; q < kRMaxTok; ++q)
          if (q == tk) pt = pe[q];
        const uint8_t* src = wreg + tk * wstride + 16u * ci;
        const uint2 lo = *reinterpret_cast<const uint2*>(src), hi = *reinterpret_cast<const uint2*>(src + 8);
        f[r] = fold8<DV>(ci, make_uint4(lo.x, lo.y, hi.x, hi.y), pt, d, Areg, sA8);
      }
    }
#pragma unroll
    for (int r = 0; r < kRItems; ++r) {
      const int it = b0 + r;
      const int tk = it / jt, ci = lane + 32 * (it - tk * jt);
      if (it < items && ci < ncw) {
        uint8_t* dst = wreg + tk * wstride + 16u * ci;
        *reinterpret_cast<uint2*>(dst) = make_uint2(f[r].x, f[r].y);
        *reinterpret_cast<uint2*>(dst + 8) = make_uint2(f[r].z, f[r].w);
      }
    }
  }
  __syncwarp();

  // ---- main loop over this warp's k-tiles ----
  float acc[2][4];
#pragma unroll
  for (int u = 0; u < 2; ++u)
#pragma unroll
    for (int e = 0; e < 4; ++e) acc[u][e] = 0.f;
  const bool act = g < M;
  const uint8_t* xl = wreg + (act ? g : 0) * wstride + 32u * t;
  for (int i0 = 0; i0 < nkw; i0 += kRDepth) {
#pragma unroll
    for (int s = 0; s < kRDepth; ++s) {
      const int i = i0 + s;
      if (i < nkw) {
        const uint32_t koff = 256u * i;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const uint32_t a0 = h ? cw[s][0].z : cw[s][0].x, a1 = h ? cw[s][0].w : cw[s][0].y;
          const uint32_t b0 = h ? cw[s][1].z : cw[s][1].x, b1 = h ? cw[s][1].w : cw[s][1].y;
          const uint32_t a0s = a0 >> 8, a1s = a1 >> 8, b0s = b0 >> 8, b1s = b1 >> 8;
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const uint32_t m = 0x00030003u << (2 * j);
            const uint2 bf = act ? *reinterpret_cast<const uint2*>(xl + koff + 128u * h + 8u * j) : make_uint2(0u, 0u);
            mma_16816(acc[0], a0 & m, a1 & m, a0s & m, a1s & m, bf);
            mma_16816(acc[1], b0 & m, b1 & m, b0s & m, b1s & m, bf);
          }
        }
        if (i + kRDepth < nkw) {
          cw[s][0] = ldg_stream_v4(cbase + static_cast<size_t>(i + kRDepth) * kTileBytes);
          cw[s][1] = ldg_stream_v4(cbase + static_cast<size_t>(i + kRDepth) * kTileBytes + kUnitBytes);
        }
      }
    }
  }

  // ---- partial sums of this warp -> red[warp][row][token], then add the 8 warps ----
  float sc[2], cv[2];
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    const int tok = 2 * t + e;
    sc[e] = 0.f;
    cv[e] = 0.f;
#pragma unroll
    for (int q = 0; q < kRMaxTok; ++q)
      if (q == tok) {
        sc[e] = exp2i(24 - pe[q]);
        cv[e] = cs[q];
      }
  }
#pragma unroll
  for (int u = 0; u < 2; ++u)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int row = 16 * u + g + ((e & 2) ? 8 : 0);
      const int tok = 2 * t + (e & 1);
      if (tok < M) red[(warp * 32 + row) * 8 + tok] = fmaf(acc[u][e], sc[e & 1], cv[e & 1]);
    }
  __syncthreads();
  for (int idx = tid; idx < 32 * M; idx += kGThreads) {
    const int tok = idx >> 5, row = idx & 31;
    float v[kGWarps];
#pragma unroll
    for (int w = 0; w < kGWarps; ++w) v[w] = red[(w * 32 + row) * 8 + tok];
    float sum = 0.f;
#pragma unroll
    for (int w = 0; w < kGWarps; ++w) sum += v[w];
    const int n = 16 * u0 + row;
    if (n < N) yout[static_cast<size_t>(tok) * N + n] = f32_to_bf16_rn(sum);
  }
}

struct GemvShape {
  size_t smem;
  int off_red, off_tok, xstride;
};

GemvShape gemv_shape(int M, int kt_per_cta, int ks, int nt) {
  GemvShape s{};
  s.xstride = kt_per_cta * kTileCols + kXPad;
  const size_t xf = static_cast<size_t>(M) * s.xstride * 2;
  const int rows_per = (kTileRows + ks - 1) / ks;
  const size_t red = static_cast<size_t>(ks) * rows_per * 8 * nt * 4;
  s.off_red = static_cast<int>((xf + 15) / 16 * 16);
  s.off_tok = static_cast<int>(s.off_red + red);
  s.smem = static_cast<size_t>(s.off_tok) + kTokBytes;
  return s;
}

// Copies a layer's affine map into a launch's parameter block.
template <int DV>
void set_affine(GemvLayer<DV>& g, const unisvq_layer* L) {
  for (int e = 0; e < DV * DV; ++e) g.A[e] = L->A[e];
  for (int e = 0; e < DV; ++e) g.B[e] = L->B[e];
}

// 8 if any layer of the launch has d = 8, else 4.
int group_dv(const unisvq_layer* const* Ls, int n) {
  for (int i = 0; i < n; ++i)
    if (Ls[i]->d == 8) return 8;
  return 4;
}

template <int NT, int DV, int BITS>
unisvq_status gemv_launch_nt(const unisvq_layer* const* Ls, int n, const DecodePlan& p, const void* x,
                             void* const* ys, int m0, int M, cudaStream_t s) {
  static bool attr_set[64] = {};
  const int dev = Ls[0]->device;
  if (dev < 0 || dev >= 64) return UNISVQ_ERR_CUDA;
  if (!attr_set[dev]) {
    if (cudaFuncSetAttribute(gemv_kernel<NT, DV, BITS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(dyn_smem_max<DV>())) != cudaSuccess ||
        cudaFuncSetAttribute(gemv_kernel<NT, DV, BITS>, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared) != cudaSuccess)
      return UNISVQ_ERR_CUDA;
    attr_set[dev] = true;
  }
  const GemvShape sh = gemv_shape(M, p.kt_per_cta, p.ks, NT);
  GemvArgs<DV> a{};
  a.x = static_cast<const uint16_t*>(x) + static_cast<size_t>(m0) * Ls[0]->K;
  a.M = M;
  a.K = Ls[0]->K;
  a.KT = Ls[0]->KT;
  a.kt_per_cta = p.kt_per_cta;
  a.xstride = sh.xstride;
  a.off_red = sh.off_red;
  a.off_tok = sh.off_tok;
  a.nlayers = n;
  a.err = device_error_word();
  int rb0 = 0;
  for (int i = 0; i < n; ++i) {
    const unisvq_layer* L = Ls[i];
    GemvLayer<DV>& g = a.layer[i];
    g.codes = L->codes;
    g.hi = L->hi;
    g.y = static_cast<uint16_t*>(ys[i]) + static_cast<size_t>(m0) * L->N;
    g.N = L->N;
    g.d = L->d;
    g.rb0 = rb0;
    g.colnorm = L->colnorm;
    set_affine(g, L);
    rb0 += L->Np / kTileRows;
  }

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.ks, p.nb, 1);
  cfg.blockDim = dim3(kGThreads, 1, 1);
  cfg.dynamicSmemBytes = sh.smem;
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
  return cudaLaunchKernelEx(&cfg, gemv_kernel<NT, DV, BITS>, a) == cudaSuccess ? UNISVQ_OK : UNISVQ_ERR_CUDA;
}

// Split K into ks <= 8 cluster CTAs for nb row blocks: the largest ks whose
// grid fits one wave of resident CTAs (two per SM); if none does, the
// smallest ks whose folded slice fits in shared memory. `sstat` is the
// kernel's static shared memory (static_smem<DV>()).
DecodePlan plan_rows(int nb, int KT, int num_sms, int M, size_t sstat) {
  DecodePlan p{};
  p.nt = M <= 8 ? 1 : (M <= 16 ? 2 : 4);
  p.nb = nb;
  const size_t cap = kSmemPerSm - kSmemPerCtaReserved - sstat;
  int best = 0, fallback = 0;
  for (int c = kMaxSplit; c >= 1; --c) {
    if (c > KT) continue;
    const int kpc = (KT + c - 1) / c;
    const int ks = (KT + kpc - 1) / kpc;
    if (ks != c) continue;
    const size_t smem = gemv_shape(M, kpc, ks, p.nt).smem;
    if (smem > cap) continue;
    fallback = ks;
    const int per_sm = static_cast<int>(kSmemPerSm / (smem + sstat + kSmemPerCtaReserved)) < 2 ? 1 : 2;
    if (!best && nb * ks <= per_sm * num_sms) best = ks;
  }
  const int ks = best ? best : (fallback ? fallback : kMaxSplit);
  p.kt_per_cta = (KT + ks - 1) / ks;
  p.ks = (KT + p.kt_per_cta - 1) / p.kt_per_cta;
  p.smem = gemv_shape(M, p.kt_per_cta, p.ks, p.nt).smem;
  return p;
}

// Row-slice kernel: k-tiles per warp, shared memory and launch.
int rows_kpw(int KT) { return (KT + kGWarps - 1) / kGWarps; }

size_t rows_smem(int M, int KT, int* off_red, int* xstride) {
  const int kpw = rows_kpw(KT);
  const int xs = kpw * kTileCols + kXPad;
  const size_t fold = static_cast<size_t>(kGWarps) * M * xs * 2;
  const size_t offr = (fold + 15) / 16 * 16;
  if (off_red) *off_red = static_cast<int>(offr);
  if (xstride) *xstride = xs;
  return offr + static_cast<size_t>(kGWarps) * 32 * 8 * 4;
}

template <int DV>
unisvq_status rows_launch(const unisvq_layer* const* Ls, int n, const void* x, void* const* ys, int m0, int M,
                          cudaStream_t s) {
  static bool attr_set[64] = {};
  const int dev = Ls[0]->device;
  if (dev < 0 || dev >= 64) return UNISVQ_ERR_CUDA;
  if (!attr_set[dev]) {
    if (cudaFuncSetAttribute(gemv_rows_kernel<DV>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(dyn_smem_max<DV>())) != cudaSuccess ||
        cudaFuncSetAttribute(gemv_rows_kernel<DV>, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared) != cudaSuccess)
      return UNISVQ_ERR_CUDA;
    attr_set[dev] = true;
  }
  GemvArgs<DV> a{};
  int off_red = 0, xstride = 0;
  const size_t smem = rows_smem(M, Ls[0]->KT, &off_red, &xstride);
  a.x = static_cast<const uint16_t*>(x) + static_cast<size_t>(m0) * Ls[0]->K;
  a.M = M;
  a.K = Ls[0]->K;
  a.KT = Ls[0]->KT;
  a.kt_per_cta = rows_kpw(Ls[0]->KT);
  a.xstride = xstride;
  a.off_red = off_red;
  a.nlayers = n;
  a.err = device_error_word();
  int pairs = 0;
  for (int i = 0; i < n; ++i) {
    const unisvq_layer* L = Ls[i];
    GemvLayer<DV>& g = a.layer[i];
    g.codes = L->codes;
    g.y = static_cast<uint16_t*>(ys[i]) + static_cast<size_t>(m0) * L->N;
    g.N = L->N;
    g.d = L->d;
    g.rb0 = pairs;
    g.colnorm = L->colnorm;
    set_affine(g, L);
    pairs += L->Np / (2 * kUnitRows);
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(pairs, 1, 1);
  cfg.blockDim = dim3(kGThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr.val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, gemv_rows_kernel<DV>, a) == cudaSuccess ? UNISVQ_OK : UNISVQ_ERR_CUDA;
}

}  // namespace

DecodePlan plan_gemv(const unisvq_layer* L, int M) {
  return plan_rows(L->Np / kTileRows, L->KT, L->num_sms, M, L->d == 8 ? static_smem<8>() : static_smem<4>());
}

unisvq_status launch_gemv_group(const unisvq_layer* const* Ls, int n, const void* x, void* const* ys, int M,
                                cudaStream_t s) {
  if (n < 1 || n > kMaxGroup) return UNISVQ_ERR_INVALID_ARG;
  int nb = 0;
  for (int i = 0; i < n; ++i) nb += Ls[i]->Np / kTileRows;
  for (int i = 1; i < n; ++i)
    if (Ls[i]->bits != Ls[0]->bits) return UNISVQ_ERR_UNSUPPORTED;
  const bool bits3 = Ls[0]->bits == 3;   // d <= 4 (unisvq_pack_bits)
  const bool d8 = group_dv(Ls, n) == 8;
  const size_t sstat = d8 ? static_smem<8>() : static_smem<4>();
  const size_t cap = kSmemPerSm - kSmemPerCtaReserved - sstat;
  for (int m0 = 0; m0 < M;) {
    // up to 32 tokens per launch; fewer when the folded slice of a long K
    // would not fit in shared memory
    int mc = M - m0 < kGMaxTok ? M - m0 : kGMaxTok;
    DecodePlan p = plan_rows(nb, Ls[0]->KT, Ls[0]->num_sms, mc, sstat);
    while (p.smem > cap && mc > 1) {
      mc = (mc + 1) / 2;
      p = plan_rows(nb, Ls[0]->KT, Ls[0]->num_sms, mc, sstat);
    }
    if (p.smem > cap) return UNISVQ_ERR_UNSUPPORTED;
    unisvq_status st;
    if (bits3)
      st = p.nt == 1   ? gemv_launch_nt<1, 4, 3>(Ls, n, p, x, ys, m0, mc, s)
           : p.nt == 2 ? gemv_launch_nt<2, 4, 3>(Ls, n, p, x, ys, m0, mc, s)
                       : gemv_launch_nt<4, 4, 3>(Ls, n, p, x, ys, m0, mc, s);
    else if (d8)
      st = p.nt == 1   ? gemv_launch_nt<1, 8, 2>(Ls, n, p, x, ys, m0, mc, s)
           : p.nt == 2 ? gemv_launch_nt<2, 8, 2>(Ls, n, p, x, ys, m0, mc, s)
                       : gemv_launch_nt<4, 8, 2>(Ls, n, p, x, ys, m0, mc, s);
    else
      st = p.nt == 1   ? gemv_launch_nt<1, 4, 2>(Ls, n, p, x, ys, m0, mc, s)
           : p.nt == 2 ? gemv_launch_nt<2, 4, 2>(Ls, n, p, x, ys, m0, mc, s)
                       : gemv_launch_nt<4, 4, 2>(Ls, n, p, x, ys, m0, mc, s);
    if (st != UNISVQ_OK) return st;
    m0 += mc;
  }
  return UNISVQ_OK;
}

unisvq_status launch_gemv(const unisvq_layer* L, const void* x, void* y, int M, cudaStream_t s) {
  return launch_gemv_group(&L, 1, x, &y, M, s);
}

namespace {
bool rows_fit(int M, int KT, bool d8) {
  return M >= 1 && M <= kRMaxTok &&
         rows_smem(M, KT, nullptr, nullptr) <= kSmemPerSm / 2 - kSmemPerCtaReserved -
                                                   (d8 ? static_smem<8>() : static_smem<4>());
}
}  // namespace

bool gemv_rows_supported(const unisvq_layer* L, int M) { return L->bits == 2 && rows_fit(M, L->KT, L->d == 8); }

unisvq_status launch_gemv_rows_group(const unisvq_layer* const* Ls, int n, const void* x, void* const* ys, int M,
                                     cudaStream_t s) {
  if (n < 1 || n > kMaxGroup) return UNISVQ_ERR_INVALID_ARG;
  const bool d8 = group_dv(Ls, n) == 8;
  for (int m0 = 0; m0 < M; m0 += kRMaxTok) {
    const int mc = M - m0 < kRMaxTok ? M - m0 : kRMaxTok;
    if (!rows_fit(mc, Ls[0]->KT, d8)) return UNISVQ_ERR_UNSUPPORTED;
    const unisvq_status st = d8 ? rows_launch<8>(Ls, n, x, ys, m0, mc, s) : rows_launch<4>(Ls, n, x, ys, m0, mc, s);
    if (st != UNISVQ_OK) return st;
  }
  return UNISVQ_OK;
}

}  // namespace unisvq
