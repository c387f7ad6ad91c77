// Decode GEMV for layers with one affine map per (output row, 128-column group).
//
// With (A, B) varying per row the affine map cannot be folded onto the
// activations (Eq. col:matmul needs one A for every row). Summed over the
// vectors v of one group, Eq. (def:unisvq) gives
//   sum_v x_v . (A z_v + B) = sum_{r,c} A[r][c] S_rc + sum_r B[r] X_r,
//   S_rc = sum_v x[v d + r] z[v d + c],   X_r = sum_v x[v d + r],
// so the codes meet the activations first (S, on the tensor cores) and the
// row's A and B are applied to the d x d moments afterwards, once per group.
//
// Packing (pack_codes_grouped_host): inside every 128-column group the codes
// are permuted so that each 16-column chunk of an m16n8k16 A fragment holds a
// single coordinate c. Chunk q = 4h + s of the tile (half h, shift s of the
// packed layout, layout.h) belongs to class c = q / (8/d); its position
// (quarter t, byte b) holds vector v = 16 (q mod 8/d) + 4t + e(b) with
// e(b) = (b >> 1) | ((b & 1) << 1), i.e. the code of group column v d + c.
// The B fragment of lane (g', t') for chunk q is then the activations of
// vectors 16 (q mod 8/d) + 4t' + 0..3 at coordinate r, for the MMA column
// n = g' + 8 nt = m d + r (token m, coordinate r), times 2^P 4^-s (the
// subnormal codes carry 4^s 2^-24, as in gemv_kernel).
//
// Metadata: fp16 [row block][k-tile][128 rows][MD], MD = d*d + d (A row-major,
// then B), copied into shared memory for the CTA's K slice by one bulk copy.
//
// Per CTA: 128 rows x one K slice, eight warps of 16 rows; the K slices of a
// row block form a cluster and add their partial sums in the owner CTA, as in
// gemv_kernel. A lane's MMA columns are (m, r) pairs with fixed r in
// {2t mod d, (2t + 1) mod d}; after the chunks of class c it adds
// A[row][r][c] * S to its running sums, and once per k-tile B[row][r] * X_r.
#include "common.cuh"
#include "mma_sync.cuh"
#include "internal.h"

namespace unisvq {
namespace {

constexpr int kWThreads = 256;   // eight warps, one 16-row unit each
constexpr int kWWarps = 8;
constexpr int kWDepth = 8;       // k-tiles of codes in flight per warp
constexpr int kWMaxSplit = 8;    // K slices per row block (cluster size)
constexpr int kWMaxGroup = UNISVQ_MAX_GROUP;
constexpr size_t kWSmemPerSm = 228 * 1024;
constexpr size_t kWSmemReserved = 1024;

__host__ __device__ constexpr int meta_words(int d) { return d * d + d; }   // fp16 per row per group

struct GrpLayer {
  const uint8_t* codes;
  const uint16_t* meta;   // fp16 [Np/128][KT][128][MD]
  uint16_t* y;            // bf16 [M][N]
  int N;
  int rb0;                // first grid.y row block of this layer
};

struct GrpArgs {
  const uint16_t* x;      // bf16 [M][K]
  int M, K, KT;
  int kt_per_cta;
  int off_b, off_xs, off_meta, off_xsum, off_red, off_tok;
  int xs_stride;          // bf16 elements per staged token row
  int nlayers;
  int* err;
  GrpLayer layer[kWMaxGroup];
};

// Shared memory of one CTA (offsets in bytes).
struct GrpShape {
  size_t smem;
  int off_b, off_xs, off_meta, off_xsum, off_red, off_tok, xs_stride;
};

// A[r][0..D-1] of one row's record as floats (fp16 in shared memory).
template <int D>
__device__ __forceinline__ void load_arow(const uint16_t* rec, int r, float (&a)[D]) {
  const uint16_t* p = rec + r * D;
  if constexpr (D == 1) {
    a[0] = __half2float(__ushort_as_half(p[0]));
  } else if constexpr (D == 2) {
    const uint32_t w = *reinterpret_cast<const uint32_t*>(p);
    a[0] = f16_lo(w);
    a[1] = f16_hi(w);
  } else if constexpr (D == 4) {
    const uint2 w = *reinterpret_cast<const uint2*>(p);
    a[0] = f16_lo(w.x);
    a[1] = f16_hi(w.x);
    a[2] = f16_lo(w.y);
    a[3] = f16_hi(w.y);
  } else {
    const uint4 w = *reinterpret_cast<const uint4*>(p);
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      a[2 * i] = f16_lo(ws[i]);
      a[2 * i + 1] = f16_hi(ws[i]);
    }
  }
}

// D: vector length; NT: n8 column tiles (columns m D + r, so 8 NT / D tokens).
template <int D, int NT>
__global__ void __launch_bounds__(kWThreads, D == 8 ? 1 : 2) gemv_grouped_kernel(const __grid_constant__ GrpArgs a) {
  constexpr int MP = 8 * NT / D;   // tokens per launch
  constexpr int NQ = 8 / D;        // 16-column chunks per coordinate class
  constexpr int MD = meta_words(D);
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
  for (int i = 1; i < kWMaxGroup; ++i)
    if (i < a.nlayers && static_cast<int>(blockIdx.y) >= a.layer[i].rb0) li = i;
  const uint8_t* codes = nullptr;
  const uint16_t* meta = nullptr;
  uint16_t* yout = nullptr;
  int N = 0, rb = 0;
#pragma unroll
  for (int i = 0; i < kWMaxGroup; ++i)
    if (i == li) {
      codes = a.layer[i].codes;
      meta = a.layer[i].meta;
      yout = a.layer[i].y;
      N = a.layer[i].N;
      rb = static_cast<int>(blockIdx.y) - a.layer[i].rb0;
    }
  const int rows_per = (kTileRows + KS - 1) / KS;   // rows whose K-slice sums this CTA adds up
  const int own0 = static_cast<int>(blockIdx.x) * rows_per;
  const int nown = max(0, min(kTileRows, own0 + rows_per) - own0);

  uint2* bsm = reinterpret_cast<uint2*>(smem + a.off_b);                 // [kt][q][nt][lane]
  uint16_t* xs = reinterpret_cast<uint16_t*>(smem + a.off_xs);           // [token][slice] bf16
  const uint16_t* ms = reinterpret_cast<const uint16_t*>(smem + a.off_meta);   // [kt][128][MD] fp16
  float* xsum = reinterpret_cast<float*>(smem + a.off_xsum);             // [kt][MP][D] X_r 2^(P-24)
  float* red = reinterpret_cast<float*>(smem + a.off_red);
  int* pexp = reinterpret_cast<int*>(smem + a.off_tok);                  // [MP]
  const uint32_t meta_bar = sbase + a.off_tok + 128;
  const uint32_t red_bar = sbase + a.off_tok + 136;
  const uint32_t meta_bytes = n_kt > 0 ? static_cast<uint32_t>(n_kt) * kTileRows * MD * 2u : 0u;

  if (tid == 0) {
    mbar_init(meta_bar, 1);
    if (KS > 1) mbar_init(red_bar, 1);
    fence_mbar_init();
    if (n_kt <= 0) record_error(a.err, kErrBadLaunch);
  }
  __syncthreads();
  if (tid == 0) {
    // The metadata does not depend on the previous kernel: fetch it now.
    if (meta_bytes) {
      mbar_arrive_expect_tx(meta_bar, meta_bytes);
      bulk_g2s(sbase + a.off_meta, meta + (static_cast<size_t>(rb) * a.KT + kt0) * kTileRows * MD, meta_bytes,
               meta_bar, policy_evict_first());
    }
    // Reduction barrier: this arrival plus the bytes the other cluster CTAs
    // store into this CTA's slots (st.async counts them).
    if (KS > 1) mbar_arrive_expect_tx(red_bar, static_cast<uint32_t>((KS - 1) * nown * M * 4));
  }
  if (KS > 1) cluster_arrive_relaxed();

  // ---- codes: unit `warp` (rows 16 warp .. +15) of every k-tile of the slice ----
  const int g = lane >> 2, t = lane & 3;
  const uint8_t* cbase =
      codes + (static_cast<size_t>(rb) * a.KT + kt0) * kTileBytes + warp * kUnitBytes + lane * 16;
  uint4 cw[kWDepth];
#pragma unroll
  for (int s = 0; s < kWDepth; ++s)
    if (s < n_kt) cw[s] = ldg_stream_v4(cbase + static_cast<size_t>(s) * kTileBytes);
  pdl_launch_dependents();

  pdl_wait();   // x may be the previous kernel's output

  // ---- pass A (warp w: tokens w, w + 8, ...): stage x, max |x|, X_r per k-tile ----
  const int kbeg = kt0 * kTileCols;
  const int kend = min(a.K, (kt0 + max(n_kt, 0)) * kTileCols);
  const int nch = max(n_kt, 0) * (kTileCols / 8);   // 8-column chunks of the slice
  const bool vec8 = (a.K & 7) == 0;
  for (int tk = warp; tk < MP; tk += kWWarps) {
    if (tk >= M) {   // absent tokens: zero X and scale
      for (int idx = lane; idx < max(n_kt, 0) * D; idx += 32) xsum[((idx / D) * MP + tk) * D + idx % D] = 0.f;
      if (lane == 0) pexp[tk] = 0;
      continue;
    }
    const uint16_t* row = a.x + static_cast<size_t>(tk) * a.K;
    uint16_t* xrow = xs + tk * a.xs_stride;
    float mx = 0.f;
    for (int c0 = 0; c0 < nch; c0 += 32 * 4) {
      uint4 u[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int ci = c0 + lane + 32 * j;
        u[j] = ci < nch ? load_x8(row, kbeg + 8 * ci, kend, vec8) : make_uint4(0, 0, 0, 0);
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int ci = c0 + lane + 32 * j;
        if (ci < nch) *reinterpret_cast<uint4*>(xrow + 8 * ci) = u[j];
        // Column kbeg + 8 ci + e has coordinate e mod D (kbeg and 8 ci are multiples of 8).
        float sr[D];
#pragma unroll
        for (int r = 0; r < D; ++r) sr[r] = 0.f;
        const uint32_t w4[4] = {u[j].x, u[j].y, u[j].z, u[j].w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float v0 = bf16_lo(w4[q]), v1 = bf16_hi(w4[q]);
          mx = fmaxf(mx, fmaxf(fabsf(v0), fabsf(v1)));
          sr[(2 * q) % D] += v0;
          sr[(2 * q + 1) % D] += v1;
        }
        // The 16 lanes of a half-warp hold the 16 chunks of one k-tile.
#pragma unroll
        for (int r = 0; r < D; ++r)
#pragma unroll
          for (int off = 8; off; off >>= 1) sr[r] += __shfl_xor_sync(0xffffffffu, sr[r], off);
        if ((lane & 15) == 0 && ci < nch) {
#pragma unroll
          for (int r = 0; r < D; ++r) xsum[((ci >> 4) * MP + tk) * D + r] = sr[r];
        }
      }
    }
#pragma unroll
    for (int off = 16; off; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    const int P = token_scale_exp(mx);
    __syncwarp();
    const float xscale = exp2i(P - 24);
    for (int idx = lane; idx < n_kt * D; idx += 32) xsum[((idx / D) * MP + tk) * D + idx % D] *= xscale;
    if (lane == 0) pexp[tk] = P;
  }
  __syncthreads();

  // ---- pass B (all threads): the B fragments of every (k-tile, chunk, n8 tile, lane) ----
  const int nent = max(n_kt, 0) * 8 * NT * 32;
  for (int e = tid; e < nent; e += kWThreads) {
    const int L = e & 31, nt = (e >> 5) % NT, q = (e / (32 * NT)) & 7, kt = e / (256 * NT);
    const int n = 8 * nt + (L >> 2);
    const int m = n / D, r = n % D;
    uint2 v = make_uint2(0u, 0u);
    if (m < M) {
      const int v0 = 16 * (q % NQ) + 4 * (L & 3);
      const uint16_t* xr = xs + m * a.xs_stride + kt * kTileCols + v0 * D + r;
      const float sc = exp2i(pexp[m] - 2 * (q & 3));
      v.x = pack_half2(__uint_as_float(static_cast<uint32_t>(xr[0]) << 16) * sc,
                       __uint_as_float(static_cast<uint32_t>(xr[D]) << 16) * sc);
      v.y = pack_half2(__uint_as_float(static_cast<uint32_t>(xr[2 * D]) << 16) * sc,
                       __uint_as_float(static_cast<uint32_t>(xr[3 * D]) << 16) * sc);
    }
    bsm[e] = v;
  }
  // A timed-out wait has recorded its error; the kernel still runs to the
  // end so that every partial sum reaches its owner.
  if (meta_bytes) mbar_wait(meta_bar, 0, a.err, kErrTimeoutFull);
  __syncthreads();

  // ---- main loop: moments per coordinate class, the row's A and B applied per k-tile ----
  // Lane columns n = 8 nt + 2t + (0, 1): coordinates rA, rB (the same for every nt).
  const int rA = (2 * t) % D, rB = (2 * t + 1) % D;
  float acc[NT][4], yacc[NT][4];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
#pragma unroll
    for (int e = 0; e < 4; ++e) yacc[nt][e] = 0.f;
  const uint2* bl = bsm + lane;
  const uint16_t* rec0 = ms + (16 * warp + g) * MD;   // rows g and g + 8 of this warp's unit
  const uint16_t* rec1 = rec0 + 8 * MD;
  for (int i0 = 0; i0 < n_kt; i0 += kWDepth) {
#pragma unroll
    for (int sd = 0; sd < kWDepth; ++sd) {
      const int i = i0 + sd;
      if (i < n_kt) {
        const uint16_t* m0 = rec0 + i * kTileRows * MD;
        const uint16_t* m1 = rec1 + i * kTileRows * MD;
        float a0A[D], a0B[D], a1A[D], a1B[D];   // A[row][rA or rB][0..D-1], rows g and g + 8
        load_arow<D>(m0, rA, a0A);
        load_arow<D>(m0, rB, a0B);
        load_arow<D>(m1, rA, a1A);
        load_arow<D>(m1, rB, a1B);
        float b0A, b0B, b1A, b1B;               // B[row][rA], B[row][rB]
        if constexpr (D == 1) {
          b0A = b0B = __half2float(__ushort_as_half(m0[1]));
          b1A = b1B = __half2float(__ushort_as_half(m1[1]));
        } else {
          const uint32_t w0 = *reinterpret_cast<const uint32_t*>(m0 + D * D + rA);
          const uint32_t w1 = *reinterpret_cast<const uint32_t*>(m1 + D * D + rA);
          b0A = f16_lo(w0);
          b0B = f16_hi(w0);
          b1A = f16_lo(w1);
          b1B = f16_hi(w1);
        }
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
          for (int e = 0; e < 4; ++e) acc[nt][e] = 0.f;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const int h = q >> 2, s = q & 3;
          const uint32_t wa = h ? cw[sd].z : cw[sd].x, wb = h ? cw[sd].w : cw[sd].y;   // rows g, g + 8
          const uint32_t msk = 0x00030003u << (2 * s);
#pragma unroll
          for (int nt = 0; nt < NT; ++nt)
            mma_16816(acc[nt], wa & msk, wb & msk, (wa >> 8) & msk, (wb >> 8) & msk,
                          bl[((i * 8 + q) * NT + nt) * 32]);
          if (q % NQ == NQ - 1) {   // last chunk of class c: apply A[row][r][c]
            const int c = q / NQ;
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
              yacc[nt][0] = fmaf(a0A[c], acc[nt][0], yacc[nt][0]);
              yacc[nt][1] = fmaf(a0B[c], acc[nt][1], yacc[nt][1]);
              yacc[nt][2] = fmaf(a1A[c], acc[nt][2], yacc[nt][2]);
              yacc[nt][3] = fmaf(a1B[c], acc[nt][3], yacc[nt][3]);
#pragma unroll
              for (int e = 0; e < 4; ++e) acc[nt][e] = 0.f;
            }
          }
        }
        // B[row][r] X_r of this group (X already carries 2^(P - 24)).
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          const int n0 = 8 * nt + 2 * t;
          const float2 X = D == 1 ? *reinterpret_cast<const float2*>(xsum + i * MP + n0)
                                  : *reinterpret_cast<const float2*>(xsum + (i * MP + n0 / D) * D + rA);
          yacc[nt][0] = fmaf(b0A, X.x, yacc[nt][0]);
          yacc[nt][1] = fmaf(b0B, X.y, yacc[nt][1]);
          yacc[nt][2] = fmaf(b1A, X.x, yacc[nt][2]);
          yacc[nt][3] = fmaf(b1B, X.y, yacc[nt][3]);
        }
        if (i + kWDepth < n_kt) cw[sd] = ldg_stream_v4(cbase + static_cast<size_t>(i + kWDepth) * kTileBytes);
      }
    }
  }

  // ---- per (row, token) partial sums -> owner CTA slot [rank][row - owner base][token] ----
  const uint32_t red_addr = sbase + a.off_red;
  if (KS > 1) cluster_wait();   // every CTA of the cluster has initialised its barrier
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
      if constexpr (D == 1) {
        const int tok = 8 * nt + 2 * t;   // columns are tokens tok, tok + 1
        if (tok < M) {
          const float v0 = yacc[nt][2 * rh] * exp2i(24 - pexp[tok]);
          const float v1 = tok + 1 < M ? yacc[nt][2 * rh + 1] * exp2i(24 - pexp[tok + 1]) : 0.f;
          if (local) {
            red[row_off + tok] = v0;
            if (tok + 1 < M) red[row_off + tok + 1] = v1;
          } else if (tok + 1 < M) {
            st_async_v2f32(rslot + tok * 4u, v0, v1, rbar);
          } else {
            st_async_f32(rslot + tok * 4u, v0, rbar);
          }
        }
      } else {
        // Sum over the coordinates r of one token: both columns of this lane,
        // then the lanes that hold the token's other coordinates.
        float v = yacc[nt][2 * rh] + yacc[nt][2 * rh + 1];
        if constexpr (D >= 4) v += __shfl_xor_sync(0xffffffffu, v, 1);
        if constexpr (D >= 8) v += __shfl_xor_sync(0xffffffffu, v, 2);
        const int tok = (8 * nt + 2 * t) / D;
        if (rA == 0 && tok < M) {
          v *= exp2i(24 - pexp[tok]);
          if (local) red[row_off + tok] = v;
          else st_async_f32(rslot + tok * 4u, v, rbar);
        }
      }
    }
  }

  // ---- reduction over the K slices of the row block ----
  __syncthreads();   // this CTA's own slots
  if (KS > 1 && nown > 0 && !mbar_wait_cluster(red_bar, 0, a.err, kErrTimeoutReduce)) return;
  for (int idx = tid; idx < nown * M; idx += kWThreads) {
    const int tok = idx / nown;
    const int rl = idx - tok * nown;
    const int n = rb * kTileRows + own0 + rl;
    float sum = 0.f;
#pragma unroll
    for (int q = 0; q < kWMaxSplit; ++q)
      if (q < KS) sum += red[(q * rows_per + rl) * MP + tok];
    if (n < N) yout[static_cast<size_t>(tok) * N + n] = f32_to_bf16_rn(sum);
  }
}

size_t align16(size_t v) { return (v + 15) / 16 * 16; }

GrpShape grp_shape(int M, int kpc, int ks, int D, int NT) {
  GrpShape s{};
  const int MP = 8 * NT / D;
  size_t off = static_cast<size_t>(kpc) * 8 * NT * 256;   // B fragments
  s.off_b = 0;
  s.xs_stride = kpc * kTileCols + 8;
  s.off_xs = static_cast<int>(align16(off));
  off = s.off_xs + static_cast<size_t>(M) * s.xs_stride * 2;
  s.off_meta = static_cast<int>(align16(off));
  off = s.off_meta + static_cast<size_t>(kpc) * kTileRows * meta_words(D) * 2;
  s.off_xsum = static_cast<int>(align16(off));
  off = s.off_xsum + static_cast<size_t>(kpc) * MP * D * 4;
  const int rows_per = (kTileRows + ks - 1) / ks;
  s.off_red = static_cast<int>(align16(off));
  off = s.off_red + static_cast<size_t>(ks) * rows_per * MP * 4;
  s.off_tok = static_cast<int>(align16(off));
  s.smem = s.off_tok + 144;   // pexp[<= 32], two mbarriers at +128 and +136
  return s;
}

int nt_for(int M, int D) {
  const int cols = M * D;
  return cols <= 8 ? 1 : (cols <= 16 ? 2 : 4);
}

// K split for nb row blocks: among the splits ks <= 8 whose slice fits in
// shared memory, the one with the least estimated time, waves x (k-tiles per
// CTA + 2), where a wave is the resident CTAs (two per SM when shared memory
// and registers allow) and the 2 stands for a CTA's fixed cost (activation
// staging, fold and reduction). ks = 0: nothing fits.
DecodePlan plan_grp(int nb, int KT, int num_sms, int M, int D) {
  DecodePlan p{};
  p.nt = nt_for(M, D);
  p.nb = nb;
  const size_t cap = kWSmemPerSm - kWSmemReserved;
  long long best_cost = -1;
  for (int c = kWMaxSplit; c >= 1; --c) {
    if (c > KT) continue;
    const int kpc = (KT + c - 1) / c;
    const int ks = (KT + kpc - 1) / kpc;
    if (ks != c) continue;
    const size_t smem = grp_shape(M, kpc, ks, D, p.nt).smem;
    if (smem > cap) continue;
    const int per_sm = (D < 8 && kWSmemPerSm / (smem + kWSmemReserved) >= 2) ? 2 : 1;
    const long long slots = static_cast<long long>(per_sm) * num_sms;
    const long long waves = (static_cast<long long>(nb) * ks + slots - 1) / slots;
    const long long cost = waves * (kpc + 2);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      p.ks = ks;
    }
  }
  if (!p.ks) return p;
  p.kt_per_cta = (KT + p.ks - 1) / p.ks;
  p.ks = (KT + p.kt_per_cta - 1) / p.kt_per_cta;
  p.smem = grp_shape(M, p.kt_per_cta, p.ks, D, p.nt).smem;
  return p;
}

// Estimated time of one launch of plan p: waves x (k-tiles per CTA x NT + 2),
// NT n8 column tiles per k-tile and 2 for a CTA's fixed cost (activation
// staging, fold, reduction).
long long grp_cost(const DecodePlan& p, int M, int D, int num_sms) {
  const size_t smem = grp_shape(M, p.kt_per_cta, p.ks, D, p.nt).smem;
  const int per_sm = (D < 8 && kWSmemPerSm / (smem + kWSmemReserved) >= 2) ? 2 : 1;
  const long long slots = static_cast<long long>(per_sm) * num_sms;
  const long long waves = (static_cast<long long>(p.nb) * p.ks + slots - 1) / slots;
  return waves * (static_cast<long long>(p.kt_per_cta) * p.nt + 2);
}

// Tokens per launch: 32/D, 16/D or 8/D (four, two or one n8 column tiles),
// whichever gives the least estimated time for the M tokens (launches x
// grp_cost): a launch that fits two CTAs per SM often beats one with twice the
// tokens that fits only one. A cap whose shared memory does not fit is skipped.
int grp_tokens(int nb, int KT, int num_sms, int M, int D, DecodePlan* out) {
  int best_mc = 0;
  long long best = -1;
  DecodePlan best_p{};
  for (int cap = 32 / D; cap >= 1 && cap >= 8 / D; cap /= 2) {
    const int mc = M < cap ? M : cap;
    const DecodePlan p = plan_grp(nb, KT, num_sms, mc, D);
    if (!p.ks) continue;
    const long long cost = static_cast<long long>((M + mc - 1) / mc) * grp_cost(p, mc, D, num_sms);
    if (best < 0 || cost < best) {
      best = cost;
      best_mc = mc;
      best_p = p;
    }
    if (M <= cap / 2) break;   // the next cap would give the same launch
  }
  if (!best_mc) {   // nothing fits at 8/D tokens: halve further
    int mc = M < 8 / D ? M : (8 / D > 0 ? 8 / D : 1);
    DecodePlan p = plan_grp(nb, KT, num_sms, mc, D);
    while (!p.ks && mc > 1) {
      mc = (mc + 1) / 2;
      p = plan_grp(nb, KT, num_sms, mc, D);
    }
    *out = p;
    return p.ks ? mc : 0;
  }
  *out = best_p;
  return best_mc;
}

template <int D, int NT>
unisvq_status grp_launch(const unisvq_layer* const* Ls, int n, const DecodePlan& p, const void* x, void* const* ys,
                         int m0, int M, cudaStream_t s) {
  static bool attr_set[64] = {};
  const int dev = Ls[0]->device;
  if (dev < 0 || dev >= 64) return UNISVQ_ERR_CUDA;
  if (!attr_set[dev]) {
    if (cudaFuncSetAttribute(gemv_grouped_kernel<D, NT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(kWSmemPerSm - kWSmemReserved)) != cudaSuccess)
      return UNISVQ_ERR_CUDA;
    attr_set[dev] = true;
  }
  const GrpShape sh = grp_shape(M, p.kt_per_cta, p.ks, D, NT);
  GrpArgs a{};
  a.x = static_cast<const uint16_t*>(x) + static_cast<size_t>(m0) * Ls[0]->K;
  a.M = M;
  a.K = Ls[0]->K;
  a.KT = Ls[0]->KT;
  a.kt_per_cta = p.kt_per_cta;
  a.off_b = sh.off_b;
  a.off_xs = sh.off_xs;
  a.off_meta = sh.off_meta;
  a.off_xsum = sh.off_xsum;
  a.off_red = sh.off_red;
  a.off_tok = sh.off_tok;
  a.xs_stride = sh.xs_stride;
  a.nlayers = n;
  a.err = device_error_word();
  int rb0 = 0;
  for (int i = 0; i < n; ++i) {
    GrpLayer& g = a.layer[i];
    g.codes = Ls[i]->codes;
    g.meta = Ls[i]->meta;
    g.y = static_cast<uint16_t*>(ys[i]) + static_cast<size_t>(m0) * Ls[i]->N;
    g.N = Ls[i]->N;
    g.rb0 = rb0;
    rb0 += Ls[i]->Np / kTileRows;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.ks, p.nb, 1);
  cfg.blockDim = dim3(kWThreads, 1, 1);
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
  return cudaLaunchKernelEx(&cfg, gemv_grouped_kernel<D, NT>, a) == cudaSuccess ? UNISVQ_OK : UNISVQ_ERR_CUDA;
}

template <int D>
unisvq_status grp_launch_d(const unisvq_layer* const* Ls, int n, const DecodePlan& p, const void* x, void* const* ys,
                           int m0, int M, cudaStream_t s) {
  if (p.nt == 1) return grp_launch<D, 1>(Ls, n, p, x, ys, m0, M, s);
  if (p.nt == 2) return grp_launch<D, 2>(Ls, n, p, x, ys, m0, M, s);
  return grp_launch<D, 4>(Ls, n, p, x, ys, m0, M, s);
}

}  // namespace

DecodePlan plan_grouped(const unisvq_layer* L, int nb, int M, int* tokens_per_launch) {
  DecodePlan p{};
  const int mc = grp_tokens(nb, L->KT, L->num_sms, M, L->d, &p);
  if (tokens_per_launch) *tokens_per_launch = mc;
  return p;
}

unisvq_status launch_grouped_group(const unisvq_layer* const* Ls, int n, const void* x, void* const* ys, int M,
                                   cudaStream_t s) {
  if (n < 1 || n > kWMaxGroup) return UNISVQ_ERR_INVALID_ARG;
  const int D = Ls[0]->d;
  int nb = 0;
  for (int i = 0; i < n; ++i) {
    if (!Ls[i]->grouped || Ls[i]->d != D || Ls[i]->K != Ls[0]->K) return UNISVQ_ERR_UNSUPPORTED;
    nb += Ls[i]->Np / kTileRows;
  }
  for (int m0 = 0; m0 < M;) {
    DecodePlan p{};
    const int mc = grp_tokens(nb, Ls[0]->KT, Ls[0]->num_sms, M - m0, D, &p);
    if (!mc) return UNISVQ_ERR_UNSUPPORTED;
    unisvq_status st;
    switch (D) {
      case 1: st = grp_launch_d<1>(Ls, n, p, x, ys, m0, mc, s); break;
      case 2: st = grp_launch_d<2>(Ls, n, p, x, ys, m0, mc, s); break;
      case 4: st = grp_launch_d<4>(Ls, n, p, x, ys, m0, mc, s); break;
      default: st = grp_launch_d<8>(Ls, n, p, x, ys, m0, mc, s); break;
    }
    if (st != UNISVQ_OK) return st;
    m0 += mc;
  }
  return UNISVQ_OK;
}

}  // namespace unisvq
