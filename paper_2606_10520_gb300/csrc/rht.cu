// Randomized Hadamard transform of activation rows (Eq. def:hadamard, Sec. 3.2.1).
//
// The weights were rotated before quantisation, R(W) = U S_U W S_V V, so the
// layer computes y = ((x S_V V) W_hat^T) U S_U: the rows of x are rotated on
// the way in (signs, then V) and the rows of the output on the way out (U,
// then signs). U and V are normalised Hadamard matrices H_n / sqrt(n) of order
// n = 2^a m: Sylvester's H_{2^a} Kronecker a Paley matrix H_m, m in
// {1, 12, 20, 28, 344}; entry [(p, q), (p', q')] (index p m + q) is
// H_{2^a}[p][p'] H_m[q][q']. m = 344 (Paley I over the field of 7^3
// elements) makes widths such as 11008 = 2^5 * 344 rotatable.
//
// A row is split over a cluster of G CTAs (rht_ctas: 8 or 16), CTA j
// holding the 2^a / G consecutive m-blocks j 2^a / G .. in shared memory
// (fp32). Phase 1, local: signs (on the way in), the row-vector product with
// H_m inside every block (registers; signs of H_m as per-column bit masks),
// and the Sylvester butterflies between blocks of the chunk (radix-8 passes,
// three stages per pass in registers, one barrier per pass). Phase 2, after a
// cluster barrier: the remaining log2 G Sylvester stages run across the
// chunks; CTA j takes the j-th G-th of the positions, reads the G values of a
// position from the G CTAs' shared memory, transforms them in registers and
// writes the scaled (and, on the way out, signed) bf16 results. A second
// cluster barrier keeps every CTA's shared memory alive until all reads end.
#include <atomic>
#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>
#include <vector>

#include "common.cuh"
#include "hadamard.cuh"
#include "internal.h"

namespace unisvq {
namespace {

constexpr int kRThreads = 256;
constexpr int kMaxPaley = 28;     // largest order whose column masks fit one word
constexpr int kP344 = 344;                        // 7^3 + 1
constexpr int kP344Steps = (kP344 + 15) / 16;     // 22 steps of 16 (mma M over columns, mma K over rows)
constexpr int kP344Blocks = 8;                    // blocks per mma column tile (mma N)
constexpr int kP344Words = 6;                     // 22 steps x 8 bits per lane
constexpr int kP344TilesPerWarp = (kP344Steps + kRThreads / 32 - 1) / (kRThreads / 32);   // 3

// Sign bits of H_344 in the A-fragment order of mma.m16n8k16 with
// A[c][q] = H_344[q][c] (the transpose): for column tile mt and lane l
// (c0 = 16 mt + l / 4, c1 = c0 + 8, t = l % 4), bits 8 ks .. 8 ks + 7 of the
// 176-bit string at words [6 (32 mt + l), 6 (32 mt + l) + 6) are set where
// H_344[q][c] = -1 for (q, c) = (16 ks + 2t, c0), (16 ks + 2t + 1, c0),
// (16 ks + 2t, c1), (16 ks + 2t + 1, c1), then the same four with q + 8:
// A registers a0 .. a3 in that order, two bits each. Entries with q or c
// past 343 are +1 (they meet zero activations or produce discarded outputs).
// Written once per device from the host.
__device__ __align__(16) uint32_t g_h344_bits[kP344Steps * 32 * kP344Words];

constexpr int kMaxRowSets = UNISVQ_MAX_GROUP;

// One set of rows of one width (a layer's output rows in a group call).
struct RhtRows {
  const uint16_t* in;       // bf16 [M][in_stride]
  uint16_t* out;            // bf16 [M][out_stride] (may equal in)
  const uint8_t* signs;     // [n], 1 = negate; null = all +1
  int p2;                   // n = p2 * m
  int in_stride, out_stride;
  float scale;              // 1 / sqrt(n)
  int sign_off;             // byte offset of the staged sign bytes in shared memory
  int cta_end;              // CTAs of sets 0 .. this one (M G each)
};

// A launch rotates M rows of every set; all sets share m (so H_m) and the
// cluster size G.
struct RhtArgs {
  int m;                        // Paley order: 1, 12, 20, 28 or 344
  int G;                        // CTAs per row (cluster size), a power of 2 <= min(16, p2)
  int signs_first;              // 1: x -> (s x) H; 0: x -> (x H) s
  int nsets;
  uint32_t hm_neg[kMaxPaley];   // bit q of column q': H_m[q][q'] = -1 (m <= 28)
  const uint32_t* h344_bits;    // g_h344_bits of this device (m = 344)
  RhtRows set[kMaxRowSets];
};

__device__ __forceinline__ float bf16_to_f32(uint16_t b) { return __uint_as_float(static_cast<uint32_t>(b) << 16); }

// Row vector times H_344 for every block of 344 consecutive entries, on the
// tensor cores as D^T = H_344^T X^T: D^T[c][b] = sum_q H_344[q][c] X[b][q]
// with mma.sync m16n8k16 (bf16 operands, fp32 accumulation). M runs over the
// 344 output columns (22 tiles of 16), N over 8 blocks, K over the 344
// positions (22 steps). The B operand is the blocks in bf16 (the rotation's
// input values, exact in bf16, so every product is exact), loaded by
// ldmatrix; blocks past nblk and positions past 343 read a zeroed 16-byte
// line. The A operand is +-1 in bf16, made per lane from 8 sign bits through
// a 16-entry table (lut: the two A registers for each 4-bit pattern). Warp w
// computes column tiles w, w + 8, w + 16 as independent accumulator chains.
// This lane's sign bits of its warp's column tiles (read before the
// programmatic-launch wait: the table never depends on the previous kernel).
__device__ __forceinline__ void load_h344_bits(const uint32_t* bits, uint32_t (&w)[kP344TilesPerWarp][kP344Words]) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll
  for (int i = 0; i < kP344TilesPerWarp; ++i) {
    const int mt = warp + i * (kRThreads / 32);
#pragma unroll
    for (int k = 0; k < kP344Words; ++k)
      w[i][k] = mt < kP344Steps ? __ldg(bits + (mt * 32 + lane) * kP344Words + k) : 0u;
  }
}

__device__ __forceinline__ void paley344_mma(const uint16_t* x_bf16, float* dst, int nblk,
                                             const uint32_t (&w)[kP344TilesPerWarp][kP344Words], const uint2* lut,
                                             const uint16_t* zero16) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
  const uint32_t x_base = smem_u32(x_bf16), z_addr = smem_u32(zero16);
  // ldmatrix.x2 row addresses: lanes 0..7 the 8 blocks at k 0..7 of the
  // step, lanes 8..15 the same blocks at k 8..15 (lanes 16..31 unused)
  const int bsel = lane & 7, bkoff = ((lane >> 3) & 1) * 8;
  for (int nb = 0; nb < nblk; nb += kP344Blocks) {
    const int b = nb + bsel;
    const bool blk_ok = b < nblk;
    const uint32_t row_addr = x_base + static_cast<uint32_t>(b * kP344 + bkoff) * 2u;
    float acc[kP344TilesPerWarp][4] = {};
#pragma unroll
    for (int ks = 0; ks < kP344Steps; ++ks) {
      // the last step's second 8 positions (q = 344 .. 351) are zeros
      const bool ok = blk_ok && (16 * ks + bkoff < kP344);
      const uint32_t addr = ok ? row_addr + 32u * ks : z_addr;
      uint32_t b0, b1;
      asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0,%1}, [%2];" : "=r"(b0), "=r"(b1) : "r"(addr));
#pragma unroll
      for (int i = 0; i < kP344TilesPerWarp; ++i) {
        if (warp + i * (kRThreads / 32) < kP344Steps) {
          const uint32_t byte = (w[i][(8 * ks) >> 5] >> ((8 * ks) & 31)) & 0xffu;
          const uint2 lo = lut[byte & 15u], hi = lut[byte >> 4];
          asm volatile(
              "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
              "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
              : "+f"(acc[i][0]), "+f"(acc[i][1]), "+f"(acc[i][2]), "+f"(acc[i][3])
              : "r"(lo.x), "r"(lo.y), "r"(hi.x), "r"(hi.y), "r"(b0), "r"(b1));
        }
      }
    }
    // D^T fragment: rows c = 16 mt + g (+ 8), columns blocks nb + 2t, + 1
#pragma unroll
    for (int i = 0; i < kP344TilesPerWarp; ++i) {
      const int mt = warp + i * (kRThreads / 32);
      if (mt >= kP344Steps) continue;
      const int c = 16 * mt + g, b0 = nb + 2 * t;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int cc = c + 8 * h;
        if (cc >= kP344) continue;
        if (b0 < nblk) dst[b0 * kP344 + cc] = acc[i][2 * h];
        if (b0 + 1 < nblk) dst[(b0 + 1) * kP344 + cc] = acc[i][2 * h + 1];
      }
    }
  }
}

// G-point Sylvester transform of position e of the chunk across the cluster.
template <int G, bool kStaged>
__device__ __forceinline__ void cross_chunk(const float* buf, uint16_t* dst, int chunk, int e, float scale,
                                            const uint8_t* gsigns, const uint8_t* osg, int sgi) {
  float v[G];
  const uint32_t local = smem_u32(buf + e);
#pragma unroll
  for (int r = 0; r < G; ++r) v[r] = ld_shared_cluster_f32(map_shared_rank(local, r));
#pragma unroll
  for (int d = 1; d < G; d <<= 1)
#pragma unroll
    for (int j = 0; j < G; ++j)
      if (!(j & d)) {
        const float x0 = v[j], x1 = v[j + d];
        v[j] = x0 + x1;
        v[j + d] = x0 - x1;
      }
#pragma unroll
  for (int r = 0; r < G; ++r) {
    const int i = r * chunk + e;
    float o = v[r] * scale;
    if constexpr (kStaged) {
      if (osg && osg[sgi + r * ((chunk + G - 1) / G)]) o = -o;
    } else {
      if (gsigns && gsigns[i]) o = -o;
    }
    dst[i] = f32_to_bf16_rn(o);
  }
}

// The sign bytes a CTA applies, into shared memory (sg): on the way in those
// of its chunk, on the way out those of the positions it writes (its chunk
// when G == 1, else G segments of span positions, segment r at
// r * chunk + rank * span). Loads are issued eight per thread before their
// stores, so the copy costs about one memory latency.
__device__ __forceinline__ void stage_signs(const RhtArgs& a, const uint8_t* signs, uint8_t* sg, int nsg, int base,
                                            int chunk, int span, int rank) {
  for (int i0 = threadIdx.x; i0 < nsg; i0 += kRThreads * 8) {
    uint8_t v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int i = i0 + k * kRThreads;
      int pos = -1;
      if (i < nsg) {
        if (a.signs_first) {
          pos = base + i;
        } else if (a.G == 1) {
          pos = i;
        } else {
          const int r = i / span, e = rank * span + (i - r * span);
          pos = e < chunk ? r * chunk + e : -1;
        }
      }
      v[k] = pos >= 0 ? signs[pos] : 0;
    }
#pragma unroll
    for (int k = 0; k < 8; ++k)
      if (i0 + k * kRThreads < nsg) sg[i0 + k * kRThreads] = v[k];
  }
}

// kP344Path: the instance for m = 344 (tensor-core block product; its
// registers do not limit the residency of the others). kStaged: the sign
// bytes never change between launches (a handle's own), so they are copied to
// shared memory before the dependency wait; otherwise (the standalone
// rotation's signs, which the previous kernel may write) they are read from
// global memory where they are applied.
template <bool kP344Path, bool kStaged>
__global__ void __launch_bounds__(kRThreads, kP344Path ? 1 : 3) rht_kernel(const __grid_constant__ RhtArgs a) {
  extern __shared__ __align__(16) float smem_f[];
  float* buf = smem_f;   // the chunk; a second chunk-sized buffer follows when m > 1
  const int G = a.G;
  const int rank = G > 1 ? static_cast<int>(cluster_ctarank()) : 0;
  // this CTA's row set, its fields read with constant parameter offsets only
  const uint16_t* s_in = a.set[0].in;
  uint16_t* s_out = a.set[0].out;
  const uint8_t* s_signs = a.set[0].signs;
  int s_p2 = a.set[0].p2, s_in_stride = a.set[0].in_stride, s_out_stride = a.set[0].out_stride;
  int s_sign_off = a.set[0].sign_off, cta0 = 0;
  float s_scale = a.set[0].scale;
#pragma unroll
  for (int l = 1; l < kMaxRowSets; ++l)
    if (l < a.nsets && static_cast<int>(blockIdx.x) >= a.set[l - 1].cta_end) {
      s_in = a.set[l].in;
      s_out = a.set[l].out;
      s_signs = a.set[l].signs;
      s_p2 = a.set[l].p2;
      s_in_stride = a.set[l].in_stride;
      s_out_stride = a.set[l].out_stride;
      s_sign_off = a.set[l].sign_off;
      s_scale = a.set[l].scale;
      cta0 = a.set[l - 1].cta_end;
    }
  const int row = (static_cast<int>(blockIdx.x) - cta0) / G;
  const int pl = s_p2 / G;             // m-blocks per CTA
  const int chunk = pl * a.m;          // values per CTA
  const int base = rank * chunk;
  const int span = (chunk + G - 1) / G;   // positions per CTA in the cross-chunk stage
  uint8_t* sg = reinterpret_cast<uint8_t*>(smem_f) + s_sign_off;
  const int nsg = !s_signs ? 0 : (a.signs_first || G == 1 ? chunk : G * span);
  pdl_launch_dependents();
  uint32_t h344w[kP344Path ? kP344TilesPerWarp : 1][kP344Words];
  if constexpr (kP344Path) load_h344_bits(a.h344_bits, h344w);
  if constexpr (kStaged) stage_signs(a, s_signs, sg, nsg, base, chunk, span, rank);
  pdl_wait();   // the row may be the previous kernel's output
  if constexpr (kStaged) __syncthreads();
  // input sign byte i of the chunk
  const uint8_t* sg_in = kStaged ? sg : s_signs + base;
  const uint16_t* src = s_in + static_cast<size_t>(row) * s_in_stride + base;
  const bool sgn_in = a.signs_first && s_signs;
  // 16-byte loads where every row's chunk starts on a 16-byte boundary
  const bool vec_ok = (reinterpret_cast<uintptr_t>(s_in) & 15) == 0 && (s_in_stride & 7) == 0;
  if constexpr (kP344Path) {
    // bf16 operand copy of the chunk (signs applied: a bf16 sign flip is
    // exact), the zeroed line and the B-register table; the fp32 region at
    // the start of shared memory receives the block products.
    uint16_t* ab = reinterpret_cast<uint16_t*>(smem_f + chunk);
    uint16_t* zero16 = ab + chunk;
    uint2* lut = reinterpret_cast<uint2*>(zero16 + 8);
    if (threadIdx.x < 16) {
      const uint32_t nib = threadIdx.x;
      lut[nib] = make_uint2(0x3f803f80u | ((nib & 1u) << 15) | ((nib & 2u) << 30),
                            0x3f803f80u | ((nib & 4u) << 13) | ((nib & 8u) << 28));
    } else if (threadIdx.x == 16) {
      *reinterpret_cast<uint4*>(zero16) = make_uint4(0u, 0u, 0u, 0u);
    }
    if (vec_ok) {   // chunk is a multiple of 344, so of 8
      for (int i8 = threadIdx.x; i8 < chunk / 8; i8 += kRThreads) {
        uint4 w = ldg_v4(src + 8 * i8);
        if (sgn_in) {
          uint32_t f[4] = {0u, 0u, 0u, 0u};
#pragma unroll
          for (int k = 0; k < 8; ++k)
            if (sg_in[8 * i8 + k]) f[k >> 1] |= (k & 1) ? 0x80000000u : 0x8000u;
          w.x ^= f[0];
          w.y ^= f[1];
          w.z ^= f[2];
          w.w ^= f[3];
        }
        *reinterpret_cast<uint4*>(ab + 8 * i8) = w;
      }
    } else {
      for (int i = threadIdx.x; i < chunk; i += kRThreads) {
        uint16_t v = src[i];
        if (sgn_in && sg_in[i]) v ^= 0x8000u;
        ab[i] = v;
      }
    }
    __syncthreads();
    paley344_mma(ab, buf, pl, h344w, lut, zero16);
    __syncthreads();
  } else if ((chunk & 7) == 0 && vec_ok) {   // 16-byte loads of 8 values
    for (int i8 = threadIdx.x; i8 < chunk / 8; i8 += kRThreads) {
      const uint4 w = ldg_v4(src + 8 * i8);
      const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        float v = (k & 1) ? bf16_hi(ws[k >> 1]) : bf16_lo(ws[k >> 1]);
        if (sgn_in && sg_in[8 * i8 + k]) v = -v;
        buf[8 * i8 + k] = v;
      }
    }
  } else {
    for (int i = threadIdx.x; i < chunk; i += kRThreads) {
      float v = bf16_to_f32(src[i]);
      if (sgn_in && sg_in[i]) v = -v;
      buf[i] = v;
    }
  }
  if constexpr (!kP344Path) {
    __syncthreads();
    if (a.m > 1) {
      float* out2 = smem_f + chunk;
      if (a.m == 12) paley_blocks<kRThreads, 12>(buf, out2, pl, a.hm_neg);
      else if (a.m == 20) paley_blocks<kRThreads, 20>(buf, out2, pl, a.hm_neg);
      else paley_blocks<kRThreads, 28>(buf, out2, pl, a.hm_neg);
      buf = out2;
      __syncthreads();
    }
  }
  sylvester_all<kRThreads>(buf, pl, a.m);
  uint16_t* dst = s_out + static_cast<size_t>(row) * s_out_stride;
  if (G == 1) {
    const bool sgn_out = !a.signs_first && s_signs;
    for (int i = threadIdx.x; i < chunk; i += kRThreads) {
      float v = buf[i] * s_scale;
      if (sgn_out && (kStaged ? sg[i] : s_signs[i])) v = -v;
      dst[i] = f32_to_bf16_rn(v);
    }
    return;
  }
  cluster_sync();   // every chunk is transformed locally
  // CTA `rank` finishes positions [rank span, (rank + 1) span) of all G
  // chunks; the output signs of position e of chunk r are staged at
  // sg[r span + e - rank span]
  const uint8_t* osg = !a.signs_first && s_signs ? sg : nullptr;
  const uint8_t* gsg = !a.signs_first ? s_signs : nullptr;
  const int e1 = min(chunk, (rank + 1) * span);
  for (int e = rank * span + static_cast<int>(threadIdx.x); e < e1; e += kRThreads) {
    const int sgi = e - rank * span;
    if (G == 16) cross_chunk<16, kStaged>(buf, dst, chunk, e, s_scale, gsg, osg, sgi);
    else if (G == 8) cross_chunk<8, kStaged>(buf, dst, chunk, e, s_scale, gsg, osg, sgi);
    else if (G == 4) cross_chunk<4, kStaged>(buf, dst, chunk, e, s_scale, gsg, osg, sgi);
    else cross_chunk<2, kStaged>(buf, dst, chunk, e, s_scale, gsg, osg, sgi);
  }
  cluster_sync();   // no CTA leaves while another still reads its shared memory
}

// chi(v) mod q for prime q: +1 on nonzero squares, -1 on non-squares, 0 at 0.
int quad_char(int v, int q) {
  v = ((v % q) + q) % q;
  if (v == 0) return 0;
  for (int t = 1; t < q; ++t)
    if ((t * t) % q == v) return 1;
  return -1;
}

// Signs of a Paley Hadamard matrix of order m in {12, 20, 28}, H[i][j] in {+1, -1}.
std::vector<int> paley_signs(int m) {
  std::vector<int> H(static_cast<size_t>(m) * m, 0);
  if (m == 12 || m == 20) {
    // Paley I, q = m - 1 = 3 mod 4: H = I + S, S = [[0, 1..1], [-1.., Q]], Q[i][j] = chi(j - i)
    const int q = m - 1;
    for (int i = 0; i < m; ++i)
      for (int j = 0; j < m; ++j) {
        int s;
        if (i == 0 && j == 0) s = 0;
        else if (i == 0) s = 1;
        else if (j == 0) s = -1;
        else s = quad_char((j - 1) - (i - 1), q);
        H[static_cast<size_t>(i) * m + j] = s + (i == j ? 1 : 0);
      }
  } else {
    // Paley II, q = 13 = 1 mod 4: C = [[0, 1..1], [1.., Q]] (order 14, symmetric),
    // H = [[C + I, C - I], [C - I, -C - I]]
    const int q = 13, c = q + 1;
    std::vector<int> C(static_cast<size_t>(c) * c, 0);
    for (int i = 0; i < c; ++i)
      for (int j = 0; j < c; ++j) {
        if (i == 0 && j == 0) C[i * c + j] = 0;
        else if (i == 0 || j == 0) C[i * c + j] = 1;
        else C[i * c + j] = quad_char((j - 1) - (i - 1), q);
      }
    for (int bi = 0; bi < 2; ++bi)
      for (int bj = 0; bj < 2; ++bj)
        for (int i = 0; i < c; ++i)
          for (int j = 0; j < c; ++j) {
            const int cij = C[i * c + j], id = i == j ? 1 : 0;
            int v;
            if (bi == 0 && bj == 0) v = cij + id;
            else if (bi == 1 && bj == 1) v = -cij - id;
            else v = cij - id;
            H[static_cast<size_t>(bi * c + i) * m + bj * c + j] = v;
          }
  }
  return H;
}

// The field of 343 elements as GF(7)[t] / (t^3 - 2). t^3 - 2 has no root mod 7
// (the cubes mod 7 are 0, 1 and 6), so it is irreducible and the quotient is
// a field. Element e = e0 + 7 e1 + 49 e2 stands for e0 + e1 t + e2 t^2.
int f343_mul(int x, int y) {
  const int a[3] = {x % 7, x / 7 % 7, x / 49}, b[3] = {y % 7, y / 7 % 7, y / 49};
  int p[5] = {0, 0, 0, 0, 0};
  for (int i = 0; i < 3; ++i)
    for (int j = 0; j < 3; ++j) p[i + j] += a[i] * b[j];
  // t^3 = 2 and t^4 = 2 t
  return (p[0] + 2 * p[3]) % 7 + 7 * ((p[1] + 2 * p[4]) % 7) + 49 * (p[2] % 7);
}

int f343_sub(int x, int y) {
  int r = 0, w = 1;
  for (int i = 0; i < 3; ++i, x /= 7, y /= 7, w *= 7) r += ((x % 7 - y % 7 + 7) % 7) * w;
  return r;
}

// Quadratic character by Euler's criterion: e^((343 - 1) / 2) is 1 on the
// nonzero squares and -1 (element 6) on the other nonzero elements.
int f343_chi(int e) {
  if (e == 0) return 0;
  int r = 1, b = e;
  for (int k = 171; k; k >>= 1) {
    if (k & 1) r = f343_mul(r, b);
    b = f343_mul(b, b);
  }
  return r == 1 ? 1 : -1;
}

// The Paley I matrix of order 344, H = I + [[0, 1^T], [-1, Q]] with
// Q[i][j] = chi(e_j - e_i) (row and column 0 the point at infinity, row
// i >= 1 the field element i - 1): true where H[r][c] = -1.
bool h344_negative(const std::vector<int>& chi, int r, int c) {
  if (r == c || r == 0) return false;
  if (c == 0) return true;
  return chi[f343_sub(c - 1, r - 1)] < 0;
}

// g_h344_bits: the sign bits of H_344 in A-fragment order (see its declaration).
std::vector<uint32_t> h344_fragment_bits() {
  std::vector<int> chi(343);
  for (int e = 0; e < 343; ++e) chi[e] = f343_chi(e);
  std::vector<uint32_t> bits(static_cast<size_t>(kP344Steps) * 32 * kP344Words, 0u);
  for (int mt = 0; mt < kP344Steps; ++mt)
    for (int l = 0; l < 32; ++l) {
      const int c0 = 16 * mt + l / 4, t = l % 4;
      for (int ks = 0; ks < kP344Steps; ++ks)
        for (int e = 0; e < 8; ++e) {
          // e: bit 0 -> q + 1, bit 1 -> column c0 + 8, bit 2 -> q + 8
          const int q = 16 * ks + 2 * t + (e & 1) + 8 * (e >> 2);
          const int c = c0 + 8 * ((e >> 1) & 1);
          if (q < kP344 && c < kP344 && h344_negative(chi, q, c)) {
            const int b = 8 * ks + e;
            bits[static_cast<size_t>(mt * 32 + l) * kP344Words + b / 32] |= 1u << (b % 32);
          }
        }
    }
  return bits;
}

std::atomic<const uint32_t*> g_h344_addr[64];
std::mutex g_h344_mu;

// Device address of g_h344_bits on device `dev`, written from the host on the
// first request (a synchronous copy, so it must not run under stream capture).
const uint32_t* h344_table(int dev) {
  const uint32_t* t = g_h344_addr[dev].load(std::memory_order_acquire);
  if (t) return t;
  std::lock_guard<std::mutex> lk(g_h344_mu);
  t = g_h344_addr[dev].load(std::memory_order_acquire);
  if (t) return t;
  static const std::vector<uint32_t> host = h344_fragment_bits();
  void* addr = nullptr;
  if (cudaMemcpyToSymbol(g_h344_bits, host.data(), host.size() * sizeof(uint32_t)) != cudaSuccess ||
      cudaGetSymbolAddress(&addr, g_h344_bits) != cudaSuccess)
    return nullptr;
  t = static_cast<const uint32_t*>(addr);
  g_h344_addr[dev].store(t, std::memory_order_release);
  return t;
}

}  // namespace

unisvq_status rht_prepare(int n) {
  int p2 = 0, m = 0;
  if (!rht_factor(n, &p2, &m)) return UNISVQ_ERR_UNSUPPORTED;
  if (m != kP344) return UNISVQ_OK;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return UNISVQ_ERR_CUDA;
  return h344_table(dev) ? UNISVQ_OK : UNISVQ_ERR_CUDA;
}

bool rht_factor(int n, int* p2, int* m) {
  if (n <= 0) return false;
  const int ms[5] = {kP344, 28, 20, 12, 1};
  for (int k = 0; k < 5; ++k) {
    if (n % ms[k]) continue;
    const int p = n / ms[k];
    if ((p & (p - 1)) == 0) {
      *p2 = p;
      *m = ms[k];
      return true;
    }
  }
  return false;
}

// Shared memory of one CTA: its chunk of n / min(8, 2^a) values (twice that
// when m > 1: the product with H_m writes a second buffer).
// CTAs per row: 16 (a non-portable cluster) for rows of 16384 values or more,
// else min(8, 2^a). Measured on GB300 at n = 28672: 6.8 us against 9.0 us with
// 8 CTAs; at n = 14336 eight CTAs are faster.
// For m = 344 a CTA takes 8 blocks where there are that many (one mma column
// tile: the block product costs the same 484 MMAs for 1 to 8 blocks), so
// 11008 = 32 * 344 runs on 4 CTAs per row.
static int rht_ctas(int n, int p2, int m) {
  if (m == kP344) return p2 <= kP344Blocks ? 1 : (p2 / kP344Blocks < 16 ? p2 / kP344Blocks : 16);
  if (n >= 16384 && p2 >= 16) return 16;
  return p2 >= 8 ? 8 : p2;
}

// Shared memory of one CTA, in this order: the fp32 chunk (m = 1), or two
// fp32 chunks (m in 12, 20, 28: the block product writes the second), or for
// m = 344 the fp32 block products, the bf16 operand copy, a zeroed 16-byte
// line and the 16-entry register table; then the staged sign bytes (at most
// chunk + 16).
static size_t rht_sign_offset(int n, int p2, int m) {
  const size_t chunk = static_cast<size_t>(n / rht_ctas(n, p2, m));
  if (m == kP344) return chunk * sizeof(float) + chunk * sizeof(uint16_t) + 16 + 16 * sizeof(uint2);
  return chunk * sizeof(float) * (m > 1 ? 2 : 1);
}

size_t rht_smem_bytes(int n) {
  int p2 = 0, m = 0;
  if (!rht_factor(n, &p2, &m)) return static_cast<size_t>(n) * sizeof(float);
  const size_t chunk = static_cast<size_t>(n / rht_ctas(n, p2, m));
  return rht_sign_offset(n, p2, m) + ((chunk + 16 + 15) / 16) * 16;
}

// Column sign masks of H_m for m in {12, 20, 28} (kMaxPaley words each, bit q
// of word c set where H_m[q][c] = -1), built once.
const uint32_t* rht_paley_masks(int m) {
  static const std::vector<uint32_t> table = [] {
    std::vector<uint32_t> t(3 * kMaxPaley, 0u);
    const int orders[3] = {12, 20, 28};
    for (int k = 0; k < 3; ++k) {
      const int mm = orders[k];
      const std::vector<int> H = paley_signs(mm);
      for (int c = 0; c < mm; ++c)
        for (int q = 0; q < mm; ++q)
          if (H[static_cast<size_t>(q) * mm + c] < 0) t[k * kMaxPaley + c] |= 1u << q;
    }
    return t;
  }();
  return table.data() + (m == 12 ? 0 : (m == 20 ? 1 : 2)) * kMaxPaley;
}

unisvq_status launch_rht_sets(const RhtSetDesc* sets, int nsets, int M, int signs_first, bool signs_const,
                              cudaStream_t s) {
  if (nsets < 1 || nsets > kMaxRowSets) return UNISVQ_ERR_INVALID_ARG;
  int p2[kMaxRowSets], mm[kMaxRowSets], gg[kMaxRowSets];
  size_t smem = 0;
  bool one_launch = true;
  for (int i = 0; i < nsets; ++i) {
    if (!rht_factor(sets[i].n, &p2[i], &mm[i])) return UNISVQ_ERR_UNSUPPORTED;
    if (rht_smem_bytes(sets[i].n) > 227 * 1024) return UNISVQ_ERR_UNSUPPORTED;
    gg[i] = rht_ctas(sets[i].n, p2[i], mm[i]);
    smem = std::max(smem, rht_smem_bytes(sets[i].n));
    one_launch = one_launch && mm[i] == mm[0] && gg[i] == gg[0];
  }
  if (M <= 0) return UNISVQ_OK;
  if (!one_launch) {   // widths with different H_m or cluster sizes: one launch per set
    for (int i = 0; i < nsets; ++i) {
      const unisvq_status st = launch_rht_sets(sets + i, 1, M, signs_first, signs_const, s);
      if (st != UNISVQ_OK) return st;
    }
    return UNISVQ_OK;
  }
  static std::atomic<bool> attr_set[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return UNISVQ_ERR_CUDA;
  if (!attr_set[dev].load(std::memory_order_acquire)) {
    bool ok = true;
    for (auto k : {rht_kernel<false, false>, rht_kernel<false, true>, rht_kernel<true, false>, rht_kernel<true, true>})
      ok = ok && cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess &&
           cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024) == cudaSuccess;
    if (!ok) return UNISVQ_ERR_CUDA;
    attr_set[dev].store(true, std::memory_order_release);
  }
  const int m = mm[0], G = gg[0];
  RhtArgs a{};
  a.m = m;
  a.G = G;
  a.signs_first = signs_first;
  a.nsets = nsets;
  for (int i = 0; i < nsets; ++i) {
    RhtRows& r = a.set[i];
    r.in = static_cast<const uint16_t*>(sets[i].in);
    r.out = static_cast<uint16_t*>(sets[i].out);
    r.signs = sets[i].signs;
    r.p2 = p2[i];
    r.in_stride = sets[i].in_stride;
    r.out_stride = sets[i].out_stride;
    r.scale = static_cast<float>(1.0 / std::sqrt(static_cast<double>(sets[i].n)));
    r.sign_off = static_cast<int>(rht_sign_offset(sets[i].n, p2[i], m));
    r.cta_end = (i + 1) * M * G;
  }
  if (m == kP344) {
    a.h344_bits = h344_table(dev);
    if (!a.h344_bits) return UNISVQ_ERR_CUDA;
  } else if (m > 1) {
    std::memcpy(a.hm_neg, rht_paley_masks(m), sizeof(a.hm_neg));
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(nsets * M * G, 1, 1);
  cfg.blockDim = dim3(kRThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attrs[2];
  attrs[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attrs[0].val.programmaticStreamSerializationAllowed = 1;
  attrs[1].id = cudaLaunchAttributeClusterDimension;
  attrs[1].val.clusterDim.x = G;
  attrs[1].val.clusterDim.y = 1;
  attrs[1].val.clusterDim.z = 1;
  cfg.attrs = attrs;
  cfg.numAttrs = 2;
  void (*kern)(RhtArgs) = m == kP344 ? (signs_const ? rht_kernel<true, true> : rht_kernel<true, false>)
                                     : (signs_const ? rht_kernel<false, true> : rht_kernel<false, false>);
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kern, a);
  return e == cudaSuccess ? UNISVQ_OK : UNISVQ_ERR_CUDA;
}

int rht_set_launches(const int* ns, int nsets) {
  int p0 = 0, m0 = 0;
  if (nsets < 1 || !rht_factor(ns[0], &p0, &m0)) return nsets;
  for (int i = 1; i < nsets; ++i) {
    int p = 0, m = 0;
    if (!rht_factor(ns[i], &p, &m) || m != m0 || rht_ctas(ns[i], p, m) != rht_ctas(ns[0], p0, m0)) return nsets;
  }
  return 1;
}

unisvq_status launch_rht(const void* in, int in_stride, void* out, int out_stride, int M, int n,
                         const uint8_t* signs, int signs_first, bool signs_const, cudaStream_t s) {
  const RhtSetDesc d{in, in_stride, out, out_stride, n, signs};
  return launch_rht_sets(&d, 1, M, signs_first, signs_const, s);
}

}  // namespace unisvq
