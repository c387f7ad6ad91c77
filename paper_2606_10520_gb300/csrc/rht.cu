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
#include <cmath>
#include <mutex>
#include <vector>

#include "common.cuh"
#include "internal.h"

namespace unisvq {
namespace {

constexpr int kRThreads = 256;
constexpr int kMaxPaley = 28;     // largest order whose column masks fit one word
constexpr int kP344 = 344;        // 7^3 + 1
constexpr int kP344Words = 12;    // words per column mask of H_344 (11 used)

// Column c of H_344 at words [12 c, 12 c + 11): bit q % 32 of word q / 32 set
// where H_344[q][c] = -1. Written once per device from the host.
__device__ __align__(16) uint32_t g_h344_neg[kP344 * kP344Words];

struct RhtArgs {
  const uint16_t* in;       // bf16 [M][in_stride]
  uint16_t* out;            // bf16 [M][out_stride] (may equal in)
  const uint8_t* signs;     // [n], 1 = negate; null = all +1
  int n, p2, m;             // n = p2 * m
  int G;                    // CTAs per row (cluster size), a power of 2 <= min(16, p2)
  int in_stride, out_stride;
  int signs_first;          // 1: x -> (s x) H; 0: x -> (x H) s
  float scale;              // 1 / sqrt(n)
  uint32_t hm_neg[kMaxPaley];   // bit q of column q': H_m[q][q'] = -1 (m <= 28)
  const uint32_t* h344_neg;     // g_h344_neg of this device (m = 344)
};

__device__ __forceinline__ float bf16_to_f32(uint16_t b) { return __uint_as_float(static_cast<uint32_t>(b) << 16); }

// Row vector times H_m for every block of M_ consecutive entries of src,
// into dst: four threads per block, each forming M_/4 of its outputs.
template <int M_>
__device__ __forceinline__ void paley_blocks(const float* src, float* dst, int nblk, const uint32_t* neg) {
  constexpr int C = M_ / 4;
  for (int it = threadIdx.x; it < nblk * 4; it += kRThreads) {
    const int p = it >> 2, c0 = (it & 3) * C;
    const float* blk = src + p * M_;
    float v[M_];
#pragma unroll
    for (int q = 0; q < M_; ++q) v[q] = blk[q];
#pragma unroll
    for (int c = 0; c < C; ++c) {
      const uint32_t mask = neg[c0 + c];
      float acc = 0.f;
#pragma unroll
      for (int q = 0; q < M_; ++q) acc += ((mask >> q) & 1u) ? -v[q] : v[q];
      dst[p * M_ + c0 + c] = acc;
    }
  }
}

__device__ __forceinline__ float neg_if_bit(float v, uint32_t w, int b) {
  return __uint_as_float(__float_as_uint(v) ^ ((w << (31 - b)) & 0x80000000u));
}

// Row vector times H_344 for every block of 344 consecutive entries of src,
// into dst: one thread per output entry (block p, column c) with its column's
// sign bits in registers; the block is read as 86 float4 from shared memory
// (lanes working on one block read the same addresses: broadcasts). Two
// accumulation chains per entry.
__device__ __forceinline__ void paley344_blocks(const float* src, float* dst, int nblk, const uint32_t* neg) {
  for (int it = threadIdx.x; it < nblk * kP344; it += kRThreads) {
    const int p = it / kP344, c = it - p * kP344;
    const uint4* col = reinterpret_cast<const uint4*>(neg + c * kP344Words);
    const uint4 u0 = __ldg(col), u1 = __ldg(col + 1), u2 = __ldg(col + 2);
    const uint32_t w[kP344Words] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w, u2.x, u2.y, u2.z, u2.w};
    const float4* blk = reinterpret_cast<const float4*>(src + p * kP344);
    float acc0 = 0.f, acc1 = 0.f;
#pragma unroll
    for (int q4 = 0; q4 < kP344 / 4; ++q4) {
      const float4 v = blk[q4];
      const uint32_t ww = w[q4 >> 3];   // entries 4 q4 .. 4 q4 + 3 sit in word q4 / 8
      const int b = (q4 & 7) * 4;
      acc0 += neg_if_bit(v.x, ww, b);
      acc1 += neg_if_bit(v.y, ww, b + 1);
      acc0 += neg_if_bit(v.z, ww, b + 2);
      acc1 += neg_if_bit(v.w, ww, b + 3);
    }
    dst[it] = acc0 + acc1;
  }
}

// Sylvester stages s0 .. s0 + R - 1 (butterfly distances 2^s0 .. 2^(s0+R-1)
// blocks) for every column of the p2 x m view, R stages per pass in registers.
template <int R>
__device__ __forceinline__ void sylvester_pass(float* buf, int p2, int m, int s0) {
  constexpr int G = 1 << R;
  const int h = 1 << s0;
  const int groups = (p2 >> R) * m;
  for (int gi = threadIdx.x; gi < groups; gi += kRThreads) {
    const int col = gi % m, rest = gi / m;
    const int lo = (rest & (h - 1)) | ((rest >> s0) << (s0 + R));   // R zero bits inserted at s0
    float v[G];
#pragma unroll
    for (int j = 0; j < G; ++j) v[j] = buf[(lo + j * h) * m + col];
#pragma unroll
    for (int st = 0; st < R; ++st) {
      const int d = 1 << st;
#pragma unroll
      for (int j = 0; j < G; ++j)
        if (!(j & d)) {
          const float a = v[j], b = v[j + d];
          v[j] = a + b;
          v[j + d] = a - b;
        }
    }
#pragma unroll
    for (int j = 0; j < G; ++j) buf[(lo + j * h) * m + col] = v[j];
  }
}

// G-point Sylvester transform of position e of the chunk across the cluster.
template <int G>
__device__ __forceinline__ void cross_chunk(const RhtArgs& a, const float* buf, uint16_t* dst, int chunk, int e) {
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
    float o = v[r] * a.scale;
    if (!a.signs_first && a.signs && a.signs[i]) o = -o;
    dst[i] = f32_to_bf16_rn(o);
  }
}

__global__ void __launch_bounds__(kRThreads) rht_kernel(const __grid_constant__ RhtArgs a) {
  extern __shared__ __align__(16) float smem_f[];
  float* buf = smem_f;   // the chunk; a second chunk-sized buffer follows when m > 1
  const int G = a.G;
  const int rank = G > 1 ? static_cast<int>(cluster_ctarank()) : 0;
  const int row = blockIdx.x / G;
  const int pl = a.p2 / G;             // m-blocks per CTA
  const int chunk = pl * a.m;          // values per CTA
  const int base = rank * chunk;
  pdl_launch_dependents();
  pdl_wait();   // the row may be the previous kernel's output
  const uint16_t* src = a.in + static_cast<size_t>(row) * a.in_stride + base;
  const bool sgn_in = a.signs_first && a.signs;
  if ((chunk & 7) == 0 && (a.in_stride & 7) == 0) {   // 16-byte loads of 8 values
    for (int i8 = threadIdx.x; i8 < chunk / 8; i8 += kRThreads) {
      const uint4 w = ldg_v4(src + 8 * i8);
      const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        float v = (k & 1) ? bf16_hi(ws[k >> 1]) : bf16_lo(ws[k >> 1]);
        if (sgn_in && a.signs[base + 8 * i8 + k]) v = -v;
        buf[8 * i8 + k] = v;
      }
    }
  } else {
    for (int i = threadIdx.x; i < chunk; i += kRThreads) {
      float v = bf16_to_f32(src[i]);
      if (sgn_in && a.signs[base + i]) v = -v;
      buf[i] = v;
    }
  }
  __syncthreads();
  if (a.m > 1) {
    float* out2 = smem_f + chunk;
    if (a.m == 12) paley_blocks<12>(buf, out2, pl, a.hm_neg);
    else if (a.m == 20) paley_blocks<20>(buf, out2, pl, a.hm_neg);
    else if (a.m == 28) paley_blocks<28>(buf, out2, pl, a.hm_neg);
    else paley344_blocks(buf, out2, pl, a.h344_neg);
    buf = out2;
    __syncthreads();
  }
  int lg = 0;
  while ((1 << lg) < pl) ++lg;
  for (int s0 = 0; s0 < lg;) {
    const int r = min(3, lg - s0);
    if (r == 3) sylvester_pass<3>(buf, pl, a.m, s0);
    else if (r == 2) sylvester_pass<2>(buf, pl, a.m, s0);
    else sylvester_pass<1>(buf, pl, a.m, s0);
    s0 += r;
    __syncthreads();
  }
  uint16_t* dst = a.out + static_cast<size_t>(row) * a.out_stride;
  if (G == 1) {
    for (int i = threadIdx.x; i < chunk; i += kRThreads) {
      float v = buf[i] * a.scale;
      if (!a.signs_first && a.signs && a.signs[i]) v = -v;
      dst[i] = f32_to_bf16_rn(v);
    }
    return;
  }
  cluster_sync();   // every chunk is transformed locally
  // CTA `rank` finishes positions [rank span, (rank + 1) span) of all G chunks
  const int span = (chunk + G - 1) / G;
  const int e1 = min(chunk, (rank + 1) * span);
  for (int e = rank * span + static_cast<int>(threadIdx.x); e < e1; e += kRThreads) {
    if (G == 16) cross_chunk<16>(a, buf, dst, chunk, e);
    else if (G == 8) cross_chunk<8>(a, buf, dst, chunk, e);
    else if (G == 4) cross_chunk<4>(a, buf, dst, chunk, e);
    else cross_chunk<2>(a, buf, dst, chunk, e);
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

// Column masks of the Paley I matrix of order 344: H = I + [[0, 1^T], [-1, Q]],
// Q[i][j] = chi(e_j - e_i) (row and column 0 the point at infinity, row i >= 1
// the field element i - 1).
std::vector<uint32_t> h344_column_masks() {
  std::vector<int> chi(343);
  for (int e = 0; e < 343; ++e) chi[e] = f343_chi(e);
  std::vector<uint32_t> masks(static_cast<size_t>(kP344) * kP344Words, 0u);
  for (int c = 0; c < kP344; ++c)
    for (int q = 0; q < kP344; ++q) {
      int h;
      if (q == c) h = 1;
      else if (q == 0) h = 1;
      else if (c == 0) h = -1;
      else h = chi[f343_sub(c - 1, q - 1)];
      if (h < 0) masks[static_cast<size_t>(c) * kP344Words + q / 32] |= 1u << (q % 32);
    }
  return masks;
}

std::atomic<const uint32_t*> g_h344_addr[64];
std::mutex g_h344_mu;

// Device address of g_h344_neg on device `dev`, written from the host on the
// first request (a synchronous copy, so it must not run under stream capture).
const uint32_t* h344_table(int dev) {
  const uint32_t* t = g_h344_addr[dev].load(std::memory_order_acquire);
  if (t) return t;
  std::lock_guard<std::mutex> lk(g_h344_mu);
  t = g_h344_addr[dev].load(std::memory_order_acquire);
  if (t) return t;
  static const std::vector<uint32_t> host = h344_column_masks();
  void* addr = nullptr;
  if (cudaMemcpyToSymbol(g_h344_neg, host.data(), host.size() * sizeof(uint32_t)) != cudaSuccess ||
      cudaGetSymbolAddress(&addr, g_h344_neg) != cudaSuccess)
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
// For m = 344 (11008 = 32 * 344), 16 CTAs hold two blocks each: the dense
// block product is most of the work there.
static int rht_ctas(int n, int p2, int m) {
  if ((n >= 16384 || m == kP344) && p2 >= 16) return 16;
  return p2 >= 8 ? 8 : p2;
}

size_t rht_smem_bytes(int n) {
  int p2 = 0, m = 0;
  if (!rht_factor(n, &p2, &m)) return static_cast<size_t>(n) * sizeof(float);
  return static_cast<size_t>(n / rht_ctas(n, p2, m)) * sizeof(float) * (m > 1 ? 2 : 1);
}

unisvq_status launch_rht(const void* in, int in_stride, void* out, int out_stride, int M, int n,
                         const uint8_t* signs, int signs_first, cudaStream_t s) {
  int p2 = 0, m = 0;
  if (!rht_factor(n, &p2, &m)) return UNISVQ_ERR_UNSUPPORTED;
  if (rht_smem_bytes(n) > 227 * 1024) return UNISVQ_ERR_UNSUPPORTED;
  if (M <= 0) return UNISVQ_OK;
  static bool attr_set[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return UNISVQ_ERR_CUDA;
  if (!attr_set[dev]) {
    if (cudaFuncSetAttribute(rht_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess ||
        cudaFuncSetAttribute(rht_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024) != cudaSuccess)
      return UNISVQ_ERR_CUDA;
    attr_set[dev] = true;
  }
  RhtArgs a{};
  a.in = static_cast<const uint16_t*>(in);
  a.out = static_cast<uint16_t*>(out);
  a.signs = signs;
  a.n = n;
  a.p2 = p2;
  a.m = m;
  a.G = rht_ctas(n, p2, m);
  a.in_stride = in_stride;
  a.out_stride = out_stride;
  a.signs_first = signs_first;
  a.scale = static_cast<float>(1.0 / std::sqrt(static_cast<double>(n)));
  if (m == kP344) {
    a.h344_neg = h344_table(dev);
    if (!a.h344_neg) return UNISVQ_ERR_CUDA;
  } else if (m > 1) {
    const std::vector<int> H = paley_signs(m);
    for (int c = 0; c < m; ++c) {
      uint32_t mask = 0;
      for (int q = 0; q < m; ++q)
        if (H[static_cast<size_t>(q) * m + c] < 0) mask |= 1u << q;
      a.hm_neg[c] = mask;
    }
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(M * a.G, 1, 1);
  cfg.blockDim = dim3(kRThreads, 1, 1);
  cfg.dynamicSmemBytes = rht_smem_bytes(n);
  cfg.stream = s;
  cudaLaunchAttribute attrs[2];
  attrs[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attrs[0].val.programmaticStreamSerializationAllowed = 1;
  attrs[1].id = cudaLaunchAttributeClusterDimension;
  attrs[1].val.clusterDim.x = a.G;
  attrs[1].val.clusterDim.y = 1;
  attrs[1].val.clusterDim.z = 1;
  cfg.attrs = attrs;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, rht_kernel, a) == cudaSuccess ? UNISVQ_OK : UNISVQ_ERR_CUDA;
}

}  // namespace unisvq
