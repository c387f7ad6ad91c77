// Host packer: canonical codes [N][K] -> packed device layout (layout.h), plus
// the exact codebook of Eq. (def:unisvq) used by the tile-dequantising GEMM
// and the debug hook.
#include <cmath>
#include <cstdint>
#include <cstring>
#include <vector>

#include "internal.h"

namespace unisvq {

void pack_codes_host(const uint8_t* codes, int N, int K, uint8_t* packed) {
  const int Np = round_up(N, kRowPad), Kp = round_up(K, kColPad);
  const int RB = Np / kTileRows, KT = Kp / kTileCols;
#pragma omp parallel for schedule(static)
  for (int rb = 0; rb < RB; ++rb) {
    for (int kt = 0; kt < KT; ++kt) {
      uint8_t* tile = packed + (static_cast<size_t>(rb) * KT + kt) * kTileBytes;
      for (int r = 0; r < kTileRows; ++r) {
        const int row = rb * kTileRows + r;
        const uint8_t* cr = row < N ? codes + static_cast<size_t>(row) * K : nullptr;
        for (int h = 0; h < 2; ++h) {
          for (int t = 0; t < 4; ++t) {
            uint32_t w = 0;
            for (int s = 0; s < 4; ++s)
              for (int b = 0; b < 4; ++b) {
                const int k = kt * kTileCols + 64 * h + 16 * t + 4 * s + b;
                const uint32_t z = (cr && k < K) ? (cr[k] & 3u) : 0u;
                w |= z << (8 * b + 2 * s);
              }
            uint8_t* dst = tile + tile_word_offset(r, h, t);
            dst[0] = static_cast<uint8_t>(w);
            dst[1] = static_cast<uint8_t>(w >> 8);
            dst[2] = static_cast<uint8_t>(w >> 16);
            dst[3] = static_cast<uint8_t>(w >> 24);
          }
        }
      }
    }
  }
}

void pack_hi_plane_host(const uint8_t* codes, int N, int K, uint8_t* hi) {
  const int Np = round_up(N, kRowPad), Kp = round_up(K, kColPad);
  const int RB = Np / kTileRows, KT = Kp / kTileCols;
#pragma omp parallel for schedule(static)
  for (int rb = 0; rb < RB; ++rb) {
    for (int kt = 0; kt < KT; ++kt) {
      uint8_t* tile = hi + (static_cast<size_t>(rb) * KT + kt) * (kTileBytes / 2);
      for (int r = 0; r < kTileRows; ++r) {
        const int row = rb * kTileRows + r;
        const uint8_t* cr = row < N ? codes + static_cast<size_t>(row) * K : nullptr;
        const int u = r >> 4, q = (r >> 3) & 1, g = r & 7;
        for (int h = 0; h < 2; ++h)
          for (int t = 0; t < 4; ++t) {
            uint32_t hw = 0;
            for (int s = 0; s < 4; ++s)
              for (int b = 0; b < 4; ++b) {
                const int k = kt * kTileCols + 64 * h + 16 * t + 4 * s + b;
                const uint32_t z = (cr && k < K) ? cr[k] : 0u;
                hw |= ((z >> 2) & 1u) << (4 * b + s);
              }
            uint8_t* dst = tile + u * (kUnitBytes / 2) + (4 * g + t) * 8 + 2 * (2 * h + q);
            dst[0] = static_cast<uint8_t>(hw);
            dst[1] = static_cast<uint8_t>(hw >> 8);
          }
      }
    }
  }
}

// Column, inside its 128-column group, whose code sits at packed position
// (half h, quarter t, shift s, byte b) of a per-group layer: chunk q = 4h + s
// holds coordinate c = q / (8/d) of vectors 16 (q mod 8/d) + 4t + e with
// e = (b >> 1) | ((b & 1) << 1), so that every 16-column chunk of an MMA A
// fragment carries a single coordinate (gemv_grouped.cu).
int grouped_column(int d, int h, int t, int s, int b) {
  const int nq = 8 / d, q = 4 * h + s;
  const int e = (b >> 1) | ((b & 1) << 1);
  const int v = 16 * (q % nq) + 4 * t + e;
  return v * d + q / nq;
}

void pack_codes_grouped_host(const uint8_t* codes, int N, int K, int d, uint8_t* packed) {
  const int Np = round_up(N, kRowPad), Kp = round_up(K, kColPad);
  const int RB = Np / kTileRows, KT = Kp / kTileCols;
  int col[2][4][4][4];
  for (int h = 0; h < 2; ++h)
    for (int t = 0; t < 4; ++t)
      for (int s = 0; s < 4; ++s)
        for (int b = 0; b < 4; ++b) col[h][t][s][b] = grouped_column(d, h, t, s, b);
#pragma omp parallel for schedule(static)
  for (int rb = 0; rb < RB; ++rb) {
    for (int kt = 0; kt < KT; ++kt) {
      uint8_t* tile = packed + (static_cast<size_t>(rb) * KT + kt) * kTileBytes;
      for (int r = 0; r < kTileRows; ++r) {
        const int row = rb * kTileRows + r;
        const uint8_t* cr = row < N ? codes + static_cast<size_t>(row) * K : nullptr;
        for (int h = 0; h < 2; ++h) {
          for (int t = 0; t < 4; ++t) {
            uint32_t w = 0;
            for (int s = 0; s < 4; ++s)
              for (int b = 0; b < 4; ++b) {
                const int k = kt * kTileCols + col[h][t][s][b];
                const uint32_t z = (cr && k < K) ? (cr[k] & 3u) : 0u;
                w |= z << (8 * b + 2 * s);
              }
            uint8_t* dst = tile + tile_word_offset(r, h, t);
            dst[0] = static_cast<uint8_t>(w);
            dst[1] = static_cast<uint8_t>(w >> 8);
            dst[2] = static_cast<uint8_t>(w >> 16);
            dst[3] = static_cast<uint8_t>(w >> 24);
          }
        }
      }
    }
  }
}

// Per-group metadata: fp16 [Np/128][KT][128][d*d + d], A[n][g] row-major then
// B[n][g]; zero for padding rows.
void pack_meta_grouped_host(const uint16_t* A_f16, const uint16_t* B_f16, int N, int K, int d, uint16_t* meta) {
  const int Np = round_up(N, kRowPad), KT = round_up(K, kColPad) / kTileCols;
  const int G = (K + kTileCols - 1) / kTileCols;   // = KT
  const int MD = d * d + d;
#pragma omp parallel for schedule(static)
  for (int n = 0; n < Np; ++n) {
    const int rb = n / kTileRows, r = n % kTileRows;
    for (int kt = 0; kt < KT; ++kt) {
      uint16_t* rec = meta + ((static_cast<size_t>(rb) * KT + kt) * kTileRows + r) * MD;
      for (int i = 0; i < MD; ++i) rec[i] = 0;
      if (n >= N || kt >= G) continue;
      const size_t ng = static_cast<size_t>(n) * G + kt;
      for (int i = 0; i < d * d; ++i) rec[i] = A_f16[ng * d * d + i];
      for (int i = 0; i < d; ++i) rec[d * d + i] = B_f16[ng * d + i];
    }
  }
}

double f16_bits_to_f64(uint16_t h) {
  const int sign = (h >> 15) & 1;
  const int e = (h >> 10) & 31;
  const int m = h & 1023;
  double v;
  if (e == 0) v = std::ldexp(static_cast<double>(m), -24);
  else if (e == 31) v = m ? NAN : INFINITY;
  else v = std::ldexp(static_cast<double>(1024 + m), e - 25);
  return sign ? -v : v;
}

// Correct RN-even of a double to bf16. RN to fp32 first is exact-or-single
// rounding; the only double-rounding case is an fp32 result sitting exactly on
// a bf16 tie while the double is not, which is resolved toward the double.
uint16_t f64_to_bf16_rne(double v) {
  if (std::isnan(v)) return 0x7FC0;
  const float f = static_cast<float>(v);
  uint32_t u;
  std::memcpy(&u, &f, 4);
  if ((u & 0x7F800000u) == 0x7F800000u) return static_cast<uint16_t>(u >> 16);   // inf
  const uint32_t low = u & 0xFFFFu;
  if (low == 0x8000u && static_cast<double>(f) != v) {
    const bool away = std::fabs(v) > std::fabs(static_cast<double>(f));
    return static_cast<uint16_t>((u >> 16) + (away ? 1u : 0u));
  }
  const uint32_t rounding = 0x7FFFu + ((u >> 16) & 1u);
  return static_cast<uint16_t>((u + rounding) >> 16);
}

// The prefill GEMM's shared-memory table of a per-matrix layer, indexed the
// way its converter warps read code bytes (unisvq_prefill_table_host in
// unisvq.h states the formats). Every entry is the exact fp64 value rounded
// once, to bf16 (whole codewords) or to fp32 (partial sums that the
// converters add).
std::vector<uint32_t> prefill_table_host(const double* A, const double* B, int d, int bits) {
  const int zmax = (1 << bits) - 1;
  // the codeword of index v (coordinate c in bits [bits (c+1) - 1 : bits c]), row r
  auto codeword = [&](int v, int r) {
    double w = B[r];
    for (int c = 0; c < d; ++c) w += A[r * d + c] * static_cast<double>((v >> (bits * c)) & zmax);
    return w;
  };
  auto bf = [](double w) { return static_cast<uint32_t>(f64_to_bf16_rne(w)); };
  auto f32 = [](double w) {
    const float f = static_cast<float>(w);
    uint32_t u;
    std::memcpy(&u, &f, sizeof(u));
    return u;
  };
  std::vector<uint32_t> t;
  if (bits == 3 && d <= 2) {   // 64 bf16 pairs, index lo | hi << 3 for columns (k, k+1)
    t.resize(64);
    for (int v = 0; v < 64; ++v) {
      const int lo = v & 7, hi = v >> 3;
      const double w0 = d == 2 ? codeword(lo | (hi << 3), 0) : codeword(lo, 0);
      const double w1 = d == 2 ? codeword(lo | (hi << 3), 1) : codeword(hi, 0);
      t[v] = bf(w0) | (bf(w1) << 16);
    }
  } else if (bits == 3 && d == 4) {
    // 8^4 codewords would take 32 KB: two pair tables, T_p[z_2p | z_2p+1 << 3][r]
    // = A[r][2p] z_2p + A[r][2p+1] z_2p+1 (+ B[r] for p = 0), 64 rows of 4 fp32
    t.resize(512);
    for (int pr = 0; pr < 2; ++pr)
      for (int v = 0; v < 64; ++v)
        for (int r = 0; r < 4; ++r)
          t[static_cast<size_t>(pr * 64 + v) * 4 + r] =
              f32(A[r * 4 + 2 * pr] * (v & 7) + A[r * 4 + 2 * pr + 1] * (v >> 3) + (pr == 0 ? B[r] : 0.0));
  } else if (bits == 2 && d == 8) {
    // 4^8 codewords do not fit: two quad tables, T_q[z_4q | .. | z_4q+3 << 6][r]
    // = sum_c A[r][4q + c] z_4q+c (+ B[r] for q = 0), 256 rows of 8 fp32; row v's
    // 16-byte halves (r = 0..3, 4..7) are swapped when bit 2 of v is set, so a
    // warp's loads of one half spread over all eight 16-byte bank groups
    t.resize(4096);
    for (int qd = 0; qd < 2; ++qd)
      for (int v = 0; v < 256; ++v)
        for (int r = 0; r < 8; ++r) {
          double w = qd == 0 ? B[r] : 0.0;
          for (int c = 0; c < 4; ++c) w += A[r * 8 + 4 * qd + c] * ((v >> (2 * c)) & 3);
          const int half = (r >> 2) ^ ((v >> 2) & 1);
          t[static_cast<size_t>(qd * 256 + v) * 8 + 4 * half + (r & 3)] = f32(w);
        }
  } else if (bits == 2 && d <= 2) {   // 16 bf16 pairs, index lo | hi << 2 for columns (k, k+1)
    t.resize(16);
    for (int v = 0; v < 16; ++v) {
      const int lo = v & 3, hi = v >> 2;
      const double w0 = d == 2 ? codeword(lo | (hi << 2), 0) : codeword(lo, 0);
      const double w1 = d == 2 ? codeword(lo | (hi << 2), 1) : codeword(hi, 0);
      t[v] = bf(w0) | (bf(w1) << 16);
    }
  } else if (bits == 2 && d == 4) {   // 256 bf16 quads, index z0 | z1 << 2 | z2 << 4 | z3 << 6
    t.resize(512);
    for (int v = 0; v < 256; ++v) {
      t[2 * v] = bf(codeword(v, 0)) | (bf(codeword(v, 1)) << 16);
      t[2 * v + 1] = bf(codeword(v, 2)) | (bf(codeword(v, 3)) << 16);
    }
  } else {   // no table (3-bit codes with d = 8 are not packed)
    t.assign(1, 0u);
  }
  return t;
}

}  // namespace unisvq
