// Host packer: canonical codes [N][K] -> packed device layout (layout.h), plus
// the exact codebook of Eq. (def:unisvq) used by the tile-dequantising GEMM
// and the debug hook.
#include <cmath>
#include <cstdint>
#include <cstring>

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

}  // namespace unisvq
