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
