// Packed code layout shared by the host packer and the device kernels.
//
// A 16-row x 128-column tile is 512 bytes; lane l of a warp owns 16 bytes =
// four 32-bit words. Word q (grp = q/2, rh = q%2) of lane l (g = l/4, t = l%4)
// holds row 16*rt + g + 8*rh and, at position p (i = p/2, h = p%2), columns
//   k = 128*kt + 64*grp + 16*i + 4*t + 2*h   in bits [2p+1:2p]
//   k + 1                                      in bits [16+2p+1:16+2p].
//
// Why this order: it is the A-operand fragment order of the m16n8k16 tensor
// core MMA after a fixed permutation of the 16 columns of each k16 block
// (MMA k-slot 2t+e <-> column 4t+e, slot 2t+8+e <-> column 4t+2+e), so
// (word & (0x00030003 << 2p)) IS an fp16x2 A-fragment register: two fp16
// subnormals of value z * 4^p * 2^-24, without shifting (positions 0..4), or
// after one shift right by 10 (positions 5..7). The activation side carries the
// 4^-s scale. Four consecutive columns 4m..4m+3 always share one word, so
// vectors of d = 1, 2, 4 are never split.
#pragma once

#include <cstdint>

#ifdef __CUDACC__
#define UNISVQ_HD __host__ __device__ __forceinline__
#else
#define UNISVQ_HD inline
#endif

namespace unisvq {

constexpr int kTileRows = 16;
constexpr int kTileCols = 128;
constexpr int kTileBytes = 512;
constexpr int kRowPad = 128;   // Np is a multiple of this
constexpr int kColPad = 128;   // Kp is a multiple of this

UNISVQ_HD int round_up(int v, int m) { return (v + m - 1) / m * m; }

// Scale class s of word position p: the fp16 subnormal extracted from
// position p encodes z * 4^s * 2^-24.
UNISVQ_HD int pos_scale_class(int p) { return p < 5 ? p : p - 5; }

// Word position p holding column kk (kk = column index within a 128-col tile,
// kk % 2 == 0 selects the low half, 1 the high half).
UNISVQ_HD int col_position(int kk) { return 2 * ((kk & 63) >> 4) + ((kk & 3) >> 1); }
UNISVQ_HD int col_lane_t(int kk) { return (kk & 15) >> 2; }
UNISVQ_HD int col_grp(int kk) { return kk >> 6; }

// Scale class of column k (any k; depends on k % 64 only).
UNISVQ_HD int col_scale_class(int k) { return pos_scale_class(col_position(k & 127)); }

// Extract the fp16x2 A-fragment register of position p from a code word:
// two fp16 subnormals (z_lo * 4^s * 2^-24, z_hi * 4^s * 2^-24), s = class(p).
UNISVQ_HD uint32_t extract_pos(uint32_t w, uint32_t w_shr10, int p) {
  return p < 5 ? (w & (0x00030003u << (2 * p))) : (w_shr10 & (0x00030003u << (2 * (p - 5))));
}

// Code pair (z_lo, z_hi) of position p recovered from its fragment register.
UNISVQ_HD uint32_t frag_code_lo(uint32_t frag, int p) { return (frag >> (2 * pos_scale_class(p))) & 3u; }
UNISVQ_HD uint32_t frag_code_hi(uint32_t frag, int p) { return (frag >> (16 + 2 * pos_scale_class(p))) & 3u; }

}  // namespace unisvq
