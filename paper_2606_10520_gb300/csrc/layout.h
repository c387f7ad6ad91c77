// Packed code layout shared by the host packer and the device kernels.
//
// The matrix is padded to Np = roundup(N, 128) rows and Kp = roundup(K, 128)
// columns (code 0) and cut into tiles of 128 rows x 128 columns, 4096 bytes
// each; tile (rb, kt) starts at byte (rb * Kp/128 + kt) * 4096, so the tiles
// of one 128-row block are consecutive along K (one bulk copy per k-tile).
//
// Inside a tile the rows form eight units of 16 (u = r / 16); unit u fills
// bytes [512u, 512u + 512). Within a unit, row r = 16u + 8q + g (g in 0..7,
// q in 0..1) and column quarter t (0..3) of half h (columns 64h .. 64h+63)
// share a 16-byte chunk with the row eight below or above it:
//   chunk (g, t) at 512u + 16 (4g + t), word 2h + q of the chunk
// and each little-endian word holds the 16 columns 64h + 16t + 4s + b
// (s, b in 0..3) in bits [8b + 2s + 1 : 8b + 2s].
//
// Why: (w >> 2s) & 0x03030303 gives four bytes, one per column 4s+b, each the
// code z in its two low bits (the e4m3 subnormal z * 2^-9, an 8-bit tensor
// operand); (w >> 8k) & (0x00030003 << 2s) gives two codes as fp16 subnormals
// z * 4^s * 2^-24 (a 16-bit tensor operand). Lane 4g + t of a warp reading a
// unit with one 16-byte load receives the words of rows g and g + 8 and column
// quarter t of both halves -- the rows and k-slots that thread owns in an
// m16n8k16 A fragment and in a 16x256b tensor-memory store -- and the 32 lanes
// read 512 contiguous bytes. Four consecutive columns 4m .. 4m+3 share the same
// four bytes of one word, so vectors of d = 1, 2 or 4 never straddle words,
// and the byte-wise code of a d = 4 vector reads off as the index
// z0 | z1 << 2 | z2 << 4 | z3 << 6.
#pragma once

#include <cstdint>

#ifdef __CUDACC__
#define UNISVQ_HD __host__ __device__ __forceinline__
#else
#define UNISVQ_HD inline
#endif

namespace unisvq {

constexpr int kTileRows = 128;
constexpr int kTileCols = 128;
constexpr int kTileBytes = 4096;
constexpr int kUnitRows = 16;
constexpr int kUnitBytes = 512;
constexpr int kRowPad = 128;   // Np is a multiple of this
constexpr int kColPad = 128;   // Kp is a multiple of this

UNISVQ_HD int round_up(int v, int m) { return (v + m - 1) / m * m; }

// Byte offset, inside a tile, of the word holding row r, half h, quarter t.
UNISVQ_HD int tile_word_offset(int r, int h, int t) {
  return (r >> 4) * kUnitBytes + ((r & 7) * 4 + t) * 16 + (2 * h + ((r >> 3) & 1)) * 4;
}

// Four codes of columns 16t + 4s + (0..3) of a word, one per byte (low 2 bits).
UNISVQ_HD uint32_t extract4(uint32_t w, int s) { return (w >> (2 * s)) & 0x03030303u; }

// Code of column c (0..15 within the word's 16 columns) of word w.
UNISVQ_HD uint32_t code_at(uint32_t w, int c) { return (w >> (8 * (c & 3) + 2 * (c >> 2))) & 3u; }

}  // namespace unisvq
