// Packed code layout shared by the host packer and the device kernels.
//
// The matrix is padded to Np = roundup(N, 128) rows and Kp = roundup(K, 128)
// columns (code 0) and cut into tiles of 128 rows x 128 columns, 4096 bytes
// each; tile (rb, kt) starts at byte (rb * Kp/128 + kt) * 4096, so the tiles
// of one 128-row block are consecutive along K (one bulk copy per k-tile).
//
// Inside a tile: half h (columns 64h .. 64h+63) occupies bytes [2048h, 2048h+2048);
// row r of that half owns the 16 bytes at 2048h + 16r: four little-endian
// words w0..w3, word wi holding columns 64h + 16wi + 4s + b (s, b in 0..3) in
// bits [8b + 2s + 1 : 8b + 2s].
//
// Why: (w >> 2s) & 0x03030303 gives four bytes, one per column 4s+b, each the
// code z in its two low bits -- exactly the e4m3 subnormal z * 2^-9 -- in the
// byte order of the tensor-memory A operand of an 8-bit MMA (TMEM lane = row,
// column j byte b = element 4j + b). One shift and one AND expand 4 weights.
// Four consecutive columns 4m .. 4m+3 share those four bytes, so vectors of
// d = 1, 2 or 4 never straddle words, and the byte-wise code of a d = 4 vector
// reads off as the index z0 | z1 << 2 | z2 << 4 | z3 << 6.
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
constexpr int kHalfBytes = 2048;
constexpr int kRowPad = 128;   // Np is a multiple of this
constexpr int kColPad = 128;   // Kp is a multiple of this

UNISVQ_HD int round_up(int v, int m) { return (v + m - 1) / m * m; }

// Byte offset, inside a tile, of the 16-byte row chunk holding (row r, half h).
UNISVQ_HD int tile_row_offset(int r, int h) { return h * kHalfBytes + r * 16; }

// Four codes of columns 16*wi + 4s + (0..3) of a word, one per byte (low 2 bits).
UNISVQ_HD uint32_t extract4(uint32_t w, int s) { return (w >> (2 * s)) & 0x03030303u; }

// Code of column c (0..15 within the word's 16 columns) of word w.
UNISVQ_HD uint32_t code_at(uint32_t w, int c) { return (w >> (8 * (c & 3) + 2 * (c >> 2))) & 3u; }

}  // namespace unisvq
