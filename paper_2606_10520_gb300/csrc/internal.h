// Internal declarations shared by the libunisvq translation units.
#pragma once

#include <cstddef>
#include <cstdint>
#include <vector>
#include <cuda_runtime.h>

#include "unisvq.h"
#include "layout.h"

struct unisvq_layer {
  int N, K, d;
  int Np, Kp, KT;          // padded shape; KT = Kp / 128 k-tiles
  int device;
  int num_sms;
  uint8_t* codes;          // device, packed layout (layout.h)
  size_t code_bytes;
  float* lut32;            // device, [4^d][d] fp32 codewords RN(A z + B)
  uint32_t* tlut;          // device, prefill codeword table (bf16 pairs / quads), see pack
  int tlut_words;
  int lut_entries;         // 4^d
  float A[64];             // fp32 (exact) copy of A, row-major d x d (d <= 8)
  float B[8];              // fp32 (exact) copy of B
  float colnorm;           // max_c sum_r |A[r][c]|: |x A|_inf <= |x|_inf * colnorm
  uint8_t* fold_ws;        // device, decode fold workspace (fold_workspace_bytes(KT))
  uint16_t A16[64], B16[8];
  // Per-(row, 128-column group) affine maps (unisvq_pack_grouped): the codes
  // are packed with pack_codes_grouped_host and the maps live in `meta`;
  // A, B, lut32, tlut and fold_ws are unused (zero / null).
  // Code width: 2, or 3 (unisvq_pack_bits). A 3-bit code z = z_lo + 4 z_hi
  // keeps z_lo in `codes` and z_hi in the bit plane `hi` (hi_plane_offset).
  int bits;
  uint8_t* hi;             // device, Np*Kp/8 bytes (bits == 3), else null
  size_t hi_bytes;
  int grouped;
  uint16_t* meta;          // device, fp16 [Np/128][KT][128][d*d + d]
  size_t meta_bytes;
  // Inverse randomized Hadamard transform around the layer (unisvq_set_rht):
  // device signs [K] (S_V) then [N] (S_U), 1 = -1, and a bf16 [rht_tokens][K]
  // buffer for the rotated activations.
  int rht;
  uint8_t* rht_signs;
  uint16_t* rht_x;
  int rht_tokens;
  std::vector<uint8_t> rht_in_host;   // host copy of S_V: layers of a grouped call that share it rotate x once
};

namespace unisvq {

struct DecodePlan {
  int nt;          // token tile (gemv: n8 tiles 1..2; skinny: MMA N 16/32/64)
  int ks;          // CTAs along K (cluster size)
  int kt_per_cta;  // k-tiles per CTA
  int nb;          // row blocks of 128 rows
  size_t smem;     // dynamic shared memory bytes
  int geom;        // skinny: k-tiles per pipeline stage (1 or 2)
};

// Streaming decode GEMV (stream.cu): one launch per call, no cluster, at most
// one CTA per SM, kStreamMaxTok tokens per launch.
constexpr int kStreamMaxTok = 8;
struct StreamPlan {
  bool ok;
  int ucta;         // most 16-row units of a CTA
  int ctas;         // grid (one CTA per SM at most)
  int WU, WK;       // warp grid: unit groups x k-groups
  int uw;           // accumulator slots per warp (2, 4 or 8)
  int mt;           // token slots of the fold buffers (1, 2, 4 or 8)
  int ck;           // k-tiles per fold chunk
  int sk;           // k-tiles per code stage
  int nslots;       // code stages resident in shared memory
  int stage_bytes;  // ucta * sk * 512
  int off_b, off_ptab, off_bars, off_tok;
  size_t smem;
};

struct PrefillPlan {
  int bn;          // tokens per tile
  int tiles;
  int grid;
  size_t smem;
};

int* device_error_word();   // device address of the library error word (current device)

// Register-operand tensor-core GEMV (gemv.cu), M <= 32 per launch.
DecodePlan plan_gemv(const unisvq_layer* L, int M);
unisvq_status launch_gemv(const unisvq_layer* L, const void* x, void* y, int M, cudaStream_t s);
// Row-slice GEMV (whole K per CTA, no cluster), M <= 4 per launch.
bool gemv_rows_supported(const unisvq_layer* L, int M);
unisvq_status launch_gemv_rows_group(const unisvq_layer* const* Ls, int n, const void* x, void* const* ys, int M,
                                     cudaStream_t s);
// Several layers with the same K that read the same x, in one launch per 32 tokens.
unisvq_status launch_gemv_group(const unisvq_layer* const* Ls, int n, const void* x, void* const* ys, int M,
                                cudaStream_t s);
// tcgen05 skinny GEMM with the codes as 8-bit TMEM operand (decode.cu), M <= 16 per launch.
// The plan of the call's launch pairs and their tokens per launch (32 where
// one 32-token launch at one CTA per SM takes fewer waves of the call's row
// blocks than two 16-token launches at two per SM, else 16).
DecodePlan plan_skinny(const unisvq_layer* const* Ls, int n, int M);
int skinny_tokens_per_launch(const unisvq_layer* const* Ls, int n);
unisvq_status launch_skinny(const unisvq_layer* L, const void* x, void* y, int M, cudaStream_t s);
// Device bytes of a handle's fold workspace for the skinny decode kernel.
size_t fold_workspace_bytes(int KT);
// Several layers with the same K that read the same x, in one launch pair per 32 tokens.
unisvq_status launch_skinny_group(const unisvq_layer* const* Ls, int n, const void* x, void* const* ys, int M,
                                  cudaStream_t s);
// The same with the input rotation of the inverse RHT, x -> (x S_V) H_K /
// sqrt(K), done by the fold kernel (rht_sv: S_V sign bytes on the device,
// 8-byte aligned). Possible where skinny_rht_foldable holds: K = 2^a m with
// m in {1, 12, 20, 28}; the launches then split K into KS full slices, KS the
// largest power of 2 up to the usual split that divides both K / 128 and
// 2^a, at least 2, each slice's bf16 and two fp32 copies within the fold
// kernel's shared memory.
bool skinny_rht_foldable(const unisvq_layer* const* Ls, int n, int M);
unisvq_status launch_skinny_group_rht(const unisvq_layer* const* Ls, int n, const void* x, void* const* ys, int M,
                                      const uint8_t* rht_sv, cudaStream_t s);
// As launch_skinny with the fold workspace in a static device array of
// static_fold_workspace_bytes() (UNSUPPORTED if the layer needs more).
unisvq_status launch_skinny_static(const unisvq_layer* L, const void* x, void* y, int M, cudaStream_t s);
size_t static_fold_workspace_bytes();

// Layers of one call (same K, 2-bit, per-matrix maps, d <= 4) in one
// streaming launch per kStreamMaxTok tokens.
StreamPlan plan_stream(const unisvq_layer* const* Ls, int n, int M);
bool stream_supported(const unisvq_layer* const* Ls, int n, int M);
unisvq_status launch_stream_group(const unisvq_layer* const* Ls, int n, const void* x, void* const* ys, int M,
                                  cudaStream_t s);

bool prefill_supported(const unisvq_layer* L, int M);
PrefillPlan plan_prefill(const unisvq_layer* L, int M);
unisvq_status launch_prefill(const unisvq_layer* L, const void* x, void* y, int M, cudaStream_t s);
// Several layers that read the same x in one persistent launch (their tiles
// one after the other): 2-bit layers with one d <= 4 and one K, all
// per-matrix or all per-group.
bool prefill_group_supported(const unisvq_layer* const* Ls, int n, int M);
PrefillPlan plan_prefill_group(const unisvq_layer* const* Ls, int n, int M);
unisvq_status launch_prefill_group(const unisvq_layer* const* Ls, int n, const void* x, void* const* ys, int M,
                                   cudaStream_t s);

unisvq_status launch_dequant(const unisvq_layer* L, float* W, cudaStream_t s);
// The bounded-wait test hook (dequant.cu): src16 device, 16 bytes, 16-byte
// aligned; out3 device, three ints.
unisvq_status launch_wait_probe(const void* src16, int* out3, cudaStream_t s);

// Randomized Hadamard transform of M rows of n bf16 values (rht.cu):
// signs_first = 1: out = (s x) H / sqrt(n); 0: out = s ((x H) / sqrt(n)).
// n = 2^a m, m in {1, 12, 20, 28, 344}; in and out may be the same rows.
// rht_prepare(n) writes the device's H_344 sign table when n needs it (a
// synchronous copy, made once per device): call it outside stream capture
// before the first launch_rht of such an n.
bool rht_factor(int n, int* p2, int* m);
unisvq_status rht_prepare(int n);
// Column sign masks of H_m for m in {12, 20, 28}: 28 words, bit q of word c
// set where H_m[q][c] = -1.
const uint32_t* rht_paley_masks(int m);
size_t rht_smem_bytes(int n);
// signs_const: the sign bytes never change between launches (a handle's own
// buffer), so the kernel reads them before waiting for the previous kernel.
unisvq_status launch_rht(const void* in, int in_stride, void* out, int out_stride, int M, int n,
                         const uint8_t* signs, int signs_first, bool signs_const, cudaStream_t s);
// Several row sets (e.g. the outputs of a group call), M rows each: one
// launch when every width has the same H_m and cluster size, else one per
// set. At most UNISVQ_MAX_GROUP sets.
struct RhtSetDesc {
  const void* in;
  int in_stride;
  void* out;
  int out_stride;
  int n;
  const uint8_t* signs;
};
unisvq_status launch_rht_sets(const RhtSetDesc* sets, int nsets, int M, int signs_first, bool signs_const,
                              cudaStream_t s);
// Launches launch_rht_sets makes for row sets of these widths (1 or nsets).
int rht_set_launches(const int* ns, int nsets);

// Per-(row, group) affine layers (gemv_grouped.cu): every M, at most 32 / d
// tokens per launch; all layers of one call must be grouped with the same d.
unisvq_status launch_grouped_group(const unisvq_layer* const* Ls, int n, const void* x, void* const* ys, int M,
                                   cudaStream_t s);
// Plan of the first launch for nb row blocks (the layers of one call) and M
// tokens; *tokens_per_launch receives the tokens each launch takes (0: none fits).
DecodePlan plan_grouped(const unisvq_layer* L, int nb, int M, int* tokens_per_launch);

// Host packer (pack.cpp).
void pack_codes_host(const uint8_t* codes, int N, int K, uint8_t* packed);
// High-bit plane of 3-bit codes: for the 16-byte chunk (unit u, lane 4g + t)
// of tile (rb, kt), four halfwords at 2048 (rb KT + kt) + 256 u + 8 (4g + t);
// halfword i belongs to word i of the chunk, and its bit 4b + s is bit 2 of
// the code whose low bits sit at bits [8b + 2s + 1 : 8b + 2s] of that word.
void pack_hi_plane_host(const uint8_t* codes, int N, int K, uint8_t* hi);
// Same layout with the columns of every 128-column group permuted by
// grouped_column (per-group layers), and their fp16 metadata.
int grouped_column(int d, int h, int t, int s, int b);
void pack_codes_grouped_host(const uint8_t* codes, int N, int K, int d, uint8_t* packed);
void pack_meta_grouped_host(const uint16_t* A_f16, const uint16_t* B_f16, int N, int K, int d, uint16_t* meta);
// fp64 -> bf16 round-to-nearest-even (single rounding).
uint16_t f64_to_bf16_rne(double v);
// The prefill GEMM's table of a per-matrix layer (A row-major d x d, B; fp64).
std::vector<uint32_t> prefill_table_host(const double* A, const double* B, int d, int bits);
double f16_bits_to_f64(uint16_t h);

}  // namespace unisvq
