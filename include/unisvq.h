/*
 * libunisvq -- GB300 (sm_103a) inference kernels for the UniSVQ linear layer.
 *
 * The method (UniSVQ, "2-bit Unified Scalar-Vector Quantization"):
 *   - Eq. (def:unisvq), Sec. 3.1: a length-d weight vector is stored as a
 *     lattice point z in {0,1,2,3}^d and reconstructed as w = A z + B, with
 *     A a d x d matrix and B a d-vector.
 *   - Eq. (col:dequant), Sec. 3.2.3: the vectors run along the INPUT dimension
 *     of the weight matrix and one (A, B) serves the whole matrix, i.e.
 *     W_hat[n, g*d + r] = sum_c A[r][c] * z[n, g*d + c] + B[r].
 *   - Eq. (col:matmul), Sec. 3.2.3: the layer Y = X W_hat^T can be computed as
 *     sum_i (X_i A) W_int,i^T + sum_i (X_i B) 1^T without a dequantised W.
 *
 * Shapes: x [M][K] bf16 (tokens x inputs), codes [N][K] (outputs x inputs),
 * y [M][N] bf16. d in {1, 2, 4, 8}. No entry point ever writes a dequantised
 * weight matrix to device memory, except the test hook unisvq_dequant_debug.
 *
 * Streams are passed as `void*` holding a cudaStream_t (NULL = legacy default
 * stream). Device pointers are plain CUDA device addresses.
 *
 * Errors: every entry point validates its arguments before touching the GPU
 * and returns a status; nothing aborts the process. CUDA runtime failures map
 * to UNISVQ_ERR_CUDA. Kernels bound every wait; a wait that runs out sets a
 * device error word that unisvq_sync_status reports as UNISVQ_ERR_TIMEOUT.
 */
#ifndef UNISVQ_H_
#define UNISVQ_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  UNISVQ_OK = 0,
  UNISVQ_ERR_INVALID_ARG = 1,
  UNISVQ_ERR_UNSUPPORTED = 2,
  UNISVQ_ERR_CUDA = 3,
  UNISVQ_ERR_OOM = 4,
  UNISVQ_ERR_TIMEOUT = 5
} unisvq_status;

/* Kernel selectors for unisvq_linear_force and unisvq_info.kernel. */
enum {
  UNISVQ_KERNEL_AUTO = 0,     /* pick by M (unisvq_linear does this)                   */
  UNISVQ_KERNEL_DECODE = 1,   /* the decode kernel auto would pick for this M (a GEMV)  */
  UNISVQ_KERNEL_PREFILL = 2,  /* tcgen05 GEMM, bf16 weight tiles in smem (exact codewords for d <= 4) */
  UNISVQ_KERNEL_GEMV = 3,     /* fold + register-operand tensor-core GEMV, M <= 32/launch */
  UNISVQ_KERNEL_SKINNY = 4,   /* fold + tcgen05 with codes as 8-bit TMEM operand, M <= 32/launch */
  UNISVQ_KERNEL_GEMV_ROWS = 5, /* GEMV with whole-K row slices per CTA (no cluster), M <= 4/launch */
  UNISVQ_KERNEL_GROUPED = 6,   /* per-(row, group) affine GEMV (layers of unisvq_pack_grouped), M <= 32/d per launch */
  UNISVQ_KERNEL_STREAM = 7     /* streaming GEMV: one launch per call, codes prefetched before the previous
                                  kernel ends, whole K per CTA, no cluster; 2-bit per-matrix d <= 4, M <= 8/launch */
};

/*
 * Packed device layout of the codes (written by unisvq_pack, documented so
 * that other tools can produce or check it).
 *
 * The matrix is padded to Np = roundup(N, 128) rows and Kp = roundup(K, 128)
 * columns with code 0 and cut into tiles of 128 rows x 128 columns, 4096
 * bytes each. Tile (rb, kt), rb < Np/128, kt < Kp/128, starts at byte
 * (rb * (Kp/128) + kt) * 4096, so the tiles of one 128-row block are
 * consecutive along K.
 *
 * Inside a tile, row r = 16u + 8q + g (unit u in 0..7, q in 0..1, g in 0..7)
 * and column quarter t (0..3) of half h (columns 64h .. 64h+63) own the
 * little-endian 32-bit word at byte
 *   512 u + 16 (4 g + t) + 4 (2 h + q),
 * so each unit of 16 rows fills 512 contiguous bytes and each 16-byte chunk
 * holds rows g and g + 8 of quarter t in both halves. The word holds the 16
 * codes of columns
 *   k = 128 kt + 64 h + 16 t + 4 s + b,   s, b in 0..3,
 * the code of column k in bits [8b+2s+1 : 8b+2s]. Shifting a word right by 2s
 * and masking with 0x03030303 yields the codes of columns 4s..4s+3 one per
 * byte; a run of 4 columns 4m..4m+3 therefore never spans two words.
 */
#define UNISVQ_TILE_ROWS 128
#define UNISVQ_TILE_COLS 128
#define UNISVQ_TILE_BYTES 4096

typedef struct unisvq_layer* unisvq_handle;

typedef struct {
  int N, K, d;            /* layer shape and vector length                      */
  int Np, Kp;             /* padded shape of the packed codes                   */
  int kernel;             /* kernel unisvq_linear runs for this M               */
  int split_k;            /* CTAs cooperating along K (decode kernel)           */
  int grid_ctas;          /* CTAs launched                                      */
  long long code_bytes;   /* packed code bytes resident on the device           */
  long long meta_bytes;   /* affine parameters: (d*d + d) * 2 bytes (fp16), times
                             N * ceil(K/128) for a unisvq_pack_grouped layer    */
  long long algo_bytes;   /* N*K/4 + meta + 2*M*K (x) + 2*M*N (y)               */
  double flops;           /* 2*M*N*K                                            */
  int launches;           /* kernel launches the call makes                     */
} unisvq_info;

/*
 * Pack a quantised weight matrix into a device-resident layer handle.
 *   codes : host, [N][K] row-major uint8, each 0..3 (lattice coordinates z)
 *   A_f16 : host, [d][d] row-major IEEE fp16 bit patterns, w = A z + B
 *   B_f16 : host, [d] fp16 bit patterns
 *   N, K  : output / input features, N >= 1, K >= d, K % d == 0
 *   d     : vector length, 1, 2, 4 or 8 (Eq. def:unisvq; the paper uses d = 4
 *           and d = 8 in its vector-length ablation, Table tab:ablation_dim).
 *           The prefill GEMM takes every d: exact bf16 codewords from a
 *           pack-time table for d <= 4, and for d = 8 the fp32 sum of two
 *           quad-table rows rounded once to bf16.
 *   stream: stream for the upload; pack synchronises it before returning
 *   out   : receives the handle
 * The host buffers are copied before return; the caller keeps ownership.
 * Errors: INVALID_ARG (null pointer, bad shape, code > 3, non-finite A/B),
 * UNSUPPORTED (d not in {1,2,4,8}), OOM, CUDA.
 * The handle owns all device memory: the packed codes, the tables of the
 * prefill kernel and a fold workspace of 2 KB + (Kp/128) * 12 KB that the
 * decode kernels rewrite on every call (the folded activations of Eq.
 * col:matmul). Calls that use the same handle must therefore be ordered on
 * the GPU (one stream, or events between streams); calls on different
 * handles may run concurrently. unisvq_clone gives a second handle with its
 * own workspace.
 */
unisvq_status unisvq_pack(const uint8_t* codes, const uint16_t* A_f16, const uint16_t* B_f16,
                          int N, int K, int d, void* stream, unisvq_handle* out);

/*
 * As unisvq_pack for codes of `bits` bits: 2, or 3 (z in {0..7}, the 3-bit
 * variant of Sec. 5.2: only the integer vectors widen, Eq. def:affine with
 * b = 3). A 3-bit code z = z_lo + 4 z_hi keeps z_lo in the packed layout
 * above and z_hi in a bit plane of Np*Kp/8 bytes: for the 16-byte chunk of
 * unit u, lane 4g + t of tile (rb, kt), four little-endian halfwords at byte
 * 2048 (rb Kp/128 + kt) + 256 u + 8 (4g + t); halfword i belongs to word i of
 * the chunk and its bit 4b + s is bit 2 of the code at bits [8b+2s+1 : 8b+2s]
 * of that word. 3-bit layers take d in {1, 2, 4} and run the GEMV
 * (UNISVQ_KERNEL_GEMV, 32 tokens per launch) up to 64 tokens; above that,
 * the prefill GEMM (also forceable): exact codewords from a 64-pair table
 * for d <= 2, and for d = 4 the fp32 sum of two 64-row pair-table rows
 * rounded once to bf16. Other forced kernels return UNSUPPORTED. Errors as
 * unisvq_pack, plus UNSUPPORTED (bits, or bits = 3 with d = 8) and
 * INVALID_ARG (a code >= 2^bits).
 */
unisvq_status unisvq_pack_bits(const uint8_t* codes, const uint16_t* A_f16, const uint16_t* B_f16,
                               int N, int K, int d, int bits, void* stream, unisvq_handle* out);

/*
 * Pack a layer whose affine map varies per output row and per group of
 * `group_cols` input columns: W_hat[n, k] = sum_c A[n][g][r][c] z[n, k - r + c]
 * + B[n][g][r], g = k / group_cols, r = k mod d (Eq. def:unisvq applied with
 * the map of the vector's row and column group). This granularity is finer
 * than the paper's (one map per matrix, Sec. 4.2: use unisvq_pack for that);
 * it cannot be folded onto the activations, so these layers run their own
 * GEMV (UNISVQ_KERNEL_GROUPED), which forms the moments
 * S_rc = sum_v x[v d + r] z[v d + c] of each group on the tensor cores and
 * applies the row's A and B to them; for M > 64 and d in {2, 4} they run the
 * prefill GEMM, whose converters dequantise with the row's map of each group.
 *   codes      : host, [N][K] uint8, each 0..3
 *   A_f16      : host, [N][G][d][d] fp16 bits, G = ceil(K / group_cols)
 *   B_f16      : host, [N][G][d] fp16 bits
 *   d          : 1, 2, 4 or 8; K % d == 0
 *   group_cols : 128 (one packed k-tile); other values UNSUPPORTED
 * The code array uses the packed layout above with the columns of every
 * 128-column group permuted (coordinate c of the group's vectors gathered
 * into 16-column runs); the maps are stored as fp16 [Np/128][Kp/128][128]
 * [d*d + d] (A row-major, then B), zero for padding rows.
 * unisvq_linear, _group (all layers grouped, same d), _force (AUTO, DECODE,
 * GROUPED, or PREFILL for d in {2, 4}; other kernels UNSUPPORTED), _noalloc,
 * _query and
 * unisvq_dequant_debug accept the handle. The host buffers are copied before
 * return. Errors: INVALID_ARG (null pointer, bad shape, code > 3, non-finite
 * A/B), UNSUPPORTED (d or group_cols, or a K whose per-CTA slice of maps does
 * not fit in shared memory: d = 8 with K above about 10240), OOM, CUDA.
 */
unisvq_status unisvq_pack_grouped(const uint8_t* codes, const uint16_t* A_f16, const uint16_t* B_f16,
                                  int N, int K, int d, int group_cols, void* stream, unisvq_handle* out);

/*
 * y = x W_hat^T (Eq. def:ptq_loss with W_hat of Eq. col:dequant).
 *   x : device, [M][K] row-major bf16, 16-byte aligned
 *   y : device, [M][N] row-major bf16, 4-byte aligned, must not overlap x
 *   M : tokens, M >= 0 (M == 0 is a no-op)
 * Never allocates and never synchronises; enqueues on `stream`. Kernels are
 * launched with programmatic dependent launch so that, in a stream or a CUDA
 * graph, a layer starts fetching its codes while the previous kernel finishes;
 * reads of x and writes of y still wait for the previous kernel to complete.
 * Errors: INVALID_ARG (null, misaligned, overlap, M < 0), CUDA.
 */
unisvq_status unisvq_linear(unisvq_handle h, const void* x, void* y, int M, void* stream);

/* As unisvq_linear but runs the given UNISVQ_KERNEL_* for any M (crossover
 * sweeps and tests). UNSUPPORTED if that kernel cannot run this shape. */
unisvq_status unisvq_linear_force(unisvq_handle h, int kernel, const void* x, void* y, int M,
                                  void* stream);

/*
 * y_i = x W_hat_i^T for n layers that read the same x (Eq. def:ptq_loss for
 * each layer, with its own codes and its own A, B of Eq. col:dequant), e.g.
 * the q, k, v projections or the gate and up projections of one transformer
 * block. The paper defines the layer, not this grouping; it is a launch
 * convenience: for M <= 64 the n layers share each kernel launch (the row
 * blocks of the layers side by side); above, 2-bit layers with one d <= 4,
 * all per-matrix or all per-group, share one persistent prefill launch (the
 * tiles of every layer, each with its own table or maps), and other layers
 * run one unisvq_linear each.
 *   hs : n handles on the current device, all with the same K
 *   n  : 1 .. UNISVQ_MAX_GROUP
 *   x  : device, [M][K] bf16, 16-byte aligned (shared by all layers)
 *   ys : host array of n device pointers, ys[i] is [M][N_i] bf16, 4-byte
 *        aligned; no y may overlap x or another y
 * Results equal those of n unisvq_linear calls up to the order of the fp32
 * partial sums. Never allocates and never synchronises.
 * Errors: INVALID_ARG (null, n out of range, K mismatch, device mismatch,
 * misaligned, overlap, M < 0), UNSUPPORTED, CUDA.
 */
#define UNISVQ_MAX_GROUP 4
unisvq_status unisvq_linear_group(const unisvq_handle* hs, int n, const void* x, void* const* ys, int M,
                                  void* stream);

/* As unisvq_linear_group but runs the given UNISVQ_KERNEL_* (crossover sweeps
 * and tests). GEMV, GEMV_ROWS and SKINNY share one launch across the layers;
 * other kernels run once per layer as unisvq_linear_force. Same arguments,
 * results and errors as unisvq_linear_group. */
unisvq_status unisvq_linear_group_force(const unisvq_handle* hs, int n, int kernel, const void* x, void* const* ys,
                                        int M, void* stream);

/*
 * y = x W_hat^T as unisvq_linear computes it (same kernel choice), with one
 * difference: where that choice is the tcgen05 decode pair
 * (UNISVQ_KERNEL_SKINNY), its fold workspace is a static device array of the
 * library (2 MiB per device) instead of the handle's workspace. The paper has
 * no counterpart: it is a deployment variant of unisvq_linear for callers
 * that may not allocate on the call path (a server that fixed its
 * device-memory budget at start-up, or code that must not enter the
 * allocator while other work runs, since cudaMalloc and cudaFree can
 * synchronise the device); it calls no allocating routine.
 * The decode pair runs 32 tokens per launch where their folded activations
 * fit the array (Kp <= 21760), else 16 (Kp <= 43648); a layer whose fold does
 * not fit even then runs the register-operand GEMV, which needs no
 * workspace. Larger M repeat the launches (ceil(M / 32) or ceil(M / 16) fold
 * + decode pairs), up to 64 tokens; above that the prefill GEMM runs as in
 * unisvq_linear.
 * The first call on a device looks up the array's device address
 * (cudaGetSymbolAddress, with that device current); make it before any
 * stream capture. A cudaDeviceReset invalidates that address: reload the
 * library after one. All calls on a device share the one array, so calls
 * that overlap on the GPU race: order them on one stream. Arguments and
 * errors as unisvq_linear.
 */
unisvq_status unisvq_linear_noalloc(unisvq_handle h, const void* x, void* y, int M, void* stream);

/*
 * Inverse randomized Hadamard transform around the layer (Eq. def:hadamard,
 * Sec. 3.2.1). The weights were rotated before quantisation, R(W) =
 * U S_U W S_V V, with U = H_N / sqrt(N), V = H_K / sqrt(K) and S_U, S_V
 * diagonal +-1; W_hat quantises R(W). After this call every unisvq_linear*
 * on the handle returns y = x W^T for W = S_U U^T W_hat V^T S_V, computed as
 *   x_t = (x S_V) V,   y_t = x_t W_hat^T,   y = (y_t U) S_U
 * (row vectors): a rotation kernel on the way in, the layer's kernel, a
 * rotation kernel on the way out, per chunk of max_tokens tokens.
 * H_n is Sylvester's H_{2^a} Kronecker a Paley matrix H_m for n = 2^a m,
 * m in {1, 12, 20, 28, 344} (entry [(p,q),(p',q')] = H_{2^a}[p][p'] H_m[q][q'],
 * index p m + q; H_12, H_20 and H_344 from Paley's first construction with
 * q = 11, 19 and 343, H_28 from the second with q = 13). For q = 343 the
 * field is GF(7)[t] / (t^3 - 2), element e = e0 + 7 e1 + 49 e2 standing for
 * e0 + e1 t + e2 t^2, and H_344 = I + [[0, 1^T], [-1, Q]] with
 * Q[i][j] = chi(e_j - e_i), chi the quadratic character. So 11008 = 32 * 344
 * is supported. n <= 58112 (n floats in shared memory). The first call for a
 * width with m = 344 on a device writes a 16 KB sign table to that device
 * (a synchronous copy): make it outside stream capture.
 *   sign_in  : host, K bytes, 1 = -1 (the diagonal of S_V), 0 = +1
 *   sign_out : host, N bytes (S_U)
 *   max_tokens : rows of the rotated-activation buffer the handle allocates
 *                here (bf16, max_tokens x K); longer calls run in chunks
 * Both sign pointers NULL removes the transform (and its buffers). Calls on
 * the handle must be stream-ordered (they share the buffer). Grouped calls
 * with such handles run one layer at a time (each layer rotates x with its
 * own S_V). Errors: INVALID_ARG (null handle, one sign pointer null, a sign
 * byte > 1, max_tokens < 1), UNSUPPORTED (K or N not of the form above),
 * OOM, CUDA.
 */
unisvq_status unisvq_set_rht(unisvq_handle h, const uint8_t* sign_in, const uint8_t* sign_out, int max_tokens,
                             void* stream);

/* The rotation by itself, on M rows of n bf16 values (device x, y; x == y
 * allowed, otherwise no overlap): signs_first = 1 gives y = (x S) H_n /
 * sqrt(n), signs_first = 0 gives y = ((x H_n) / sqrt(n)) S, S the diagonal
 * of `signs` (device, n bytes, 1 = -1; NULL = identity). fp32 inside, bf16
 * rounding once at the end. H_n as for unisvq_set_rht; the first call with
 * m = 344 on a device writes its sign table (outside stream capture).
 * Errors: INVALID_ARG, UNSUPPORTED (n), CUDA. */
unisvq_status unisvq_hadamard(const void* x, void* y, int M, int n, const uint8_t* signs, int signs_first,
                              void* stream);

/* Test hook: writes W_hat as fp32 [N][K] row-major to device memory W (each
 * entry RN_fp32 of the exact A z + B), unpacking the device layout with the
 * same code-extraction helpers the layer kernels use. */
unisvq_status unisvq_dequant_debug(unisvq_handle h, float* W, void* stream);

/* Test hook for the unwind path of the kernels' bounded waits (every wait on
 * the device gives up after 2 s, records a code in the library's error word
 * and unwinds). One CTA allocates tensor memory, starts a 16-byte bulk copy
 * from src16 (device, 16-byte aligned) into shared memory and waits on an
 * mbarrier that nothing arrives at; after 2 s that wait records a timeout,
 * the CTA waits for its own copy, frees the tensor memory and returns.
 * out3 (device, 3 ints) receives: whether the first wait succeeded (0), whether
 * the copy landed (1), and the copy's first byte. unisvq_sync_status on the
 * stream then returns UNISVQ_ERR_TIMEOUT (and clears the error word); the
 * context stays usable. Errors: INVALID_ARG, CUDA. */
unisvq_status unisvq_debug_wait_timeout(const void* src16, int* out3, void* stream);

/* Describe the launch unisvq_linear would make for M tokens (host only). */
unisvq_status unisvq_query(unisvq_handle h, int M, unisvq_info* info);

/* Describe the launches unisvq_linear_group would make for the n layers hs
 * and M tokens (host only): N, Np and the byte and flop counts are sums over
 * the layers (x counted once), K, Kp and d those of hs[0].
 * Errors: INVALID_ARG (null, n out of range, K mismatch, M < 0). */
unisvq_status unisvq_query_group(const unisvq_handle* hs, int n, int M, unisvq_info* info);

/* Synchronise `stream`, then report and clear the device error word:
 * UNISVQ_ERR_TIMEOUT if a kernel gave up on a bounded wait since the last
 * call, UNISVQ_ERR_CUDA on a CUDA error, else UNISVQ_OK. */
unisvq_status unisvq_sync_status(void* stream);

/* Free the handle and its device memory. NULL is a no-op. The caller must
 * make sure no work using the handle is still in flight. */
unisvq_status unisvq_destroy(unisvq_handle h);

/* Device-to-device copy of a packed layer into a new handle. */
unisvq_status unisvq_clone(unisvq_handle h, void* stream, unisvq_handle* out);

const char* unisvq_status_string(unisvq_status s);

/* ---- host-only helpers (no GPU needed) ---------------------------------- */

/* Bytes of the packed code array for an N x K layer (see layout above). */
size_t unisvq_packed_code_bytes(int N, int K);

/* The prefill GEMM's shared-memory table of a per-matrix layer with this A,
 * B, d and bits, exactly as unisvq_pack builds it (host only). Every entry is
 * the exact fp64 value rounded once:
 *   bits 2, d <= 2: 16 words; word v = bf16 pair (low half first) for the
 *     index v = z_k | z_k+1 << 2 of two adjacent columns: the codeword of the
 *     vector (d = 2) or the codewords of z_k and z_k+1 (d = 1);
 *   bits 2, d = 4: 512 words; quad v = z0 | z1 << 2 | z2 << 4 | z3 << 6 is the
 *     bf16 codeword in words 2v (w0, w1) and 2v + 1 (w2, w3);
 *   bits 2, d = 8: 4096 words of fp32, quad tables q = 0, 1 of 256 rows:
 *     row v of table q holds sum_c A[r][4q + c] z_c(v) (+ B[r] for q = 0),
 *     r = 0..7, at word 2048 q + 8 v + 4 h + (r % 4), h = r/4 XOR bit 2 of v;
 *   bits 3, d <= 2: 64 words as for bits 2, d <= 2, index z_k | z_k+1 << 3;
 *   bits 3, d = 4: 512 words of fp32, pair tables p = 0, 1 of 64 rows: word
 *     256 p + 4 v + r holds A[r][2p] z_2p + A[r][2p+1] z_2p+1 (+ B[r] for
 *     p = 0), v = z_2p | z_2p+1 << 3.
 *   A_f16, B_f16: as for unisvq_pack; out: NULL to query *words only.
 * Errors: INVALID_ARG (null A, B or words, d not in {1, 2, 4, 8}, bits not
 * in {2, 3}, bits = 3 with d = 8, non-finite A/B, out_words too small), OOM. */
unisvq_status unisvq_prefill_table_host(const uint16_t* A_f16, const uint16_t* B_f16, int d, int bits,
                                        uint32_t* out, size_t out_words, size_t* words);

/* Write the packed layout of `codes` ([N][K], each 0..3) into the host
 * buffer `packed` of unisvq_packed_code_bytes(N, K) bytes. */
unisvq_status unisvq_pack_host(const uint8_t* codes, int N, int K, uint8_t* packed,
                               size_t packed_bytes);

/* Library version as an integer MAJOR*10000 + MINOR*100 + PATCH. */
int unisvq_version(void);

#ifdef __cplusplus
}
#endif

#endif /* UNISVQ_H_ */
