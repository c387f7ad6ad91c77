// C-ABI entry points of libunisvq: argument validation, the layer handle,
// kernel dispatch and the device error word.
#include <atomic>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <new>
#include <vector>

#include "common.cuh"
#include "internal.h"

namespace unisvq {

namespace {
__device__ int g_error_word;

// Per-device cache of the error word's device address (atomic: concurrent
// first calls from several host threads store the same value).
std::atomic<int*> g_err_ptr[64] = {};

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

bool overlaps(const void* a, size_t na, const void* b, size_t nb) {
  const uintptr_t a0 = reinterpret_cast<uintptr_t>(a), b0 = reinterpret_cast<uintptr_t>(b);
  return a0 < b0 + nb && b0 < a0 + na;
}

unisvq_status cuda_status(cudaError_t e) {
  if (e == cudaSuccess) return UNISVQ_OK;
  if (e == cudaErrorMemoryAllocation) return UNISVQ_ERR_OOM;
  return UNISVQ_ERR_CUDA;
}

}  // namespace

int* device_error_word() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  int* cached = g_err_ptr[dev].load(std::memory_order_acquire);
  if (!cached) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_error_word) != cudaSuccess) return nullptr;
    cached = static_cast<int*>(p);
    g_err_ptr[dev].store(cached, std::memory_order_release);
  }
  return cached;
}

}  // namespace unisvq

using namespace unisvq;

extern "C" {

int unisvq_version(void) { return 100; }

const char* unisvq_status_string(unisvq_status s) {
  switch (s) {
    case UNISVQ_OK: return "ok";
    case UNISVQ_ERR_INVALID_ARG: return "invalid argument";
    case UNISVQ_ERR_UNSUPPORTED: return "unsupported shape or kernel";
    case UNISVQ_ERR_CUDA: return "CUDA runtime error";
    case UNISVQ_ERR_OOM: return "out of device memory";
    case UNISVQ_ERR_TIMEOUT: return "a kernel gave up on a bounded wait";
  }
  return "unknown status";
}

size_t unisvq_packed_code_bytes(int N, int K) {
  if (N <= 0 || K <= 0) return 0;
  return static_cast<size_t>(round_up(N, kRowPad) / kTileRows) *
         static_cast<size_t>(round_up(K, kColPad) / kTileCols) * kTileBytes;
}

unisvq_status unisvq_prefill_table_host(const uint16_t* A_f16, const uint16_t* B_f16, int d, int bits,
                                        uint32_t* out, size_t out_words, size_t* words) {
  if (!A_f16 || !B_f16 || !words || (d != 1 && d != 2 && d != 4 && d != 8) || (bits != 2 && bits != 3) ||
      (bits == 3 && d == 8))
    return UNISVQ_ERR_INVALID_ARG;
  double A[64], B[8];
  for (int i = 0; i < d * d; ++i) {
    A[i] = f16_bits_to_f64(A_f16[i]);
    if (!std::isfinite(A[i])) return UNISVQ_ERR_INVALID_ARG;
  }
  for (int i = 0; i < d; ++i) {
    B[i] = f16_bits_to_f64(B_f16[i]);
    if (!std::isfinite(B[i])) return UNISVQ_ERR_INVALID_ARG;
  }
  std::vector<uint32_t> t;
  try {
    t = prefill_table_host(A, B, d, bits);
  } catch (...) {
    return UNISVQ_ERR_OOM;
  }
  *words = t.size();
  if (!out) return UNISVQ_OK;
  if (out_words < t.size()) return UNISVQ_ERR_INVALID_ARG;
  std::memcpy(out, t.data(), t.size() * sizeof(uint32_t));
  return UNISVQ_OK;
}

unisvq_status unisvq_pack_host(const uint8_t* codes, int N, int K, uint8_t* packed,
                               size_t packed_bytes) {
  if (!codes || !packed || N <= 0 || K <= 0) return UNISVQ_ERR_INVALID_ARG;
  if (packed_bytes < unisvq_packed_code_bytes(N, K)) return UNISVQ_ERR_INVALID_ARG;
  pack_codes_host(codes, N, K, packed);
  return UNISVQ_OK;
}

unisvq_status unisvq_pack(const uint8_t* codes, const uint16_t* A_f16, const uint16_t* B_f16,
                          int N, int K, int d, void* stream, unisvq_handle* out) {
  return unisvq_pack_bits(codes, A_f16, B_f16, N, K, d, 2, stream, out);
}

unisvq_status unisvq_pack_bits(const uint8_t* codes, const uint16_t* A_f16, const uint16_t* B_f16,
                               int N, int K, int d, int bits, void* stream, unisvq_handle* out) {
  if (!out) return UNISVQ_ERR_INVALID_ARG;
  *out = nullptr;
  if (!codes || !A_f16 || !B_f16) return UNISVQ_ERR_INVALID_ARG;
  if (d != 1 && d != 2 && d != 4 && d != 8) return UNISVQ_ERR_UNSUPPORTED;
  if (bits != 2 && bits != 3) return UNISVQ_ERR_UNSUPPORTED;
  if (bits == 3 && d == 8) return UNISVQ_ERR_UNSUPPORTED;   // 8^8 codewords: no debug codebook
  if (N <= 0 || K <= 0 || K % d != 0) return UNISVQ_ERR_INVALID_ARG;
  if (static_cast<long long>(round_up(N, kRowPad)) * round_up(K, kColPad) >= (1ll << 40))
    return UNISVQ_ERR_UNSUPPORTED;

  const size_t total = static_cast<size_t>(N) * K;
  int bad = 0;
  const int zmax = (1 << bits) - 1;
#pragma omp parallel for reduction(| : bad) schedule(static)
  for (long long i = 0; i < static_cast<long long>(total); ++i) bad |= codes[i] > zmax;
  if (bad) return UNISVQ_ERR_INVALID_ARG;

  double A[64], B[8];
  for (int i = 0; i < d * d; ++i) {
    A[i] = f16_bits_to_f64(A_f16[i]);
    if (!std::isfinite(A[i])) return UNISVQ_ERR_INVALID_ARG;
  }
  for (int i = 0; i < d; ++i) {
    B[i] = f16_bits_to_f64(B_f16[i]);
    if (!std::isfinite(B[i])) return UNISVQ_ERR_INVALID_ARG;
  }

  unisvq_layer* L = new (std::nothrow) unisvq_layer();
  if (!L) return UNISVQ_ERR_OOM;
  L->N = N;
  L->K = K;
  L->d = d;
  L->bits = bits;
  L->Np = round_up(N, kRowPad);
  L->Kp = round_up(K, kColPad);
  L->KT = L->Kp / kTileCols;
  if (cudaGetDevice(&L->device) != cudaSuccess ||
      cudaDeviceGetAttribute(&L->num_sms, cudaDevAttrMultiProcessorCount, L->device) != cudaSuccess) {
    delete L;
    return UNISVQ_ERR_CUDA;
  }
  std::memset(L->A, 0, sizeof(L->A));
  std::memset(L->B, 0, sizeof(L->B));
  double colnorm = 0;
  for (int c = 0; c < d; ++c) {
    double s = 0;
    for (int r = 0; r < d; ++r) s += std::fabs(A[r * d + c]);
    colnorm = s > colnorm ? s : colnorm;
  }
  for (int i = 0; i < d * d; ++i) {
    L->A[i] = static_cast<float>(A[i]);   // exact: fp16 -> fp32
    L->A16[i] = A_f16[i];
  }
  for (int i = 0; i < d; ++i) {
    L->B[i] = static_cast<float>(B[i]);
    L->B16[i] = B_f16[i];
  }
  // Rounded up so the activation scale never underestimates |x A|.
  L->colnorm = static_cast<float>(colnorm) * (1.0f + 1e-6f);

  // Codebook of Eq. (def:unisvq) for the dequant hook: entry v holds A z(v) + B
  // with z_c(v) the bit-field [bits (c+1) - 1 : bits c] of v, exact in fp64 and
  // rounded once to fp32.
  const int E = 1 << (bits * d);
  L->lut_entries = E;
  std::vector<float> lut32(static_cast<size_t>(E) * d);
  for (int v = 0; v < E; ++v)
    for (int r = 0; r < d; ++r) {
      double w = B[r];
      for (int c = 0; c < d; ++c) w += A[r * d + c] * static_cast<double>((v >> (bits * c)) & zmax);
      lut32[static_cast<size_t>(v) * d + r] = static_cast<float>(w);
    }
  // Prefill tile table (prefill_table_host; formats in unisvq.h at
  // unisvq_prefill_table_host).
  std::vector<uint32_t> tlut;
  try {
    tlut = prefill_table_host(A, B, d, bits);
  } catch (...) {
    delete L;
    return UNISVQ_ERR_OOM;
  }
  L->tlut_words = static_cast<int>(tlut.size());

  L->code_bytes = unisvq_packed_code_bytes(N, K);
  std::vector<uint8_t> packed;
  try {
    packed.resize(L->code_bytes);
  } catch (...) {
    delete L;
    return UNISVQ_ERR_OOM;
  }
  pack_codes_host(codes, N, K, packed.data());
  std::vector<uint8_t> hi;
  if (bits == 3) {
    L->hi_bytes = L->code_bytes / 2;
    try {
      hi.resize(L->hi_bytes);
    } catch (...) {
      delete L;
      return UNISVQ_ERR_OOM;
    }
    pack_hi_plane_host(codes, N, K, hi.data());
  }

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  L->fold_ws = nullptr;
  const size_t ws_bytes = fold_workspace_bytes(L->KT);
  cudaError_t e = cudaMalloc(&L->codes, L->code_bytes);
  if (e == cudaSuccess) e = cudaMalloc(&L->lut32, lut32.size() * sizeof(float));
  if (e == cudaSuccess) e = cudaMalloc(&L->tlut, tlut.size() * sizeof(uint32_t));
  if (e == cudaSuccess) e = cudaMalloc(&L->fold_ws, ws_bytes);
  if (e == cudaSuccess) e = cudaMemsetAsync(L->fold_ws, 0, ws_bytes, s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(L->codes, packed.data(), L->code_bytes, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess && bits == 3) e = cudaMalloc(&L->hi, L->hi_bytes);
  if (e == cudaSuccess && bits == 3) e = cudaMemcpyAsync(L->hi, hi.data(), L->hi_bytes, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(L->lut32, lut32.data(), lut32.size() * sizeof(float), cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(L->tlut, tlut.data(), tlut.size() * sizeof(uint32_t), cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e == cudaSuccess && !device_error_word()) e = cudaErrorUnknown;
  if (e != cudaSuccess) {
    cudaFree(L->codes);
    cudaFree(L->hi);
    cudaFree(L->lut32);
    cudaFree(L->tlut);
    cudaFree(L->fold_ws);
    delete L;
    return cuda_status(e);
  }
  *out = L;
  return UNISVQ_OK;
}

unisvq_status unisvq_pack_grouped(const uint8_t* codes, const uint16_t* A_f16, const uint16_t* B_f16,
                                  int N, int K, int d, int group_cols, void* stream, unisvq_handle* out) {
  if (!out) return UNISVQ_ERR_INVALID_ARG;
  *out = nullptr;
  if (!codes || !A_f16 || !B_f16) return UNISVQ_ERR_INVALID_ARG;
  if (d != 1 && d != 2 && d != 4 && d != 8) return UNISVQ_ERR_UNSUPPORTED;
  if (group_cols != kTileCols) return UNISVQ_ERR_UNSUPPORTED;
  if (N <= 0 || K <= 0 || K % d != 0) return UNISVQ_ERR_INVALID_ARG;
  if (static_cast<long long>(round_up(N, kRowPad)) * round_up(K, kColPad) >= (1ll << 40))
    return UNISVQ_ERR_UNSUPPORTED;
  const size_t total = static_cast<size_t>(N) * K;
  const int G = (K + group_cols - 1) / group_cols;
  const size_t nA = static_cast<size_t>(N) * G * d * d, nB = static_cast<size_t>(N) * G * d;
  int bad = 0;
#pragma omp parallel for reduction(| : bad) schedule(static)
  for (long long i = 0; i < static_cast<long long>(total); ++i) bad |= codes[i] > 3;
  // fp16 exponent field all ones: inf or NaN
#pragma omp parallel for reduction(| : bad) schedule(static)
  for (long long i = 0; i < static_cast<long long>(nA); ++i) bad |= (A_f16[i] & 0x7C00u) == 0x7C00u;
#pragma omp parallel for reduction(| : bad) schedule(static)
  for (long long i = 0; i < static_cast<long long>(nB); ++i) bad |= (B_f16[i] & 0x7C00u) == 0x7C00u;
  if (bad) return UNISVQ_ERR_INVALID_ARG;

  unisvq_layer* L = new (std::nothrow) unisvq_layer();
  if (!L) return UNISVQ_ERR_OOM;
  L->N = N;
  L->K = K;
  L->d = d;
  L->Np = round_up(N, kRowPad);
  L->Kp = round_up(K, kColPad);
  L->KT = L->Kp / kTileCols;
  L->bits = 2;
  L->grouped = 1;
  if (cudaGetDevice(&L->device) != cudaSuccess ||
      cudaDeviceGetAttribute(&L->num_sms, cudaDevAttrMultiProcessorCount, L->device) != cudaSuccess) {
    delete L;
    return UNISVQ_ERR_CUDA;
  }
  {   // the per-group GEMV stages a CTA's K slice of maps in shared memory
    int per = 0;
    plan_grouped(L, L->Np / kTileRows, 1, &per);
    if (!per) {   // e.g. d = 8 with K above about 10240 (18 KB of maps per k-tile)
      delete L;
      return UNISVQ_ERR_UNSUPPORTED;
    }
  }
  L->code_bytes = unisvq_packed_code_bytes(N, K);
  L->meta_bytes = static_cast<size_t>(L->Np / kTileRows) * L->KT * kTileRows * (d * d + d) * sizeof(uint16_t);
  std::vector<uint8_t> packed;
  std::vector<uint16_t> meta;
  try {
    packed.resize(L->code_bytes);
    meta.resize(L->meta_bytes / sizeof(uint16_t));
  } catch (...) {
    delete L;
    return UNISVQ_ERR_OOM;
  }
  pack_codes_grouped_host(codes, N, K, d, packed.data());
  pack_meta_grouped_host(A_f16, B_f16, N, K, d, meta.data());
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaMalloc(&L->codes, L->code_bytes);
  if (e == cudaSuccess) e = cudaMalloc(&L->meta, L->meta_bytes);
  if (e == cudaSuccess) e = cudaMemcpyAsync(L->codes, packed.data(), L->code_bytes, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(L->meta, meta.data(), L->meta_bytes, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e == cudaSuccess && !device_error_word()) e = cudaErrorUnknown;
  if (e != cudaSuccess) {
    cudaFree(L->codes);
    cudaFree(L->meta);
    cudaFree(L->hi);
    cudaFree(L->rht_signs);
    cudaFree(L->rht_x);
    delete L;
    return cuda_status(e);
  }
  *out = L;
  return UNISVQ_OK;
}

unisvq_status unisvq_clone(unisvq_handle h, void* stream, unisvq_handle* out) {
  if (!h || !out) return UNISVQ_ERR_INVALID_ARG;
  *out = nullptr;
  unisvq_layer* L = new (std::nothrow) unisvq_layer(*h);
  if (!L) return UNISVQ_ERR_OOM;
  L->codes = nullptr;
  L->lut32 = nullptr;
  L->tlut = nullptr;
  L->fold_ws = nullptr;
  L->meta = nullptr;
  L->hi = nullptr;
  L->rht_signs = nullptr;
  L->rht_x = nullptr;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // A device buffer of the source handle copied into a new allocation (none if the source has none).
  auto copy = [&](void** dst, const void* src, size_t bytes) -> cudaError_t {
    if (!src || !bytes) return cudaSuccess;
    cudaError_t e = cudaMalloc(dst, bytes);
    if (e == cudaSuccess) e = cudaMemcpyAsync(*dst, src, bytes, cudaMemcpyDeviceToDevice, s);
    return e;
  };
  cudaError_t e = copy(reinterpret_cast<void**>(&L->codes), h->codes, h->code_bytes);
  if (e == cudaSuccess) e = copy(reinterpret_cast<void**>(&L->hi), h->hi, h->hi_bytes);
  if (e == cudaSuccess && !h->grouped) {
    e = copy(reinterpret_cast<void**>(&L->lut32), h->lut32,
             static_cast<size_t>(h->lut_entries) * h->d * sizeof(float));
    if (e == cudaSuccess)
      e = copy(reinterpret_cast<void**>(&L->tlut), h->tlut, static_cast<size_t>(h->tlut_words) * sizeof(uint32_t));
    const size_t ws_bytes = fold_workspace_bytes(h->KT);
    if (e == cudaSuccess) e = cudaMalloc(&L->fold_ws, ws_bytes);
    if (e == cudaSuccess) e = cudaMemsetAsync(L->fold_ws, 0, ws_bytes, s);
  }
  if (e == cudaSuccess && h->grouped) e = copy(reinterpret_cast<void**>(&L->meta), h->meta, h->meta_bytes);
  if (e == cudaSuccess && h->rht) {
    e = copy(reinterpret_cast<void**>(&L->rht_signs), h->rht_signs, static_cast<size_t>(h->K) + h->N);
    if (e == cudaSuccess) e = cudaMalloc(&L->rht_x, static_cast<size_t>(h->rht_tokens) * h->K * sizeof(uint16_t));
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) {
    cudaFree(L->codes);
    cudaFree(L->lut32);
    cudaFree(L->tlut);
    cudaFree(L->fold_ws);
    cudaFree(L->meta);
    cudaFree(L->hi);
    cudaFree(L->rht_signs);
    cudaFree(L->rht_x);
    delete L;
    return cuda_status(e);
  }
  *out = L;
  return UNISVQ_OK;
}

unisvq_status unisvq_destroy(unisvq_handle h) {
  if (!h) return UNISVQ_OK;
  cudaError_t e1 = cudaFree(h->codes);
  cudaError_t e2 = cudaFree(h->lut32);
  cudaError_t e3 = cudaFree(h->tlut);
  cudaError_t e4 = cudaFree(h->fold_ws);
  cudaError_t e5 = cudaFree(h->meta);
  cudaError_t e6 = cudaFree(h->rht_signs);
  cudaError_t e7 = cudaFree(h->rht_x);
  cudaFree(h->hi);
  delete h;
  return (e1 == cudaSuccess && e2 == cudaSuccess && e3 == cudaSuccess && e4 == cudaSuccess && e5 == cudaSuccess &&
          e6 == cudaSuccess && e7 == cudaSuccess)
             ? UNISVQ_OK
             : UNISVQ_ERR_CUDA;
}

// Decode kernel for M <= 64 tokens over `weights` = sum of N*K of the layers
// of one launch and `nb` = their 128-row blocks (measured crossovers on
// GB300, Llama-shaped layers): the tcgen05 skinny kernel (fold + streaming
// kernel, cost nearly independent of M) for launches of at least 2^26
// weights, or of at least 2^25 weights over 64 or more row blocks or above 16
// tokens (Llama-2-7B down, 4096 x 11008, at M = 32: 16.4 us against 22.5 on
// the GEMV); the K-split cluster GEMV (lower fixed latency, better for few
// row blocks) otherwise.
// The whole-K row-slice GEMV is reachable through the force calls only.
static int decode_kernel_for(long long weights, int nb, int M) {
  if (weights >= (1ll << 26)) return UNISVQ_KERNEL_SKINNY;
  if (weights >= (1ll << 25) && (nb >= 64 || M > 16)) return UNISVQ_KERNEL_SKINNY;
  return UNISVQ_KERNEL_GEMV;
}

static int auto_kernel(const unisvq_layer* L, int M) {
  if (M > 64 && prefill_supported(L, M)) return UNISVQ_KERNEL_PREFILL;
  return decode_kernel_for(static_cast<long long>(L->N) * L->K, L->Np / kTileRows, M);
}

static unisvq_status check_io(unisvq_handle h, const void* x, void* y, int M) {
  if (!h || M < 0) return UNISVQ_ERR_INVALID_ARG;
  if (M == 0) return UNISVQ_OK;
  if (!x || !y) return UNISVQ_ERR_INVALID_ARG;
  if (!aligned(x, 16) || !aligned(y, 4)) return UNISVQ_ERR_INVALID_ARG;
  const size_t nx = static_cast<size_t>(M) * h->K * 2, ny = static_cast<size_t>(M) * h->N * 2;
  if (overlaps(x, nx, y, ny)) return UNISVQ_ERR_INVALID_ARG;
  return UNISVQ_OK;
}

// The layer itself (no RHT): `kernel` on x -> y; `noalloc` takes the tcgen05
// decode path with the library's static fold workspace.
static unisvq_status linear_inner(unisvq_handle h, int kernel, const void* x, void* y, int M, cudaStream_t s,
                                  bool noalloc) {
  if (h->bits == 3) {   // 3-bit codes: the prefill GEMM (d <= 4) above 64 tokens, else the tcgen05
                        // decode path (large layers) or the GEMV, as for 2-bit codes
    if (!noalloc && ((kernel == UNISVQ_KERNEL_AUTO && M > 64 && prefill_supported(h, M)) ||
                     kernel == UNISVQ_KERNEL_PREFILL))
      return prefill_supported(h, M) ? launch_prefill(h, x, y, M, s) : UNISVQ_ERR_UNSUPPORTED;
    if (noalloc) return launch_gemv(h, x, y, M, s);
    if (kernel != UNISVQ_KERNEL_AUTO && kernel != UNISVQ_KERNEL_DECODE && kernel != UNISVQ_KERNEL_GEMV &&
        kernel != UNISVQ_KERNEL_SKINNY)
      return kernel >= 0 && kernel <= UNISVQ_KERNEL_STREAM ? UNISVQ_ERR_UNSUPPORTED : UNISVQ_ERR_INVALID_ARG;
    if (kernel == UNISVQ_KERNEL_AUTO || kernel == UNISVQ_KERNEL_DECODE)
      kernel = decode_kernel_for(static_cast<long long>(h->N) * h->K, h->Np / kTileRows, M);
    if (kernel == UNISVQ_KERNEL_SKINNY) return h->d <= 4 ? launch_skinny(h, x, y, M, s) : UNISVQ_ERR_UNSUPPORTED;
    return launch_gemv(h, x, y, M, s);
  }
  if (noalloc) {
    if (h->grouped) {   // the per-group GEMV has no workspace
      const unisvq_layer* Ls[1] = {h};
      void* ys[1] = {y};
      return launch_grouped_group(Ls, 1, x, ys, M, s);
    }
    // unisvq_linear's own pick; only the tcgen05 decode kernels use a fold
    // workspace, here the static one, or the GEMV where the fold does not fit it
    const int k = auto_kernel(h, M);
    if (k == UNISVQ_KERNEL_PREFILL) return launch_prefill(h, x, y, M, s);
    if (k == UNISVQ_KERNEL_SKINNY) {
      const unisvq_status st = launch_skinny_static(h, x, y, M, s);
      if (st != UNISVQ_ERR_UNSUPPORTED) return st;
    }
    return launch_gemv(h, x, y, M, s);
  }
  if (h->grouped) {   // per-group maps: the prefill GEMM (d = 2, 4) for M > 64, else the per-group GEMV
    if ((kernel == UNISVQ_KERNEL_AUTO && M > 64 && prefill_supported(h, M)) || kernel == UNISVQ_KERNEL_PREFILL)
      return prefill_supported(h, M) ? launch_prefill(h, x, y, M, s) : UNISVQ_ERR_UNSUPPORTED;
    if (kernel != UNISVQ_KERNEL_AUTO && kernel != UNISVQ_KERNEL_DECODE && kernel != UNISVQ_KERNEL_GROUPED)
      return kernel >= 0 && kernel <= UNISVQ_KERNEL_STREAM ? UNISVQ_ERR_UNSUPPORTED : UNISVQ_ERR_INVALID_ARG;
    const unisvq_layer* Ls[1] = {h};
    void* ys[1] = {y};
    return launch_grouped_group(Ls, 1, x, ys, M, s);
  }
  if (kernel == UNISVQ_KERNEL_GROUPED) return UNISVQ_ERR_UNSUPPORTED;
  if (kernel == UNISVQ_KERNEL_AUTO) kernel = auto_kernel(h, M);
  if (kernel == UNISVQ_KERNEL_DECODE) kernel = decode_kernel_for(static_cast<long long>(h->N) * h->K, h->Np / kTileRows, M);
  if (kernel == UNISVQ_KERNEL_GEMV) return launch_gemv(h, x, y, M, s);
  if (kernel == UNISVQ_KERNEL_GEMV_ROWS) {
    if (!gemv_rows_supported(h, M < 4 ? M : 4)) return UNISVQ_ERR_UNSUPPORTED;
    const unisvq_layer* Ls[1] = {h};
    void* ys[1] = {y};
    return launch_gemv_rows_group(Ls, 1, x, ys, M, s);
  }
  if (kernel == UNISVQ_KERNEL_SKINNY) return launch_skinny(h, x, y, M, s);
  if (kernel == UNISVQ_KERNEL_STREAM) {
    const unisvq_layer* Ls[1] = {h};
    if (!stream_supported(Ls, 1, M)) return UNISVQ_ERR_UNSUPPORTED;
    void* ys[1] = {y};
    return launch_stream_group(Ls, 1, x, ys, M, s);
  }
  if (kernel == UNISVQ_KERNEL_PREFILL) {
    if (!prefill_supported(h, M)) return UNISVQ_ERR_UNSUPPORTED;
    return launch_prefill(h, x, y, M, s);
  }
  return UNISVQ_ERR_INVALID_ARG;
}

// Whether the layers of a call with the inverse RHT (one S_V) run the tcgen05
// decode path with the input rotation fused into its fold kernel: 2-bit
// per-matrix layers whose call resolves to UNISVQ_KERNEL_SKINNY, K foldable.
static bool rht_fused(const unisvq_handle* hs, int n, int kernel, int M) {
  long long weights = 0;
  int nb = 0;
  for (int i = 0; i < n; ++i) {
    if (hs[i]->bits != 2 || hs[i]->grouped) return false;
    weights += static_cast<long long>(hs[i]->N) * hs[i]->K;
    nb += hs[i]->Np / kTileRows;
  }
  if (kernel == UNISVQ_KERNEL_AUTO)
    kernel = M > 64 && prefill_supported(hs[0], M) ? UNISVQ_KERNEL_PREFILL : decode_kernel_for(weights, nb, M);
  else if (kernel == UNISVQ_KERNEL_DECODE)
    kernel = decode_kernel_for(weights, nb, M);
  if (kernel != UNISVQ_KERNEL_SKINNY) return false;
  const unisvq_layer* Ls[UNISVQ_MAX_GROUP];
  for (int i = 0; i < n; ++i) Ls[i] = hs[i];
  return skinny_rht_foldable(Ls, n, M);
}

// The layer with the inverse RHT around it when the handle has one (Eq.
// def:hadamard: y = ((x S_V V) W_hat^T) U S_U): on the tcgen05 decode path
// the fold kernel rotates x itself and one kernel rotates y; otherwise a
// rotation kernel, the layer and a rotation kernel per chunk of the handle's
// rotated-activation buffer. Without the RHT, the layer alone.
static unisvq_status linear_rht(unisvq_handle h, int kernel, const void* x, void* y, int M, cudaStream_t s,
                                bool noalloc) {
  if (!h->rht) return linear_inner(h, kernel, x, y, M, s, noalloc);
  if (kernel < UNISVQ_KERNEL_AUTO || kernel > UNISVQ_KERNEL_STREAM) return UNISVQ_ERR_INVALID_ARG;
  const uint8_t* s_in = h->rht_signs;
  const uint8_t* s_out = h->rht_signs + h->K;
  if (!noalloc && rht_fused(&h, 1, kernel, M)) {
    const unisvq_layer* Ls[1] = {h};
    void* ys[1] = {y};
    unisvq_status st = launch_skinny_group_rht(Ls, 1, x, ys, M, s_in, s);
    if (st == UNISVQ_OK) st = launch_rht(y, h->N, y, h->N, M, h->N, s_out, 0, true, s);
    return st;
  }
  for (int m0 = 0; m0 < M; m0 += h->rht_tokens) {
    const int mc = M - m0 < h->rht_tokens ? M - m0 : h->rht_tokens;
    const uint16_t* xc = static_cast<const uint16_t*>(x) + static_cast<size_t>(m0) * h->K;
    uint16_t* yc = static_cast<uint16_t*>(y) + static_cast<size_t>(m0) * h->N;
    unisvq_status st = launch_rht(xc, h->K, h->rht_x, h->K, mc, h->K, s_in, 1, true, s);
    if (st == UNISVQ_OK) st = linear_inner(h, kernel, h->rht_x, yc, mc, s, noalloc);
    if (st == UNISVQ_OK) st = launch_rht(yc, h->N, yc, h->N, mc, h->N, s_out, 0, true, s);
    if (st != UNISVQ_OK) return st;
  }
  return UNISVQ_OK;
}

unisvq_status unisvq_linear_force(unisvq_handle h, int kernel, const void* x, void* y, int M,
                                  void* stream) {
  unisvq_status st = check_io(h, x, y, M);
  if (st != UNISVQ_OK || M == 0) return st;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return UNISVQ_ERR_CUDA;
  if (dev != h->device) return UNISVQ_ERR_INVALID_ARG;
  return linear_rht(h, kernel, x, y, M, static_cast<cudaStream_t>(stream), false);
}

unisvq_status unisvq_linear(unisvq_handle h, const void* x, void* y, int M, void* stream) {
  return unisvq_linear_force(h, UNISVQ_KERNEL_AUTO, x, y, M, stream);
}

unisvq_status unisvq_linear_noalloc(unisvq_handle h, const void* x, void* y, int M, void* stream) {
  unisvq_status st = check_io(h, x, y, M);
  if (st != UNISVQ_OK || M == 0) return st;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return UNISVQ_ERR_CUDA;
  if (dev != h->device) return UNISVQ_ERR_INVALID_ARG;
  return linear_rht(h, UNISVQ_KERNEL_AUTO, x, y, M, static_cast<cudaStream_t>(stream), true);
}

unisvq_status unisvq_set_rht(unisvq_handle h, const uint8_t* sign_in, const uint8_t* sign_out, int max_tokens,
                             void* stream) {
  if (!h) return UNISVQ_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (!sign_in && !sign_out) {   // remove the transform
    if (cudaStreamSynchronize(s) != cudaSuccess) return UNISVQ_ERR_CUDA;
    cudaFree(h->rht_signs);
    cudaFree(h->rht_x);
    h->rht_signs = nullptr;
    h->rht_x = nullptr;
    h->rht = 0;
    h->rht_tokens = 0;
    h->rht_in_host.clear();
    return UNISVQ_OK;
  }
  if (!sign_in || !sign_out || max_tokens < 1) return UNISVQ_ERR_INVALID_ARG;
  for (int i = 0; i < h->K; ++i)
    if (sign_in[i] > 1) return UNISVQ_ERR_INVALID_ARG;
  for (int i = 0; i < h->N; ++i)
    if (sign_out[i] > 1) return UNISVQ_ERR_INVALID_ARG;
  int p2 = 0, m = 0;
  if (!rht_factor(h->K, &p2, &m) || !rht_factor(h->N, &p2, &m)) return UNISVQ_ERR_UNSUPPORTED;
  if (rht_smem_bytes(h->K) > 227 * 1024 || rht_smem_bytes(h->N) > 227 * 1024) return UNISVQ_ERR_UNSUPPORTED;
  for (const int n : {h->K, h->N}) {
    const unisvq_status st = rht_prepare(n);
    if (st != UNISVQ_OK) return st;
  }
  std::vector<uint8_t> signs(static_cast<size_t>(h->K) + h->N);
  std::memcpy(signs.data(), sign_in, h->K);
  std::memcpy(signs.data() + h->K, sign_out, h->N);
  uint8_t* d_signs = nullptr;
  uint16_t* d_x = nullptr;
  cudaError_t e = cudaMalloc(&d_signs, signs.size());
  if (e == cudaSuccess) e = cudaMalloc(&d_x, static_cast<size_t>(max_tokens) * h->K * sizeof(uint16_t));
  if (e == cudaSuccess) e = cudaMemcpyAsync(d_signs, signs.data(), signs.size(), cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) {
    cudaFree(d_signs);
    cudaFree(d_x);
    return cuda_status(e);
  }
  cudaFree(h->rht_signs);
  cudaFree(h->rht_x);
  h->rht_signs = d_signs;
  h->rht_x = d_x;
  h->rht_tokens = max_tokens;
  h->rht = 1;
  h->rht_in_host.assign(sign_in, sign_in + h->K);
  return UNISVQ_OK;
}

unisvq_status unisvq_hadamard(const void* x, void* y, int M, int n, const uint8_t* signs, int signs_first,
                              void* stream) {
  if (M < 0 || n <= 0 || (signs_first != 0 && signs_first != 1)) return UNISVQ_ERR_INVALID_ARG;
  if (M == 0) return UNISVQ_OK;
  if (!x || !y || !aligned(x, 2) || !aligned(y, 2)) return UNISVQ_ERR_INVALID_ARG;
  const size_t bytes = static_cast<size_t>(M) * n * 2;
  if (x != y && overlaps(x, bytes, y, bytes)) return UNISVQ_ERR_INVALID_ARG;
  int p2 = 0, m = 0;
  if (!rht_factor(n, &p2, &m)) return UNISVQ_ERR_UNSUPPORTED;
  const unisvq_status st = rht_prepare(n);
  if (st != UNISVQ_OK) return st;
  return launch_rht(x, n, y, n, M, n, signs, signs_first, false, static_cast<cudaStream_t>(stream));
}

static unisvq_status group_inner(const unisvq_handle* hs, int n, int kernel, const void* x, void* const* ys, int M,
                                 cudaStream_t s);

unisvq_status unisvq_linear_group_force(const unisvq_handle* hs, int n, int kernel, const void* x, void* const* ys,
                                        int M, void* stream) {
  if (!hs || !ys || n < 1 || n > UNISVQ_MAX_GROUP || M < 0) return UNISVQ_ERR_INVALID_ARG;
  for (int i = 0; i < n; ++i) {
    if (!hs[i] || hs[i]->K != hs[0]->K || hs[i]->device != hs[0]->device) return UNISVQ_ERR_INVALID_ARG;
    const unisvq_status st = check_io(hs[i], x, ys[i], M);
    if (st != UNISVQ_OK) return st;
    for (int j = 0; j < i; ++j)
      if (ys[j] && ys[i] &&
          overlaps(ys[i], static_cast<size_t>(M) * hs[i]->N * 2, ys[j], static_cast<size_t>(M) * hs[j]->N * 2))
        return UNISVQ_ERR_INVALID_ARG;
  }
  if (M == 0) return UNISVQ_OK;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return UNISVQ_ERR_CUDA;
  if (dev != hs[0]->device) return UNISVQ_ERR_INVALID_ARG;
  const cudaStream_t s = static_cast<cudaStream_t>(stream);
  int nrht = 0;
  for (int i = 0; i < n; ++i) nrht += hs[i]->rht ? 1 : 0;
  if (!nrht) return group_inner(hs, n, kernel, x, ys, M, s);
  bool shared = nrht == n;
  for (int i = 1; i < n && shared; ++i) shared = hs[i]->rht_in_host == hs[0]->rht_in_host;
  if (!shared) {   // each layer rotates x with its own S_V: one call per layer
    for (int i = 0; i < n; ++i) {
      const unisvq_status st = linear_rht(hs[i], kernel, x, ys[i], M, s, false);
      if (st != UNISVQ_OK) return st;
    }
    return UNISVQ_OK;
  }
  // One S_V for every layer: rotate x once (into the first handle's buffer),
  // run the layers as one group, rotate each output with its own U S_U.
  if (kernel < UNISVQ_KERNEL_AUTO || kernel > UNISVQ_KERNEL_STREAM) return UNISVQ_ERR_INVALID_ARG;
  const int K = hs[0]->K;
  if (rht_fused(hs, n, kernel, M)) {   // the fold kernel rotates x; one launch rotates the outputs
    const unisvq_layer* Ls[UNISVQ_MAX_GROUP];
    RhtSetDesc sets[UNISVQ_MAX_GROUP];
    for (int i = 0; i < n; ++i) {
      Ls[i] = hs[i];
      sets[i] = RhtSetDesc{ys[i], hs[i]->N, ys[i], hs[i]->N, hs[i]->N, hs[i]->rht_signs + K};
    }
    unisvq_status st = launch_skinny_group_rht(Ls, n, x, ys, M, hs[0]->rht_signs, s);
    if (st == UNISVQ_OK) st = launch_rht_sets(sets, n, M, 0, true, s);
    return st;
  }
  int cap = hs[0]->rht_tokens;
  for (int i = 1; i < n; ++i) cap = hs[i]->rht_tokens < cap ? hs[i]->rht_tokens : cap;
  for (int m0 = 0; m0 < M; m0 += cap) {
    const int mc = M - m0 < cap ? M - m0 : cap;
    void* yc[UNISVQ_MAX_GROUP];
    for (int i = 0; i < n; ++i) yc[i] = static_cast<uint16_t*>(ys[i]) + static_cast<size_t>(m0) * hs[i]->N;
    unisvq_status st = launch_rht(static_cast<const uint16_t*>(x) + static_cast<size_t>(m0) * K, K, hs[0]->rht_x, K,
                                  mc, K, hs[0]->rht_signs, 1, true, s);
    if (st == UNISVQ_OK) st = group_inner(hs, n, kernel, hs[0]->rht_x, yc, mc, s);
    if (st == UNISVQ_OK) {   // the output rotations of all layers, one launch where the widths allow
      RhtSetDesc sets[UNISVQ_MAX_GROUP];
      for (int i = 0; i < n; ++i) sets[i] = RhtSetDesc{yc[i], hs[i]->N, yc[i], hs[i]->N, hs[i]->N, hs[i]->rht_signs + K};
      st = launch_rht_sets(sets, n, mc, 0, true, s);
    }
    if (st != UNISVQ_OK) return st;
  }
  return UNISVQ_OK;
}

// A grouped call without the RHT: one launch across the layers where the
// kernel allows it, else one per layer.
static unisvq_status group_inner(const unisvq_handle* hs, int n, int kernel, const void* x, void* const* ys, int M,
                                 cudaStream_t s) {
  int n3 = 0;
  for (int i = 0; i < n; ++i) n3 += hs[i]->bits == 3 ? 1 : 0;
  if (n3) {   // 3-bit layers: one decode launch (tcgen05 or GEMV) when every layer is 3-bit, else layer by layer
    bool pf = kernel == UNISVQ_KERNEL_AUTO && M > 64;
    for (int i = 0; i < n && pf; ++i) pf = prefill_supported(hs[i], M);
    if (!pf && n3 == n &&
        (kernel == UNISVQ_KERNEL_AUTO || kernel == UNISVQ_KERNEL_DECODE || kernel == UNISVQ_KERNEL_GEMV ||
         kernel == UNISVQ_KERNEL_SKINNY)) {
      const unisvq_layer* Ls[UNISVQ_MAX_GROUP];
      long long w3 = 0;
      int nb3 = 0;
      bool d_ok = true;
      for (int i = 0; i < n; ++i) {
        Ls[i] = hs[i];
        w3 += static_cast<long long>(hs[i]->N) * hs[i]->K;
        nb3 += hs[i]->Np / kTileRows;
        d_ok = d_ok && hs[i]->d <= 4;
      }
      int k = kernel;
      if (k == UNISVQ_KERNEL_AUTO || k == UNISVQ_KERNEL_DECODE) k = decode_kernel_for(w3, nb3, M);
      if (k == UNISVQ_KERNEL_SKINNY) return d_ok ? launch_skinny_group(Ls, n, x, ys, M, s) : UNISVQ_ERR_UNSUPPORTED;
      return launch_gemv_group(Ls, n, x, ys, M, s);
    }
    for (int i = 0; i < n; ++i) {
      const unisvq_status st = linear_inner(hs[i], kernel, x, ys[i], M, s, false);
      if (st != UNISVQ_OK) return st;
    }
    return UNISVQ_OK;
  }
  int ngrouped = 0;
  for (int i = 0; i < n; ++i) ngrouped += hs[i]->grouped ? 1 : 0;
  if (ngrouped) {   // all layers per-group with one d, run by the per-group GEMV
    if (ngrouped != n) return UNISVQ_ERR_UNSUPPORTED;
    bool pf = kernel == UNISVQ_KERNEL_PREFILL || (kernel == UNISVQ_KERNEL_AUTO && M > 64);
    for (int i = 0; i < n && pf; ++i) pf = prefill_supported(hs[i], M);
    if (pf || kernel == UNISVQ_KERNEL_PREFILL) {   // the prefill GEMM: one launch where it can, else layer by layer
      const unisvq_layer* Lp[UNISVQ_MAX_GROUP];
      for (int i = 0; i < n; ++i) Lp[i] = hs[i];
      if (prefill_group_supported(Lp, n, M)) return launch_prefill_group(Lp, n, x, ys, M, s);
      for (int i = 0; i < n; ++i) {
        const unisvq_status st = linear_inner(hs[i], kernel, x, ys[i], M, s, false);
        if (st != UNISVQ_OK) return st;
      }
      return UNISVQ_OK;
    }
    if (kernel != UNISVQ_KERNEL_AUTO && kernel != UNISVQ_KERNEL_DECODE && kernel != UNISVQ_KERNEL_GROUPED)
      return UNISVQ_ERR_UNSUPPORTED;
    const unisvq_layer* Ls[UNISVQ_MAX_GROUP];
    for (int i = 0; i < n; ++i) {
      if (hs[i]->d != hs[0]->d) return UNISVQ_ERR_UNSUPPORTED;
      Ls[i] = hs[i];
    }
    return launch_grouped_group(Ls, n, x, ys, M, s);
  }
  if (kernel == UNISVQ_KERNEL_GROUPED) return UNISVQ_ERR_UNSUPPORTED;
  long long weights = 0;
  int nb = 0;
  for (int i = 0; i < n; ++i) {
    weights += static_cast<long long>(hs[i]->N) * hs[i]->K;
    nb += hs[i]->Np / kTileRows;
  }
  if (kernel == UNISVQ_KERNEL_AUTO)
    kernel = M > 64 && prefill_supported(hs[0], M) ? UNISVQ_KERNEL_PREFILL : decode_kernel_for(weights, nb, M);
  else if (kernel == UNISVQ_KERNEL_DECODE)
    kernel = decode_kernel_for(weights, nb, M);
  const unisvq_layer* Ls[UNISVQ_MAX_GROUP];
  for (int i = 0; i < n; ++i) Ls[i] = hs[i];
  if (kernel == UNISVQ_KERNEL_GEMV) return launch_gemv_group(Ls, n, x, ys, M, s);
  if (kernel == UNISVQ_KERNEL_SKINNY) return launch_skinny_group(Ls, n, x, ys, M, s);
  if (kernel == UNISVQ_KERNEL_STREAM) {
    if (!stream_supported(Ls, n, M)) return UNISVQ_ERR_UNSUPPORTED;
    return launch_stream_group(Ls, n, x, ys, M, s);
  }
  if (kernel == UNISVQ_KERNEL_GEMV_ROWS) {
    for (int i = 0; i < n; ++i)
      if (!gemv_rows_supported(Ls[i], M < 4 ? M : 4)) return UNISVQ_ERR_UNSUPPORTED;
    return launch_gemv_rows_group(Ls, n, x, ys, M, s);
  }
  // the prefill GEMM: one persistent launch over every layer's tiles where the
  // layers allow it, else layer by layer below
  if (kernel == UNISVQ_KERNEL_PREFILL && prefill_group_supported(Ls, n, M))
    return launch_prefill_group(Ls, n, x, ys, M, s);
  for (int i = 0; i < n; ++i) {
    const unisvq_status st = linear_inner(hs[i], kernel, x, ys[i], M, s, false);
    if (st != UNISVQ_OK) return st;
  }
  return UNISVQ_OK;
}

unisvq_status unisvq_linear_group(const unisvq_handle* hs, int n, const void* x, void* const* ys, int M,
                                  void* stream) {
  return unisvq_linear_group_force(hs, n, UNISVQ_KERNEL_AUTO, x, ys, M, stream);
}

unisvq_status unisvq_debug_wait_timeout(const void* src16, int* out3, void* stream) {
  if (!src16 || !out3 || !aligned(src16, 16) || !aligned(out3, 4)) return UNISVQ_ERR_INVALID_ARG;
  return launch_wait_probe(src16, out3, static_cast<cudaStream_t>(stream));
}

unisvq_status unisvq_dequant_debug(unisvq_handle h, float* W, void* stream) {
  if (!h || !W || !aligned(W, 4)) return UNISVQ_ERR_INVALID_ARG;
  return launch_dequant(h, W, static_cast<cudaStream_t>(stream));
}

// Algorithmic metadata bytes: one fp16 (A, B) per matrix, or per (row, group)
// of 128 columns for a per-group layer (padding excluded).
static long long meta_bytes_of(const unisvq_layer* h) {
  const long long per = static_cast<long long>(h->d * h->d + h->d) * 2;
  return h->grouped ? per * h->N * ((h->K + kTileCols - 1) / kTileCols) : per;
}

// Launch geometry of `kernel` for the n layers of one call (query helpers).
static void describe_launch(const unisvq_layer* const* Ls, int n, int kernel, int M, unisvq_info* info) {
  const unisvq_layer* h = Ls[0];
  const int m = M > 0 ? M : 1;
  info->kernel = kernel;
  if (kernel == UNISVQ_KERNEL_GROUPED) {
    int nb = 0;
    for (int i = 0; i < n; ++i) nb += Ls[i]->Np / kTileRows;
    int per = 0;
    const DecodePlan p = plan_grouped(h, nb, m, &per);
    info->split_k = p.ks;
    info->launches = per > 0 ? (m + per - 1) / per : 0;
    info->grid_ctas = p.ks * nb * info->launches;
  } else if (kernel == UNISVQ_KERNEL_STREAM) {
    const StreamPlan p = plan_stream(Ls, n, m < kStreamMaxTok ? m : kStreamMaxTok);
    info->split_k = 1;
    info->launches = (m + kStreamMaxTok - 1) / kStreamMaxTok;
    info->grid_ctas = p.ctas * info->launches;
  } else if (kernel == UNISVQ_KERNEL_GEMV_ROWS) {
    info->split_k = 1;
    info->grid_ctas = 0;
    for (int i = 0; i < n; ++i) info->grid_ctas += Ls[i]->Np / 32;
    info->launches = (m + 3) / 4;
  } else if (kernel == UNISVQ_KERNEL_GEMV) {
    const DecodePlan p = plan_gemv(h, m > 32 ? 32 : m);
    info->split_k = p.ks;
    int nb = 0;
    for (int i = 0; i < n; ++i) nb += Ls[i]->Np / kTileRows;
    info->launches = (m + 31) / 32;
    info->grid_ctas = p.ks * nb * info->launches;
  } else if (kernel == UNISVQ_KERNEL_SKINNY) {
    const DecodePlan p = plan_skinny(Ls, n, m);
    const int per = skinny_tokens_per_launch(Ls, n);
    int nb = 0;
    for (int i = 0; i < n; ++i) nb += Ls[i]->Np / kTileRows;
    info->split_k = p.ks;
    const int chunks = (m + per - 1) / per;
    info->launches = 2 * chunks;   // fold kernel + streaming kernel per 32 (or 16) tokens
    info->grid_ctas = p.ks * nb * chunks;
  } else if (prefill_group_supported(Ls, n, m)) {   // one launch over every layer's tiles
    const PrefillPlan p = plan_prefill_group(Ls, n, m);
    info->split_k = 1;
    info->grid_ctas = p.grid;
    info->launches = 1;
  } else {
    info->split_k = 1;
    info->grid_ctas = 0;
    for (int i = 0; i < n; ++i) info->grid_ctas += plan_prefill(Ls[i], m).grid;
    info->launches = n;
  }
}

unisvq_status unisvq_query(unisvq_handle h, int M, unisvq_info* info) {
  if (!h || !info || M < 0) return UNISVQ_ERR_INVALID_ARG;
  std::memset(info, 0, sizeof(*info));
  info->N = h->N;
  info->K = h->K;
  info->d = h->d;
  info->Np = h->Np;
  info->Kp = h->Kp;
  info->code_bytes = static_cast<long long>(h->code_bytes + h->hi_bytes);
  info->meta_bytes = meta_bytes_of(h);
  info->algo_bytes = static_cast<long long>(h->N) * h->K * h->bits / 8 + info->meta_bytes +
                     2ll * M * h->K + 2ll * M * h->N;
  info->flops = 2.0 * M * static_cast<double>(h->N) * h->K;
  const unisvq_layer* Ls[1] = {h};
  const int mq = M > 0 ? M : 1;
  const int kq = h->grouped ? (mq > 64 && prefill_supported(h, mq) ? UNISVQ_KERNEL_PREFILL : UNISVQ_KERNEL_GROUPED)
                             : auto_kernel(h, mq);
  describe_launch(Ls, 1, kq, M, info);
  if (h->rht) {
    // fused: one output rotation; else an input and an output rotation per
    // chunk of the rotated-activation buffer
    if (rht_fused(&h, 1, UNISVQ_KERNEL_AUTO, mq))
      info->launches += 1;
    else
      info->launches += 2 * ((mq + h->rht_tokens - 1) / h->rht_tokens);
  }
  return UNISVQ_OK;
}

unisvq_status unisvq_query_group(const unisvq_handle* hs, int n, int M, unisvq_info* info) {
  if (!hs || !info || n < 1 || n > UNISVQ_MAX_GROUP || M < 0) return UNISVQ_ERR_INVALID_ARG;
  for (int i = 0; i < n; ++i)
    if (!hs[i] || hs[i]->K != hs[0]->K) return UNISVQ_ERR_INVALID_ARG;
  std::memset(info, 0, sizeof(*info));
  long long weights = 0;
  int nb = 0;
  for (int i = 0; i < n; ++i) {
    const unisvq_layer* h = hs[i];
    info->N += h->N;
    info->Np += h->Np;
    info->code_bytes += static_cast<long long>(h->code_bytes + h->hi_bytes);
    info->meta_bytes += meta_bytes_of(h);
    info->algo_bytes += static_cast<long long>(h->N) * h->K * h->bits / 8 + 2ll * M * h->N;
    info->flops += 2.0 * M * static_cast<double>(h->N) * h->K;
    weights += static_cast<long long>(h->N) * h->K;
    nb += h->Np / kTileRows;
  }
  info->K = hs[0]->K;
  info->Kp = hs[0]->Kp;
  info->d = hs[0]->d;
  info->algo_bytes += info->meta_bytes + 2ll * M * hs[0]->K;   // x is read once per call
  const int m = M > 0 ? M : 1;
  const int kernel = hs[0]->grouped ? (m > 64 && prefill_supported(hs[0], m) ? UNISVQ_KERNEL_PREFILL
                                                                            : UNISVQ_KERNEL_GROUPED)
                     : m > 64 && prefill_supported(hs[0], m) ? UNISVQ_KERNEL_PREFILL
                                                             : decode_kernel_for(weights, nb, m);
  const unisvq_layer* Ls[UNISVQ_MAX_GROUP];
  for (int i = 0; i < n; ++i) Ls[i] = hs[i];
  describe_launch(Ls, n, kernel, M, info);
  int nrht = 0;
  for (int i = 0; i < n; ++i) nrht += hs[i]->rht ? 1 : 0;
  if (nrht) {   // the rotations of unisvq_linear_group_force's RHT paths
    bool shared = nrht == n;
    for (int i = 1; i < n && shared; ++i) shared = hs[i]->rht_in_host == hs[0]->rht_in_host;
    if (!shared) {   // one unisvq_linear per layer: count each layer's own launches
      info->launches = 0;
      for (int i = 0; i < n; ++i) {
        unisvq_info one;
        unisvq_query(hs[i], M, &one);
        info->launches += one.launches;
      }
    } else {
      int ns[UNISVQ_MAX_GROUP], cap = hs[0]->rht_tokens;
      for (int i = 0; i < n; ++i) {
        ns[i] = hs[i]->N;
        cap = hs[i]->rht_tokens < cap ? hs[i]->rht_tokens : cap;
      }
      const int outs = rht_set_launches(ns, n);
      if (rht_fused(hs, n, UNISVQ_KERNEL_AUTO, m))
        info->launches += outs;
      else
        info->launches += (1 + outs) * ((m + cap - 1) / cap);
    }
  }
  return UNISVQ_OK;
}

unisvq_status unisvq_sync_status(void* stream) {
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return UNISVQ_ERR_CUDA;
  int* ew = device_error_word();
  if (!ew) return UNISVQ_ERR_CUDA;
  int v = 0;
  if (cudaMemcpy(&v, ew, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return UNISVQ_ERR_CUDA;
  if (v != 0) {
    const int zero = 0;
    cudaMemcpy(ew, &zero, sizeof(int), cudaMemcpyHostToDevice);
    return UNISVQ_ERR_TIMEOUT;
  }
  return UNISVQ_OK;
}

}  // extern "C"
