// Prefill GEMM (M >= 64): tcgen05 kernel (not yet built in this revision).
#include "internal.h"

namespace unisvq {

bool prefill_supported(const unisvq_layer*, int) { return false; }

PrefillPlan plan_prefill(const unisvq_layer*, int) { return PrefillPlan{}; }

unisvq_status launch_prefill(const unisvq_layer*, const void*, void*, int, cudaStream_t) {
  return UNISVQ_ERR_UNSUPPORTED;
}

}  // namespace unisvq
