// Tensor-core prefill product for the asymmetric package with per-stage
// code widths (see prefill_kernel.cuh).
#include "prefill_kernel.cuh"

namespace rrq {

cudaError_t prefill_launch_asym_bits(int k, const PrefillBatch& p, cudaStream_t stream) {
  return prefill_launch_f<kAsymBits>(k, p, stream);
}

}  // namespace rrq
