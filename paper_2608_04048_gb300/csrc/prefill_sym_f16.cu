// Tensor-core prefill product for the sym f16 package format (see
// prefill_kernel.cuh).
#include "prefill_kernel.cuh"

namespace rrq {

cudaError_t prefill_launch_sym_f16(int k, const PrefillBatch& p, cudaStream_t stream) {
  return prefill_launch_f<kSymF16>(k, p, stream);
}

}  // namespace rrq
