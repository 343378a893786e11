// Stage-wise product kernels for the asymmetric package with per-stage code
// widths (see gemv_kernel.cuh).
#include "gemv_kernel.cuh"

namespace rrq {

cudaError_t gemv_prepare_asym_bits() { return prepare_format<kAsymBits>(); }

cudaError_t gemv_launch_asym_bits(int k, int nb, int64_t max_cols, GemvBatch& p, cudaStream_t stream, int sms) {
  return launch_format<kAsymBits>(k, nb, max_cols, p, stream, sms);
}

}  // namespace rrq
