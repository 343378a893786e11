// Stage-wise product kernels for one package format (see gemv_kernel.cuh).
#include "gemv_kernel.cuh"

namespace rrq {

cudaError_t gemv_prepare_sym_f16() { return prepare_format<kSymF16>(); }

cudaError_t gemv_launch_sym_f16(int k, int nb, int64_t max_cols, GemvBatch& p, cudaStream_t stream, int sms) {
  return launch_format<kSymF16>(k, nb, max_cols, p, stream, sms);
}

}  // namespace rrq
