// Stage-wise product kernels for one package format (see gemv_kernel.cuh).
#include "gemv_kernel.cuh"

namespace rrq {

cudaError_t gemv_prepare_sym_f16() {
  cudaError_t e = prepare_format<kSymF16>();
  return e != cudaSuccess ? e : gemv_mma_prepare_sym_f16();
}

cudaError_t gemv_launch_sym_f16(int k, int nb, int64_t max_cols, GemvBatch& p, cudaStream_t stream, int sms) {
  // groups of 64 and more: the stage-wise form on the tensor cores
  // (gemv_mma_{format}.cu); groups of 32: the prefix-weight form
  if (p.log2g >= 6) return gemv_mma_launch_sym_f16(1 << p.log2g, k, nb, max_cols, p, stream, sms);
  return launch_format<kSymF16>(k, nb, max_cols, p, stream, sms);
}

}  // namespace rrq
