// Stage-wise product on the tensor cores for one package format (see
// gemv_mma_kernel.cuh): groups of 64 and more, 2-bit stages.
#include "gemv_mma_kernel.cuh"

namespace rrq {

cudaError_t gemv_mma_prepare_sym_f16() { return mma_prepare_format<kSymF16>(); }

cudaError_t gemv_mma_launch_sym_f16(int group, int k, int nb, int64_t max_cols, GemvBatch& p, cudaStream_t stream,
                                int sms) {
  return mma_launch_format<kSymF16>(group, k, nb, max_cols, p, stream, sms);
}

}  // namespace rrq
