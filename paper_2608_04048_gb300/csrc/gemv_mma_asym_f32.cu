// Stage-wise product on the tensor cores for one package format (see
// gemv_mma_kernel.cuh): groups of 64 and more, 2-bit stages.
#include "gemv_mma_kernel.cuh"

namespace rrq {

cudaError_t gemv_mma_prepare_asym_f32() { return mma_prepare_format<kAsymF32>(); }

cudaError_t gemv_mma_launch_asym_f32(int group, int k, int nb, int64_t max_cols, GemvBatch& p, cudaStream_t stream,
                                int sms) {
  return mma_launch_format<kAsymF32>(group, k, nb, max_cols, p, stream, sms);
}

}  // namespace rrq
