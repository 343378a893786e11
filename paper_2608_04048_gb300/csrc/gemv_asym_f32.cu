// Stage-wise product kernels for one package format (see gemv_kernel.cuh).
#include "gemv_kernel.cuh"

namespace rrq {

cudaError_t gemv_prepare_asym_f32() { return prepare_format<kAsymF32>(); }

cudaError_t gemv_launch_asym_f32(int k, int nb, int64_t max_cols, GemvBatch& p, cudaStream_t stream, int sms) {
  return launch_format<kAsymF32>(k, nb, max_cols, p, stream, sms);
}

// activation rows one launch takes (the same for every format)
int gemv_rows_per_launch(Format, int k, int64_t max_cols) { return tokens_per_launch(max_cols, k); }

}  // namespace rrq
