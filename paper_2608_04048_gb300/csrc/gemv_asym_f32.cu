// Stage-wise product kernels for one package format (see gemv_kernel.cuh).
#include "gemv_kernel.cuh"

namespace rrq {

cudaError_t gemv_launch_asym_f32(int k, int nb, int64_t max_cols, const GemvBatch& p, cudaStream_t stream, int sms) {
  return launch_format<kAsymF32>(k, nb, max_cols, p, stream, sms);
}

// (the ring, and so the room left for activations, depends only on the stage
// size: the same for the three 2-bit formats)
template <int F>
int rows_per_launch(int k, int64_t max_cols) {
  switch (k) {
    case 1: return tokens_per_launch<F, 1>(max_cols);
    case 2: return tokens_per_launch<F, 2>(max_cols);
    case 3: return tokens_per_launch<F, 3>(max_cols);
    case 4: return tokens_per_launch<F, 4>(max_cols);
    default: return 0;
  }
}

int gemv_rows_per_launch(Format fmt, int k, int64_t max_cols) {
  return fmt == kAsymBits ? rows_per_launch<kAsymBits>(k, max_cols) : rows_per_launch<kAsymF32>(k, max_cols);
}

}  // namespace rrq
