// Stage-wise product kernels for one package format (see gemv_kernel.cuh).
#include "gemv_mma_kernel.cuh"

namespace rrq {

cudaError_t gemv_prepare_asym_f32() {
  cudaError_t e = prepare_format<kAsymF32>();
  return e != cudaSuccess ? e : gemv_mma_prepare_asym_f32();
}

cudaError_t gemv_launch_asym_f32(int k, int nb, int64_t max_cols, GemvBatch& p, cudaStream_t stream, int sms) {
  // groups of 64 and more: the stage-wise form on the tensor cores
  // (gemv_mma_{format}.cu); groups of 32: the prefix-weight form
  if (p.log2g >= 6) return gemv_mma_launch_asym_f32(1 << p.log2g, k, nb, max_cols, p, stream, sms);
  return launch_format<kAsymF32>(k, nb, max_cols, p, stream, sms);
}

// activation rows one launch takes: the tensor-core form (2-bit stages,
// groups of 64 and more) holds them as bf16 B fragments, the prefix-weight
// form as binary32 windows
int gemv_rows_per_launch(Format fmt, int k, int64_t max_cols, int group) {
  if (fmt != kAsymBits && group >= 64) return mma_rows_per_launch(fmt == kSymF32 || fmt == kSymF16, max_cols, group);
  return tokens_per_launch(max_cols, k);
}

}  // namespace rrq
