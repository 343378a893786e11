// Package construction that also writes the bf16 reconstruction after every
// stage (see quantize_kernel.cuh).
#include "quantize_kernel.cuh"

namespace rrq {

cudaError_t quantize_prepare_emit() { return prepare_all<kModeEmit>(); }

cudaError_t quantize_launch_emit(int group, Format fmt, const QuantizeBatch& p, cudaStream_t stream,
                                 int sms) {
  return launch_all<kModeEmit>(group, fmt, p, stream, sms);
}

}  // namespace rrq
