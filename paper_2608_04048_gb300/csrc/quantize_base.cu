// Package construction from a given base checkpoint (Algorithm 1, second
// branch): stage 0 read and dequantized, stages 1.. computed (see
// quantize_kernel.cuh).
#include "quantize_kernel.cuh"

namespace rrq {

cudaError_t quantize_prepare_base() { return prepare_all<kModeBase>(); }

cudaError_t quantize_launch_base(int group, Format fmt, const QuantizeBatch& p, cudaStream_t stream,
                                 int sms) {
  return launch_all<kModeBase>(group, fmt, p, stream, sms);
}

}  // namespace rrq
