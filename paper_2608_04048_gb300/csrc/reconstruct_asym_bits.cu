// Prefix reconstruction kernels for one package format (see
// reconstruct_kernel.cuh for the arithmetic and the work decomposition).
#include "reconstruct_kernel.cuh"

namespace rrq {

cudaError_t reconstruct_prepare_asym_bits() { return prepare_format<kAsymBits>(); }

cudaError_t reconstruct_launch_asym_bits(int group, int k, bool all_prefixes, const ReconstructBatch& p,
                                         cudaStream_t stream, int sms) {
  return launch_format<kAsymBits>(group, k, all_prefixes, p, stream, sms);
}

}  // namespace rrq
