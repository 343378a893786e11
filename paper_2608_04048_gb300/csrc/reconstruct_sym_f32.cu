// Prefix reconstruction kernels for one package format (see
// reconstruct_kernel.cuh for the arithmetic and the work decomposition).
#include "reconstruct_tile_kernel.cuh"

namespace rrq {

cudaError_t reconstruct_prepare_sym_f32() {
  cudaError_t e = prepare_format<kSymF32>();
  return e != cudaSuccess ? e : rt_prepare_format<kSymF32>();
}

cudaError_t reconstruct_launch_sym_f32(int group, int k, bool all_prefixes, const ReconstructBatch& p,
                                  cudaStream_t stream, int sms) {
  // one prefix of matrices whose size is a multiple of 2048: the wide-lane
  // kernel (reconstruct_tile_kernel.cuh); otherwise, and for every prefix
  // at once, the kernel of reconstruct_kernel.cuh (the same bits)
  if (!all_prefixes && rt_batch_ok(p)) {
    static thread_local ReconstructTileBatch t;
    if (rt_make_batch(p, t)) return rt_launch_format<kSymF32>(group, k, t, stream, sms);
  }
  return launch_format<kSymF32>(group, k, all_prefixes, p, stream, sms);
}

}  // namespace rrq
