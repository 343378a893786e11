// Group peak-to-mean ratio (Section 3.1 motivates RRQ with it; Table 9
// reports its tensor-wise maximum as K/MAE): for every group of `group`
// consecutive weights, max |x| / (sum |x| / group), 0 for an all-zero group,
// and per matrix the maximum and mean over its groups -- the statistic for
// choosing a stage split (Section 3.3).
//
// Kernel 1 (HBM-bound, 2 bytes per weight): a lane reads its 32 bf16 weights
// (four 16-byte loads, a warp covering 2 KiB contiguously), forms max |x| and
// the binary32 sum of |x|, and the group/32 lanes of a group combine them by
// shuffles; the ratio is max / fl(sum / group) (the division by a power of
// two is exact).  Kernel 2: one CTA per matrix reduces the per-group ratios
// to their maximum and their mean (binary64 sum) in a fixed order, so the
// results are deterministic with no atomics and no workspace.
#include "rrq_device.cuh"

namespace rrq {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

template <int G>
__global__ void __launch_bounds__(kThreads) pmr_kernel(const __grid_constant__ PmrBatch p) {
  constexpr int L = G / 32;  // lanes per group
  const int lane = threadIdx.x & 31;
  const int64_t first = static_cast<int64_t>(blockIdx.x) * kWarps + (threadIdx.x >> 5);
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kWarps;
  int m = 0;
  for (int64_t chunk = first; chunk < p.total_chunks; chunk += stride) {
    while (m + 1 < p.count && chunk >= p.item[m + 1].chunk_begin) ++m;
    const PmrItem& it = p.item[m];
    const int64_t e0 = (chunk - it.chunk_begin) * kChunkElems + static_cast<int64_t>(lane) * kLaneElems;
    float peak = 0.0f, sum = 0.0f;
    if (e0 < it.n) {
      const uint4* src = reinterpret_cast<const uint4*>(it.W + e0);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint4 r = __ldcs(src + j);
        const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float a = fabsf(__uint_as_float(w[q] << 16)), b = fabsf(__uint_as_float(w[q] & 0xffff0000u));
          peak = fmaxf(peak, fmaxf(a, b));
          sum = __fadd_rn(sum, __fadd_rn(a, b));
        }
      }
    }
#pragma unroll
    for (int off = 1; off < L; off <<= 1) {
      peak = fmaxf(peak, __shfl_xor_sync(kFullMask, peak, off));
      sum = __fadd_rn(sum, __shfl_xor_sync(kFullMask, sum, off));
    }
    if (e0 < it.n && (lane & (L - 1)) == 0) {
      const float mean = __fmul_rn(sum, 1.0f / G);  // exact: power-of-two scaling
      it.pmr[e0 / G] = sum > 0.0f ? __fdiv_rn(peak, mean) : 0.0f;
    }
  }
}

// One CTA per matrix: max and mean of its per-group ratios.
__global__ void __launch_bounds__(kThreads) pmr_stats_kernel(const __grid_constant__ PmrBatch p) {
  const PmrItem& it = p.item[blockIdx.x];
  if (!it.stats) return;
  const int64_t groups = it.n / p.group;
  float mx = 0.0f;
  double sum = 0.0;
  for (int64_t g = threadIdx.x; g < groups; g += kThreads) {
    const float v = it.pmr[g];
    mx = fmaxf(mx, v);
    sum += static_cast<double>(v);
  }
  __shared__ float smx[kThreads];
  __shared__ double ssum[kThreads];
  smx[threadIdx.x] = mx;
  ssum[threadIdx.x] = sum;
  __syncthreads();
  for (int h = kThreads / 2; h > 0; h >>= 1) {
    if (threadIdx.x < h) {
      smx[threadIdx.x] = fmaxf(smx[threadIdx.x], smx[threadIdx.x + h]);
      ssum[threadIdx.x] += ssum[threadIdx.x + h];
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    it.stats[0] = smx[0];
    it.stats[1] = static_cast<float>(ssum[0] / static_cast<double>(groups));
  }
}

template <int G>
cudaError_t launch_g(const PmrBatch& p, cudaStream_t stream, int sms) {
  const int64_t want = (p.total_chunks + kWarps - 1) / kWarps;
  const int64_t cap = static_cast<int64_t>(sms) * 8;
  pmr_kernel<G><<<static_cast<int>(want < cap ? want : cap), kThreads, 0, stream>>>(p);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  pmr_stats_kernel<<<p.count, kThreads, 0, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t pmr_launch(int group, const PmrBatch& p, cudaStream_t stream, int sms) {
  switch (group) {
    case 32: return launch_g<32>(p, stream, sms);
    case 64: return launch_g<64>(p, stream, sms);
    case 128: return launch_g<128>(p, stream, sms);
    case 256: return launch_g<256>(p, stream, sms);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace rrq
