// RRQ prefix reconstruction (Section 3.2 Eq. 8; Appendix C): the bf16 weight
// at operating point k (k = 1..4 -> 2/4/6/8 bits) is
//     acc = L_0;  acc = fl(acc + L_i) for i = 1..k-1;  out = bf16_rne(acc)
// with L_i = fl(zero_i + fl(Q_i * scale_i)) the dequantized value of stage i.
//
// A warp owns a chunk of 1024 consecutive weights, a lane owns 32 consecutive
// weights (one 8-byte code word per stage, one scale and one zero per stage).
// Code words and metadata are loaded one chunk ahead into registers; the
// 2 KiB of bf16 output of a chunk is staged in shared memory and written by a
// 1-D bulk copy (TMA store), double-buffered per warp.
#include <cuda_bf16.h>

#include "rrq_device.cuh"

namespace rrq {
namespace {

constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;
constexpr int kSmemBytes = kWarps * 2 * kChunkBytes;
constexpr float kTwo23 = 8388608.0f;  // bits 0x4B000000 | q encode 2^23 + q for 0 <= q < 2^23

template <int K>
struct ChunkInputs {
  uint2 code[K];
  float scale[K];
  float zero[K];
};

template <int G, int K>
__device__ __forceinline__ void load_chunk(const ReconstructParams& p, int64_t e0, bool valid,
                                           ChunkInputs<K>& in) {
#pragma unroll
  for (int i = 0; i < K; ++i) {
    if (valid) {
      in.code[i] = __ldcs(reinterpret_cast<const uint2*>(p.codes[i] + (e0 >> 2)));
      in.scale[i] = __ldg(p.scales[i] + e0 / G);
      in.zero[i] = __ldg(p.zeros[i] + e0 / G);
    } else {
      in.code[i] = make_uint2(0u, 0u);
      in.scale[i] = 0.0f;
      in.zero[i] = 0.0f;
    }
  }
}

template <int G, int K>
__global__ void __launch_bounds__(kThreads, 2) reconstruct_kernel(const ReconstructParams p) {
  extern __shared__ __align__(128) uint8_t smem[];
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  uint8_t* stage_buf = smem + warp * (2 * kChunkBytes);

  const int64_t n_chunks = (p.n + kChunkElems - 1) / kChunkElems;
  const int64_t first = static_cast<int64_t>(blockIdx.x) * kWarps + warp;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kWarps;
  if (first >= n_chunks) return;

  // Slot j of a lane handles its 16-byte output piece (j + rot) & 3, so that
  // the shared-memory stores of a quarter warp hit distinct bank groups; the
  // code words are rotated right by 16*rot bits to match.
  const int rot = (lane >> 1) & 3;
  const uint32_t sel_lo = rot == 0 ? 0x3210u : rot == 1 ? 0x5432u : rot == 2 ? 0x7654u : 0x1076u;
  const uint32_t sel_hi = rot == 0 ? 0x7654u : rot == 1 ? 0x1076u : rot == 2 ? 0x3210u : 0x5432u;

  ChunkInputs<K> cur;
  {
    const int64_t e0 = first * kChunkElems + static_cast<int64_t>(lane) * kLaneElems;
    load_chunk<G, K>(p, e0, e0 < p.n, cur);
  }
  uint32_t it = 0;
  for (int64_t chunk = first; chunk < n_chunks; chunk += stride, ++it) {
    const int64_t e0 = chunk * kChunkElems + static_cast<int64_t>(lane) * kLaneElems;
    ChunkInputs<K> nxt;
    {
      const int64_t e1 = e0 + stride * kChunkElems;
      load_chunk<G, K>(p, e1, e1 < p.n, nxt);
    }

    f32x2 acc[16];
#pragma unroll
    for (int i = 0; i < K; ++i) {
      const uint32_t w0 = __byte_perm(cur.code[i].x, cur.code[i].y, sel_lo);
      const uint32_t w1 = __byte_perm(cur.code[i].x, cur.code[i].y, sel_hi);
      const f32x2 LO = pack2(cur.zero[i], cur.zero[i]);
      const f32x2 S = pack2(cur.scale[i], cur.scale[i]);
      const float c = __fmul_rn(-kTwo23, cur.scale[i]);  // exact: power-of-two scaling
      const f32x2 C = pack2(c, c);
#pragma unroll
      for (int m = 0; m < 16; ++m) {  // pair m: slot m/4, elements 2*(m%4), +1
        const uint32_t word = m < 8 ? w0 : w1;
        const int sh = 4 * (m & 7);
        const f32x2 t = pack2u(0x4B000000u | ((word >> sh) & 3u), 0x4B000000u | ((word >> (sh + 2)) & 3u));
        // fl(Q*s) as one fused multiply-add (t = 2^23 + Q), then fl(zero + step)
        const f32x2 level = add2(LO, fma2(t, S, C));
        acc[m] = (i == 0) ? level : add2(acc[m], level);
      }
    }

    // bf16 round-to-nearest-even, two weights per word
    uint32_t outw[16];
#pragma unroll
    for (int m = 0; m < 16; ++m) {
      float a, b;
      unpack2(acc[m], a, b);
      const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
      outw[m] = *reinterpret_cast<const uint32_t*>(&h);
    }

    const int b = it & 1;
    if (lane == 0) bulk_wait_read<1>();  // the store that last used buffer b has read it
    __syncwarp();
    uint4* dst = reinterpret_cast<uint4*>(stage_buf + b * kChunkBytes + lane * 64);
#pragma unroll
    for (int j = 0; j < 4; ++j)
      dst[(j + rot) & 3] = make_uint4(outw[4 * j], outw[4 * j + 1], outw[4 * j + 2], outw[4 * j + 3]);
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      const int64_t e = chunk * kChunkElems;
      const int64_t left = p.n - e;
      const uint32_t bytes = static_cast<uint32_t>((left < kChunkElems ? left : kChunkElems) * 2);
      bulk_store(p.out + e, smem_u32(stage_buf + b * kChunkBytes), bytes);
      bulk_commit();
    }
    cur = nxt;
  }
  if (lane == 0) bulk_wait<0>();
}

template <int G, int K>
cudaError_t launch_gk(const ReconstructParams& p, cudaStream_t stream, int sms) {
  static int blocks_per_sm = 0;
  if (blocks_per_sm == 0) {
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
        &blocks_per_sm, reconstruct_kernel<G, K>, kThreads, kSmemBytes);
    if (e != cudaSuccess) return e;
    if (blocks_per_sm < 1) blocks_per_sm = 1;
  }
  const int64_t n_chunks = (p.n + kChunkElems - 1) / kChunkElems;
  const int64_t want = (n_chunks + kWarps - 1) / kWarps;
  const int64_t cap = static_cast<int64_t>(sms) * blocks_per_sm;
  const int grid = static_cast<int>(want < cap ? want : cap);
  reconstruct_kernel<G, K><<<grid, kThreads, kSmemBytes, stream>>>(p);
  return cudaGetLastError();
}

template <int G>
cudaError_t launch_g(int k, const ReconstructParams& p, cudaStream_t stream, int sms) {
  switch (k) {
    case 1: return launch_gk<G, 1>(p, stream, sms);
    case 2: return launch_gk<G, 2>(p, stream, sms);
    case 3: return launch_gk<G, 3>(p, stream, sms);
    case 4: return launch_gk<G, 4>(p, stream, sms);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

cudaError_t reconstruct_prepare() { return cudaSuccess; }  // < 48 KiB shared memory

cudaError_t reconstruct_launch(int group, int k, const ReconstructParams& p, cudaStream_t stream,
                               int sms) {
  switch (group) {
    case 32: return launch_g<32>(k, p, stream, sms);
    case 64: return launch_g<64>(k, p, stream, sms);
    case 128: return launch_g<128>(k, p, stream, sms);
    case 256: return launch_g<256>(k, p, stream, sms);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace rrq
