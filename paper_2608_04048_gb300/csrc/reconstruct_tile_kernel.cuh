// Prefix reconstruction at one prefix k (Eq. 8; Appendix C), wide-lane form
// for matrices whose size is a multiple of 2048 weights: the same arithmetic
// as reconstruct_kernel.cuh (acc = L_0; acc = fl(acc + L_i); bf16
// round-to-nearest-even, with L_i formed by asym_levels / sym_offsets).
//
// A warp owns a chunk of 2048 consecutive weights; lane l owns 64 of them.
// Lane 0 brings the chunk's package into a per-warp ring with one 1-D bulk
// copy per stage and array (codes 512 bytes, the 2048/g scales and zeros),
// completing on the slot's mbarrier; each lane reads its 16 code bytes and
// its group's scale and zero from there.  The bf16 result goes out through a
// 2-D TMA store of the matrix viewed as [n/64, 64] with the 128-byte swizzle:
// a lane writes its 16-byte piece j at piece j ^ (l & 7) of its 128-byte row
// (the eight lanes of a quarter warp hit eight bank groups) and the copy
// puts every piece back in memory order.
#pragma once

#include <atomic>

#include "reconstruct_kernel.cuh"

namespace rrq {
namespace {

#ifndef RRQ_RT_WARPS
#define RRQ_RT_WARPS 8
#endif
#ifndef RRQ_RT_RING
#define RRQ_RT_RING 3
#endif
#ifndef RRQ_RT_CTAS_PER_SM
#define RRQ_RT_CTAS_PER_SM 2
#endif
#ifndef RRQ_RT_SLEEP
#define RRQ_RT_SLEEP 0
#endif
constexpr int kRtWarps = RRQ_RT_WARPS;
constexpr int kRtThreads = kRtWarps * 32;
constexpr int kRtRing = RRQ_RT_RING;             // chunks of package per warp in flight
constexpr int kRtChunk = 2048;                   // weights per warp chunk
constexpr int kRtOutBytes = kRtChunk * 2;        // bf16 output of a chunk (one TMA box)

template <int G, int F>
struct RtStage {  // bytes of one stage of one chunk in the ring
  static constexpr int kCodes = kRtChunk / 4;
  static constexpr int kScales = (kRtChunk / G) * (F == kSymF16 ? 2 : 4);
  static constexpr int kZeros = (F == kSymF32 || F == kSymF16) ? 0 : (kRtChunk / G) * 4;
  static constexpr int kBytes = kCodes + kScales + kZeros;
  static_assert(kScales % 16 == 0 && kZeros % 16 == 0, "bulk copies of whole 16-byte units");
};

template <int G, int K, int F>
__host__ __device__ constexpr int rt_slot_bytes() { return K * RtStage<G, F>::kBytes; }
template <int G, int K, int F>
__host__ __device__ constexpr int rt_warp_bytes() { return kRtRing * rt_slot_bytes<G, K, F>() + kRtOutBytes; }
template <int G, int K, int F>
__host__ __device__ constexpr int rt_smem_bytes() { return kRtWarps * rt_warp_bytes<G, K, F>() + kRtWarps * kRtRing * 8 + 1024; }

__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, int x, int y, uint32_t src) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.tile.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(src)
               : "memory");
}

// Bounded wait that suspends in the barrier between checks (a time hint of
// up to 1 ms per try) instead of returning at once.
__device__ __forceinline__ bool rt_wait(uint32_t bar, uint32_t parity, uint32_t limit_us) {
#if RRQ_RT_SLEEP
  if (limit_us == 0) return false;
  const uint64_t t0 = globaltimer_ns();
  const uint64_t limit_ns = static_cast<uint64_t>(limit_us) * 1000u;
  while (true) {
    uint32_t done;
    asm volatile(
        "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3; selp.u32 %0, 1, 0, p; }"
        : "=r"(done)
        : "r"(bar), "r"(parity), "r"(1000000u)
        : "memory");
    if (done) return true;
    if (globaltimer_ns() - t0 > limit_ns) return false;
  }
#else
  return mbar_wait(bar, parity, limit_us);
#endif
}

template <int G, int K, int F>
__global__ void __launch_bounds__(kRtThreads, RRQ_RT_CTAS_PER_SM) reconstruct_tile_kernel(const __grid_constant__ ReconstructTileBatch p) {
  constexpr bool kSym = F == kSymF32 || F == kSymF16;
  constexpr bool kF16 = F == kSymF16;
  using St = RtStage<G, F>;
  extern __shared__ uint8_t smem_raw[];
  // output staging holds 128-byte swizzled rows: 1024-byte alignment
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const ReconstructBatch& b = p.b;
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  uint8_t* out_stage = smem + warp * kRtOutBytes;                                      // 4 KiB, 1024-aligned
  uint8_t* ring = smem + kRtWarps * kRtOutBytes + warp * kRtRing * rt_slot_bytes<G, K, F>();
  const uint32_t ring_s = smem_u32(ring);
  const uint32_t bar0 = smem_u32(smem + kRtWarps * (kRtOutBytes + kRtRing * rt_slot_bytes<G, K, F>())) + warp * kRtRing * 8;

  const int64_t first = static_cast<int64_t>(blockIdx.x) * kRtWarps + warp;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kRtWarps;
  if (first >= b.total_chunks) return;  // warp-uniform: nothing issued

  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < kRtRing; ++i) mbar_init(bar0 + 8 * i, 1);
    fence_mbarrier_init();
  }
  __syncwarp();

  int m_issue = 0, m_work = 0;
  auto item_of = [&](int64_t chunk, int& m) {
    while (m + 1 < b.count && chunk >= b.item[m + 1].chunk_begin) ++m;
    return m;
  };
  auto issue = [&](int64_t chunk, int slot) {  // lane 0 only
    const int m = item_of(chunk, m_issue);
    const ReconstructItem& it = b.item[m];
    const int64_t c = chunk - it.chunk_begin;
    const uint32_t bar = bar0 + 8 * slot;
    const uint32_t dst = ring_s + slot * rt_slot_bytes<G, K, F>();
    mbar_arrive_expect_tx(bar, rt_slot_bytes<G, K, F>());
#pragma unroll
    for (int i = 0; i < K; ++i) {
      bulk_load(dst + i * St::kCodes, it.codes[i] + c * St::kCodes, St::kCodes, bar);
      bulk_load(dst + K * St::kCodes + i * St::kScales, static_cast<const uint8_t*>(it.scales[i]) + c * St::kScales,
                St::kScales, bar);
      if constexpr (!kSym)
        bulk_load(dst + K * (St::kCodes + St::kScales) + i * St::kZeros,
                  reinterpret_cast<const uint8_t*>(it.zeros[i]) + c * St::kZeros, St::kZeros, bar);
    }
  };
  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < kRtRing; ++i) {
      const int64_t c = first + i * stride;
      if (c < b.total_chunks) issue(c, i);
    }
  }

  // this lane's groups within the chunk: groups of 32 weights sit two to a
  // lane (bytes 0-7 and 8-15 of its code word), larger groups one
  constexpr int NH = G == 32 ? 2 : 1;
  const int gi = (lane * 64) / G;
  uint32_t iter = 0;
  bool stored = false;
  for (int64_t chunk = first; chunk < b.total_chunks; chunk += stride, ++iter) {
    const int slot = iter % kRtRing;
    const bool ready = rt_wait(bar0 + 8 * slot, (iter / kRtRing) & 1, b.wait_limit_us);
    if (!__all_sync(kFullMask, ready)) {
      // Give up: record it, wait (bounded) for this warp's copies in flight
      // so that none lands in freed shared memory, and leave.
      if (lane == 0) {
        atomicOr(b.status, kStatusTimeout);
        for (int j = 0; j < kRtRing; ++j) {
          if (chunk + j * stride >= b.total_chunks) break;
          const uint32_t jt = iter + j;
          mbar_wait(bar0 + 8 * (jt % kRtRing), (jt / kRtRing) & 1, kDrainLimitUs);
        }
        bulk_wait<0>();
      }
      __syncwarp();
      return;
    }
    const uint8_t* sl = ring + slot * rt_slot_bytes<G, K, F>();
    uint4 code[K];
    float scale[K][NH], zero[K][NH];
    bool ok = true;
#pragma unroll
    for (int i = 0; i < K; ++i) {
      code[i] = *reinterpret_cast<const uint4*>(sl + i * St::kCodes + lane * 16);
#pragma unroll
      for (int h = 0; h < NH; ++h) {
        const int g = gi + h;
        if (kF16)
          scale[i][h] = __half2float(*reinterpret_cast<const __half*>(sl + K * St::kCodes + i * St::kScales + g * 2));
        else
          scale[i][h] = *reinterpret_cast<const float*>(sl + K * St::kCodes + i * St::kScales + g * 4);
        zero[i][h] = kSym ? 0.0f
                          : *reinterpret_cast<const float*>(sl + K * (St::kCodes + St::kScales) + i * St::kZeros + g * 4);
        ok = ok && (kSym || prescale_ok(scale[i][h]));
      }
    }
    fence_proxy_async_smem();  // this lane's reads before the next async write of the slot
    __syncwarp();
    if (lane == 0) {
      const int64_t next = chunk + kRtRing * stride;
      if (next < b.total_chunks) issue(next, slot);
    }
    const int m = item_of(chunk, m_work);
    const ReconstructItem& it = b.item[m];

    f32x2 acc[32];
    const bool all_ok = __all_sync(kFullMask, ok);
#pragma unroll
    for (int i = 0; i < K; ++i) {
      const uint32_t words[4] = {code[i].x, code[i].y, code[i].z, code[i].w};
#pragma unroll
      for (int h = 0; h < NH; ++h) {
        constexpr int kBytesPerHalf = 16 / NH;
        if (kSym) {
          const f32x2 S = pack2(scale[i][h], scale[i][h]);
#pragma unroll
          for (int j = h * kBytesPerHalf; j < (h + 1) * kBytesPerHalf; ++j) {  // byte j: elements 4j..4j+3
            const uint32_t word = words[j >> 2];
            const uint32_t b8 = (j & 3) == 0 ? word : (word >> (8 * (j & 3)));
            f32x2 u01, u23;
            sym_offsets(b8, u01, u23);
            acc[2 * j] = (i == 0) ? mul2(u01, S) : fma2(u01, S, acc[2 * j]);
            acc[2 * j + 1] = (i == 0) ? mul2(u23, S) : fma2(u23, S, acc[2 * j + 1]);
          }
        } else if (all_ok) {
          const StageConsts c = stage_consts(scale[i][h], zero[i][h]);
#pragma unroll
          for (int j = h * kBytesPerHalf; j < (h + 1) * kBytesPerHalf; ++j) {
            const uint32_t word = words[j >> 2];
            const uint32_t b8 = (j & 3) == 0 ? word : (word >> (8 * (j & 3)));
            f32x2 l01, l23;
            asym_levels(b8, c, l01, l23);
            acc[2 * j] = (i == 0) ? l01 : add2(acc[2 * j], l01);
            acc[2 * j + 1] = (i == 0) ? l23 : add2(acc[2 * j + 1], l23);
          }
        } else {  // a scale outside [2^-100, 2^100] in the warp: fl(Q s) as a plain (t - 2^23) s
          const f32x2 Z = pack2(zero[i][h], zero[i][h]), S = pack2(scale[i][h], scale[i][h]);
          const f32x2 T23 = pack2(kTwo23, kTwo23), Z0 = pack2(0.0f, 0.0f);
#pragma unroll
          for (int j = h * kBytesPerHalf; j < (h + 1) * kBytesPerHalf; ++j) {
            const uint32_t word = words[j >> 2];
            const uint32_t b8 = (j & 3) == 0 ? word : (word >> (8 * (j & 3)));
            const f32x2 t01 = pack2u(magic23<3u>(b8), magic23<3u>(b8 >> 2));
            const f32x2 t23 = pack2u(magic23<3u>(b8 >> 4), magic23<3u>(b8 >> 6));
            const f32x2 l01 = add2(Z, fma2(sub2(t01, T23), S, Z0));
            const f32x2 l23 = add2(Z, fma2(sub2(t23, T23), S, Z0));
            acc[2 * j] = (i == 0) ? l01 : add2(acc[2 * j], l01);
            acc[2 * j + 1] = (i == 0) ? l23 : add2(acc[2 * j + 1], l23);
          }
        }
      }
    }

    // bf16 round-to-nearest-even into this lane's swizzled 128-byte row
    uint32_t h[32];
#pragma unroll
    for (int q = 0; q < 32; ++q) {
      float x, y;
      unpack2(acc[q], x, y);
      const __nv_bfloat162 v = __floats2bfloat162_rn(x, y);
      h[q] = *reinterpret_cast<const uint32_t*>(&v);
    }
    if (stored && lane == 0) bulk_wait_read<0>();  // the previous chunk's store has read the buffer
    __syncwarp();
    uint8_t* row = out_stage + lane * 128;
#pragma unroll
    for (int j = 0; j < 8; ++j)
      *reinterpret_cast<uint4*>(row + ((j ^ (lane & 7)) << 4)) = make_uint4(h[4 * j], h[4 * j + 1], h[4 * j + 2], h[4 * j + 3]);
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      tma_store_2d(&p.out[m], 0, static_cast<int>((chunk - it.chunk_begin) * 32), smem_u32(out_stage));
      bulk_commit();
    }
    stored = true;
  }
  if (lane == 0) bulk_wait<0>();  // output copies done before the CTA exits
}

// Every matrix of the launch a whole number of 2048-weight chunks that the
// tensor-map view can address.
inline bool rt_batch_ok(const ReconstructBatch& p) {
  for (int i = 0; i < p.count; ++i)
    if (p.item[i].n % kRtChunk != 0 || p.item[i].n / 64 >= (int64_t{1} << 31)) return false;
  return true;
}

// The batch re-counted in 2048-weight chunks, with each output's tensor map.
inline bool rt_make_batch(const ReconstructBatch& p, ReconstructTileBatch& t) {
  t.b = p;
  int64_t chunks = 0;
  for (int i = 0; i < p.count; ++i) {
    if (!encode_lane_tiles(&t.out[i], p.item[i].out[0], p.item[i].n, 64)) return false;
    t.b.item[i].chunk_begin = chunks;
    chunks += p.item[i].n / kRtChunk;
  }
  t.b.total_chunks = chunks;
  return true;
}

template <int G, int K, int F>
cudaError_t rt_launch_gk(const ReconstructTileBatch& p, cudaStream_t stream, int sms) {
  // resident CTAs per multiprocessor: the same for every device of this
  // build, asked once (an atomic: any thread may launch)
  static std::atomic<int> cached{0};
  int blocks_per_sm = cached.load(std::memory_order_relaxed);
  if (blocks_per_sm == 0) {
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&blocks_per_sm, reconstruct_tile_kernel<G, K, F>,
                                                                  kRtThreads, rt_smem_bytes<G, K, F>());
    if (e != cudaSuccess) return e;
    if (blocks_per_sm < 1) blocks_per_sm = 1;
    cached.store(blocks_per_sm, std::memory_order_relaxed);
  }
  const int64_t want = (p.b.total_chunks + kRtWarps - 1) / kRtWarps;
  const int64_t cap = static_cast<int64_t>(sms) * blocks_per_sm;
  const int grid = static_cast<int>(want < cap ? want : cap);
  reconstruct_tile_kernel<G, K, F><<<grid, kRtThreads, rt_smem_bytes<G, K, F>(), stream>>>(p);
  return cudaGetLastError();
}

template <int G, int F>
cudaError_t rt_launch_g(int k, const ReconstructTileBatch& p, cudaStream_t stream, int sms) {
  switch (k) {
    case 1: return rt_launch_gk<G, 1, F>(p, stream, sms);
    case 2: return rt_launch_gk<G, 2, F>(p, stream, sms);
    case 3: return rt_launch_gk<G, 3, F>(p, stream, sms);
    case 4: return rt_launch_gk<G, 4, F>(p, stream, sms);
    default: return cudaErrorInvalidValue;
  }
}

template <int F>
cudaError_t rt_launch_format(int group, int k, const ReconstructTileBatch& p, cudaStream_t stream, int sms) {
  switch (group) {
    case 32: return rt_launch_g<32, F>(k, p, stream, sms);
    case 64: return rt_launch_g<64, F>(k, p, stream, sms);
    case 128: return rt_launch_g<128, F>(k, p, stream, sms);
    case 256: return rt_launch_g<256, F>(k, p, stream, sms);
    default: return cudaErrorInvalidValue;
  }
}

template <int G, int F>
cudaError_t rt_prepare_g() {
  cudaError_t e;
  const cudaFuncAttribute a = cudaFuncAttributeMaxDynamicSharedMemorySize;
  if ((e = cudaFuncSetAttribute(reconstruct_tile_kernel<G, 1, F>, a, rt_smem_bytes<G, 1, F>()))) return e;
  if ((e = cudaFuncSetAttribute(reconstruct_tile_kernel<G, 2, F>, a, rt_smem_bytes<G, 2, F>()))) return e;
  if ((e = cudaFuncSetAttribute(reconstruct_tile_kernel<G, 3, F>, a, rt_smem_bytes<G, 3, F>()))) return e;
  return cudaFuncSetAttribute(reconstruct_tile_kernel<G, 4, F>, a, rt_smem_bytes<G, 4, F>());
}

template <int F>
cudaError_t rt_prepare_format() {
  cudaError_t e;
  if ((e = rt_prepare_g<32, F>())) return e;
  if ((e = rt_prepare_g<64, F>())) return e;
  if ((e = rt_prepare_g<128, F>())) return e;
  return rt_prepare_g<256, F>();
}

}  // namespace
}  // namespace rrq
