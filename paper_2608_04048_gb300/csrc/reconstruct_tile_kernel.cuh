// Prefix reconstruction at one prefix k (Eq. 8; Appendix C), wide-lane form
// for matrices whose size is a multiple of 2048 weights: the same arithmetic
// as reconstruct_kernel.cuh (acc = L_0; acc = fl(acc + L_i); bf16
// round-to-nearest-even, with L_i formed by asym_levels / sym_offsets).
//
// A warp owns a chunk of 2048 consecutive weights; lane l owns 64 of them.
// The chunk's package (per stage: codes 512 bytes, the 2048/g scales and
// zeros) comes into a per-warp ring of shared-memory slots, completing on the
// slot's mbarrier: by one bulk copy per stage and array from lane 0 up to
// k = 2, by per-lane 16-byte cp.async copies from k = 3 (RtCfg).  Each lane
// reads its 16 code bytes and its group's scale and zero from there.  At k = 1 the lane forms its 64
// levels and then converts them; for k >= 2 it sums 4 weights over all k
// stages (in stage order, as Eq. 8 reads) before the next 4, converting as
// it goes, which keeps few accumulators live and leaves room for 12 warps a
// CTA (RtCfg).  The bf16 result goes out through a
// 2-D TMA store of the matrix viewed as [n/64, 64] with the 128-byte swizzle:
// a lane writes its 16-byte piece j at piece j ^ (l & 7) of its 128-byte row
// (the eight lanes of a quarter warp hit eight bank groups) and the copy
// puts every piece back in memory order.
#pragma once

#include <atomic>

#include "reconstruct_kernel.cuh"

namespace rrq {
namespace {

// Launch shape by prefix.  At k = 1 a lane sums nothing: it keeps its 64
// levels in registers and writes them after, 8 warps a CTA with three chunks
// of package in flight per warp.  For k >= 2 a lane finishes 4 weights over
// all k stages before the next 4 (few live accumulators), which leaves room
// for 12 warps a CTA with two chunks in flight.  Two CTAs per multiprocessor
// in both.  Up to k = 2 lane 0 brings a chunk in with one bulk copy per
// array; from k = 3 on (3k copies, most of them of 64 bytes) every lane
// copies its own 16-byte units with cp.async instead, and the warp index is
// taken by a broadcast so that the copy and store operands are known to be
// warp-uniform.
template <int K>
struct RtCfg {
  static constexpr bool kOuter = K > 1;
  static constexpr bool kLaneCopies = K > 2;
  static constexpr int kWarps = kOuter ? 12 : 8;
  static constexpr int kThreads = kWarps * 32;
  static constexpr int kRing = kOuter ? 2 : 3;  // chunks of package per warp in flight
};
constexpr int kRtCtasPerSm = 2;
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
__host__ __device__ constexpr int rt_warp_bytes() { return RtCfg<K>::kRing * rt_slot_bytes<G, K, F>() + kRtOutBytes; }
template <int G, int K, int F>
__host__ __device__ constexpr int rt_smem_bytes() {
  return RtCfg<K>::kWarps * (rt_warp_bytes<G, K, F>() + RtCfg<K>::kRing * 8) + 1024;
}

__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, int x, int y, uint32_t src) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.tile.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(src)
               : "memory");
}

template <int G, int K, int F>
__global__ void __launch_bounds__(RtCfg<K>::kThreads, kRtCtasPerSm) reconstruct_tile_kernel(const __grid_constant__ ReconstructTileBatch p) {
  constexpr int kRtWarps = RtCfg<K>::kWarps;
  constexpr int kRtRing = RtCfg<K>::kRing;
  constexpr bool kSym = F == kSymF32 || F == kSymF16;
  constexpr bool kF16 = F == kSymF16;
  using St = RtStage<G, F>;
  extern __shared__ uint8_t smem_raw[];
  // output staging holds 128-byte swizzled rows: 1024-byte alignment
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const ReconstructBatch& b = p.b;
  const int lane = threadIdx.x & 31;
  const int warp = RtCfg<K>::kLaneCopies ? __shfl_sync(kFullMask, static_cast<int>(threadIdx.x >> 5), 0)
                                         : static_cast<int>(threadIdx.x >> 5);
  uint8_t* out_stage = smem + warp * kRtOutBytes;                                      // 4 KiB, 1024-aligned
  uint8_t* ring = smem + kRtWarps * kRtOutBytes + warp * kRtRing * rt_slot_bytes<G, K, F>();
  const uint32_t ring_s = smem_u32(ring);
  const uint32_t bar0 = smem_u32(smem + kRtWarps * (kRtOutBytes + kRtRing * rt_slot_bytes<G, K, F>())) + warp * kRtRing * 8;

  const int64_t first = static_cast<int64_t>(blockIdx.x) * kRtWarps + warp;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kRtWarps;
  if (first >= b.total_chunks) return;  // warp-uniform: nothing issued

  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < kRtRing; ++i) mbar_init(bar0 + 8 * i, RtCfg<K>::kLaneCopies ? 32 : 1);
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
  // (from k = 3) every lane copies its 16-byte units of the slot (the slot
  // holds the K code arrays, then the K scale arrays, then the K zero
  // arrays, each unit at its own index) and arrives on the slot's barrier
  // when they land
  auto issue_all = [&](int64_t chunk, int slot) {
    const int m = item_of(chunk, m_issue);
    const ReconstructItem& it = b.item[m];
    const int64_t c = chunk - it.chunk_begin;
    constexpr int kCodeU = St::kCodes / 16, kScaleU = St::kScales / 16, kZeroU = St::kZeros / 16;
    constexpr int kUnits = K * (kCodeU + kScaleU + kZeroU);
    static_assert(kCodeU == 32, "one code unit per lane and stage");
    const uint32_t dst = ring_s + slot * rt_slot_bytes<G, K, F>() + lane * 16;
#pragma unroll
    for (int t = 0; t < (kUnits + 31) / 32; ++t) {
      const int u = t * 32 + lane;
      if (t < K) {
        cp_async_16(dst + t * 512, it.codes[t] + c * St::kCodes + lane * 16, 16);
      } else if (u < kUnits) {
        const int v = u - K * kCodeU;
        const uint8_t* src;
        constexpr int kZeroD = kZeroU > 0 ? kZeroU : 1;  // no zeros on the symmetric grid
        if (kZeroU == 0 || v < K * kScaleU)
          src = static_cast<const uint8_t*>(it.scales[v / kScaleU]) + c * St::kScales + (v % kScaleU) * 16;
        else
          src = reinterpret_cast<const uint8_t*>(it.zeros[(v - K * kScaleU) / kZeroD]) + c * St::kZeros +
                ((v - K * kScaleU) % kZeroD) * 16;
        cp_async_16(dst + t * 512, src, 16);
      }
    }
    cp_async_mbar_arrive_noinc(bar0 + 8 * slot);
  };
#pragma unroll
  for (int i = 0; i < kRtRing; ++i) {
    const int64_t c = first + i * stride;
    if (c >= b.total_chunks) break;
    if constexpr (RtCfg<K>::kLaneCopies) {
      issue_all(c, i);
    } else if (lane == 0) {
      issue(c, i);
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
    const bool ready = mbar_wait(bar0 + 8 * slot, (iter / kRtRing) & 1, b.wait_limit_us);
    if (!__all_sync(kFullMask, ready)) {
      // Give up: record it, wait (bounded) for this warp's copies in flight
      // so that none lands in freed shared memory, and leave.
      if constexpr (RtCfg<K>::kLaneCopies) {  // this lane's copies landed
        cp_async_commit();
        cp_async_wait<0>();
      }
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
    if constexpr (RtCfg<K>::kLaneCopies) {
      __syncwarp();  // every lane's reads of the slot before its refill
      const int64_t next = chunk + kRtRing * stride;
      if (next < b.total_chunks) issue_all(next, slot);
    } else {
      fence_proxy_async_smem();  // this lane's reads before the next async write of the slot
      __syncwarp();
      if (lane == 0) {
        const int64_t next = chunk + kRtRing * stride;
        if (next < b.total_chunks) issue(next, slot);
      }
    }
    const int m = item_of(chunk, m_work);
    const ReconstructItem& it = b.item[m];

    const bool all_ok = __all_sync(kFullMask, ok);
    if constexpr (RtCfg<K>::kOuter) {
      if (stored && lane == 0) bulk_wait_read<0>();  // the previous chunk's store has read the buffer
      __syncwarp();
      uint8_t* row = out_stage + lane * 128;
      // Weights in 16-byte output pieces: piece q holds code bytes 2q and 2q+1
      // (8 weights), each summed over all k stages before the next, so that
      // only a few accumulators are live.  form(i, h, b8, a01, a23) adds stage
      // i's levels of the four codes of byte b8 (group half h) in stage order.
      auto run = [&](auto form) {
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          uint32_t hw[4];
#pragma unroll
          for (int jj = 0; jj < 2; ++jj) {
            const int j = 2 * q + jj;
            constexpr int kBytesPerHalf = 16 / NH;
            const int h = j / kBytesPerHalf;
            f32x2 a01, a23;
#pragma unroll
            for (int i = 0; i < K; ++i) {
              const uint32_t w = (j >> 2) == 0 ? code[i].x : (j >> 2) == 1 ? code[i].y : (j >> 2) == 2 ? code[i].z : code[i].w;
              const uint32_t b8 = (j & 3) == 0 ? w : (w >> (8 * (j & 3)));
              form(i, h, b8, a01, a23);
            }
            float x, y;
            unpack2(a01, x, y);
            __nv_bfloat162 v = __floats2bfloat162_rn(x, y);
            hw[2 * jj] = *reinterpret_cast<const uint32_t*>(&v);
            unpack2(a23, x, y);
            v = __floats2bfloat162_rn(x, y);
            hw[2 * jj + 1] = *reinterpret_cast<const uint32_t*>(&v);
          }
          *reinterpret_cast<uint4*>(row + ((q ^ (lane & 7)) << 4)) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
        }
      };
      if constexpr (kSym) {
        run([&](int i, int h, uint32_t b8, f32x2& a01, f32x2& a23) {
          const f32x2 S = pack2(scale[i][h], scale[i][h]);
          f32x2 u01, u23;
          sym_offsets(b8, u01, u23);
          a01 = (i == 0) ? mul2(u01, S) : fma2(u01, S, a01);
          a23 = (i == 0) ? mul2(u23, S) : fma2(u23, S, a23);
        });
      } else if (all_ok) {
        StageConsts cs[K][NH];
#pragma unroll
        for (int i = 0; i < K; ++i)
#pragma unroll
          for (int h = 0; h < NH; ++h) cs[i][h] = stage_consts(scale[i][h], zero[i][h]);
        run([&](int i, int h, uint32_t b8, f32x2& a01, f32x2& a23) {
          f32x2 l01, l23;
          asym_levels(b8, cs[i][h], l01, l23);
          a01 = (i == 0) ? l01 : add2(a01, l01);
          a23 = (i == 0) ? l23 : add2(a23, l23);
        });
      } else {  // a scale outside [2^-100, 2^100] in the warp: fl(Q s) as a plain (t - 2^23) s
        run([&](int i, int h, uint32_t b8, f32x2& a01, f32x2& a23) {
          const f32x2 Z = pack2(zero[i][h], zero[i][h]), S = pack2(scale[i][h], scale[i][h]);
          const f32x2 T23 = pack2(kTwo23, kTwo23), Z0 = pack2(0.0f, 0.0f);
          const f32x2 t01 = pack2u(magic23<3u>(b8), magic23<3u>(b8 >> 2));
          const f32x2 t23 = pack2u(magic23<3u>(b8 >> 4), magic23<3u>(b8 >> 6));
          const f32x2 l01 = add2(Z, fma2(sub2(t01, T23), S, Z0));
          const f32x2 l23 = add2(Z, fma2(sub2(t23, T23), S, Z0));
          a01 = (i == 0) ? l01 : add2(a01, l01);
          a23 = (i == 0) ? l23 : add2(a23, l23);
        });
      }
    } else {
      f32x2 acc[32];
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
    }
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
                                                                  RtCfg<K>::kThreads, rt_smem_bytes<G, K, F>());
    if (e != cudaSuccess) return e;
    if (blocks_per_sm < 1) blocks_per_sm = 1;
    cached.store(blocks_per_sm, std::memory_order_relaxed);
  }
  const int64_t want = (p.b.total_chunks + RtCfg<K>::kWarps - 1) / RtCfg<K>::kWarps;
  const int64_t cap = static_cast<int64_t>(sms) * blocks_per_sm;
  const int grid = static_cast<int>(want < cap ? want : cap);
  reconstruct_tile_kernel<G, K, F><<<grid, RtCfg<K>::kThreads, rt_smem_bytes<G, K, F>(), stream>>>(p);
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
