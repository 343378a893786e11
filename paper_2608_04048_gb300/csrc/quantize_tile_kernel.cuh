// RRQ package construction, wide-lane form (sm_103a): the same arithmetic as
// quantize_kernel.cuh (Section 3.1 Eq. 1-3 per stage, Section 3.2 Eq. 4-7 and
// Algorithm 1 for the recursion; the two-float quotient and its exactness
// argument are described there), laid out for fewer instructions per weight.
//
// Work decomposition.  A warp owns a chunk of 32 * LW consecutive weights of
// one matrix; lane l owns the LW consecutive weights [l * LW, (l + 1) * LW) of
// it.  A matrix is viewed as a 2-D array [n / LW, LW] of bf16 and each chunk
// is one 2-D TMA tile of 32 rows x LW columns, loaded with the 128-byte (LW =
// 64) or 64-byte (LW = 32) swizzle: row r's 16-byte piece c lands at piece
// c ^ (r & 7) (c ^ ((r >> 1) & 3)) of its row, so the eight lanes of a
// quarter warp that read piece c of their own rows touch eight different
// bank groups and every lane reads its weights in natural order.  Rows past
// the end of a matrix arrive as zeros and store nothing.
//
// Per stage a lane packs the 2-bit codes of its LW weights with funnel shifts
// into LW / 16 words in natural order (element e at bits 2e of word e / 16)
// and writes them with one 16-byte (8-byte) store; the lane that holds the
// start of a group writes its scale (and zero).  Group reductions: groups of
// 32 weights sit two to a lane at LW = 64 (no shuffle), groups of 64 one to a
// lane, groups of 128 and 256 over 2 and 4 lanes.  The stage loop is unrolled
// so that every stage's output pointers are compile-time offsets into the
// matrix descriptor.
#pragma once

#include <atomic>

#include "quantize_kernel.cuh"

namespace rrq {
namespace {

template <int LW>
struct Tile {
  static constexpr int kPairs = LW / 2;        // f32x2 pairs per lane
  static constexpr int kPieces = LW / 8;       // 16-byte pieces of bf16 per lane
  static constexpr int kChunk = 32 * LW;       // weights per warp chunk (one TMA tile)
  static constexpr int kBytes = kChunk * 2;    // bytes per tile
  static constexpr int kWords = LW / 16;       // 32-bit code words per lane and stage
  static constexpr uint32_t kSwz = LW == 64 ? 7u : 3u;
  static constexpr int kRowShift = LW == 64 ? 0 : 1;
};

#ifndef RRQ_TILE_RING
#define RRQ_TILE_RING 3
#endif
#ifndef RRQ_TILE_CTAS_PER_SM
#define RRQ_TILE_CTAS_PER_SM 2
#endif
#ifndef RRQ_TILE_UNROLL_STAGES
#define RRQ_TILE_UNROLL_STAGES 0
#endif
constexpr int kTileWarps = 8;
constexpr int kTileThreads = kTileWarps * 32;
constexpr int kTileRing = RRQ_TILE_RING;       // TMA tiles in flight per warp

template <int LW>
constexpr int tile_smem_bytes() {
  return kTileWarps * kTileRing * Tile<LW>::kBytes + kTileWarps * kTileRing * 8 + 1024;  // + alignment slack
}

// 2-D tiled TMA load of box (x, y) of `map` into this CTA's shared memory.
__device__ __forceinline__ void tma_tile_load(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

// lo = -0 instead of +0 where a group's minimum is zero and it holds a -0
// (the definition orders -0 before +0); NH groups per lane, L lanes per group
template <int NH, int L, int P>
__device__ __forceinline__ void signed_zero_min(const f32x2 (&v)[P], float (&lo)[NH]) {
  bool any_zero = false;
#pragma unroll
  for (int h = 0; h < NH; ++h) any_zero |= lo[h] == 0.0f;
  if (__any_sync(kFullMask, any_zero)) {
    constexpr int PH = P / NH;
#pragma unroll
    for (int h = 0; h < NH; ++h) {
      uint32_t neg = 0;
      if (lo[h] == 0.0f) {
#pragma unroll
        for (int i = h * PH; i < (h + 1) * PH; ++i)
          neg |= (static_cast<uint32_t>(v[i]) == 0x80000000u) | (static_cast<uint32_t>(v[i] >> 32) == 0x80000000u);
      }
      neg = group_or<L>(neg);
      if (lo[h] == 0.0f) lo[h] = neg ? -0.0f : 0.0f;
    }
  }
}

// One chunk of a lane: every stage of the asymmetric grid (binary32 scale and
// zero), stores of codes, scales and zeros (valid lanes only).
template <int G, int LW>
__device__ __forceinline__ void tile_chunk_asym(const QuantizeBatch& p, const QuantizeItem& it, int64_t e0,
                                                bool valid, int lane, const uint4 (&raw)[Tile<LW>::kPieces]) {
  using T = Tile<LW>;
  constexpr int NH = G < LW ? LW / G : 1;      // groups per lane
  constexpr int L = G > LW ? G / LW : 1;       // lanes per group
  constexpr int PH = T::kPairs / NH;           // pairs per group and lane
  f32x2 v[T::kPairs];
#pragma unroll
  for (int j = 0; j < T::kPieces; ++j) {
    const uint32_t w4[4] = {raw[j].x, raw[j].y, raw[j].z, raw[j].w};
#pragma unroll
    for (int m = 0; m < 4; ++m) v[4 * j + m] = pack2u(w4[m] << 16, w4[m] & 0xffff0000u);
  }
  float lo[NH], hi[NH];
#pragma unroll
  for (int h = 0; h < NH; ++h) {
    float a, b, c, d;
    unpack2(v[h * PH], a, b);
    unpack2(v[h * PH + 1], c, d);
    float lo0 = fminf(a, b), hi0 = fmaxf(a, b), lo1 = fminf(c, d), hi1 = fmaxf(c, d);
#pragma unroll
    for (int i = h * PH + 2; i < (h + 1) * PH; i += 2) {
      unpack2(v[i], a, b);
      unpack2(v[i + 1], c, d);
      lo0 = min3(lo0, a, b);
      hi0 = max3(hi0, a, b);
      lo1 = min3(lo1, c, d);
      hi1 = max3(hi1, c, d);
    }
    lo[h] = fminf(lo0, lo1);
    hi[h] = fmaxf(hi0, hi1);
    group_minmax<L>(lo[h], hi[h]);
  }
  const int64_t g0 = e0 / G;                   // first group of this lane
  const bool writes_meta = valid && (L == 1 || (lane & (L - 1)) == 0);
  const bool force_exact = (p.flags & kDebugForceExact) != 0;

#if RRQ_TILE_UNROLL_STAGES
#pragma unroll
#else
#pragma unroll 1
#endif
  for (int k = 0; k < kMaxStages; ++k) {
    if (k >= p.n_stages) break;
    signed_zero_min<NH, L>(v, lo);
    float s[NH], r_hi[NH], r_lo[NH];
    bool fast = !force_exact;
#pragma unroll
    for (int h = 0; h < NH; ++h) {
      s[h] = div3(__fsub_rn(hi[h], lo[h]));
      fast = fast && (s[h] == 0.0f || corrected_quotient_safe(s[h]));
      recip2(s[h], r_hi[h], r_lo[h]);
      if (!(s[h] > 0.0f)) r_hi[h] = r_lo[h] = 0.0f;  // s = 0: every quotient 0
    }
    uint32_t acc[T::kWords];
#pragma unroll
    for (int w = 0; w < T::kWords; ++w) acc[w] = 0u;
    float mn[NH][2], mx[NH][2];
#pragma unroll
    for (int h = 0; h < NH; ++h) {
      mn[h][0] = mn[h][1] = __int_as_float(0x7f800000);
      mx[h][0] = mx[h][1] = __int_as_float(0xff800000);
    }
    const bool last = k + 1 == p.n_stages;  // its residual and range are never used
    if (fast && last) {
#pragma unroll
      for (int h = 0; h < NH; ++h) {
        const f32x2 LO = pack2(lo[h], lo[h]), RH = pack2(r_hi[h], r_hi[h]), RL = pack2(r_lo[h], r_lo[h]);
        const f32x2 T23 = pack2(kTwo23, kTwo23);
#pragma unroll
        for (int i = h * PH; i < (h + 1) * PH; ++i) {
          const f32x2 d = sub2(v[i], LO);
          const f32x2 t = add2(fma2(d, RH, mul2(d, RL)), T23);  // 2^23 + rhe(d/s)
          acc[i >> 3] = push_code(push_code(acc[i >> 3], static_cast<uint32_t>(t)), static_cast<uint32_t>(t >> 32));
        }
      }
    } else if (fast) {
#pragma unroll
      for (int h = 0; h < NH; ++h) {
        const float c = __fmul_rn(-kTwo23, s[h]);  // exact: power-of-two scaling
        const f32x2 LO = pack2(lo[h], lo[h]), RH = pack2(r_hi[h], r_hi[h]), RL = pack2(r_lo[h], r_lo[h]);
        const f32x2 S = pack2(s[h], s[h]), C = pack2(c, c), T23 = pack2(kTwo23, kTwo23);
#pragma unroll
        for (int i = h * PH; i < (h + 1) * PH; ++i) {
          const f32x2 d = sub2(v[i], LO);
          const f32x2 q = fma2(d, RH, mul2(d, RL));  // d/s to 2^-45.3
          const f32x2 t = add2(q, T23);              // 2^23 + rhe(q)
          const f32x2 lv = add2(LO, fma2(t, S, C));  // fl(lo + fl(Q*s))
          v[i] = sub2(v[i], lv);                     // v - fl(lo + fl(Q*s))
          acc[i >> 3] = push_code(push_code(acc[i >> 3], static_cast<uint32_t>(t)), static_cast<uint32_t>(t >> 32));
          float a, b;
          unpack2(v[i], a, b);
          mn[h][i & 1] = min3(mn[h][i & 1], a, b);
          mx[h][i & 1] = max3(mx[h][i & 1], a, b);
        }
      }
    } else {  // IEEE division element by element (scales next to a rounding boundary, or forced)
#pragma unroll
      for (int h = 0; h < NH; ++h) {
#pragma unroll
        for (int i = h * PH; i < (h + 1) * PH; ++i) {
          const ExactPair x = exact_pair(v[i], lo[h], s[h]);
          v[i] = x.w;
          acc[i >> 3] = push_code(push_code(acc[i >> 3], x.q0), x.q1);
          float a, b;
          unpack2(v[i], a, b);
          mn[h][i & 1] = min3(mn[h][i & 1], a, b);
          mx[h][i & 1] = max3(mx[h][i & 1], a, b);
        }
      }
    }
    if (valid) {
      uint8_t* cp = it.codes[k] + (e0 >> 2);
      if constexpr (T::kWords == 4)
        __stcs(reinterpret_cast<uint4*>(cp), make_uint4(acc[0], acc[1], acc[2], acc[3]));
      else
        __stcs(reinterpret_cast<uint2*>(cp), make_uint2(acc[0], acc[1]));
    }
    if (writes_meta) {
      float* sp = static_cast<float*>(it.scales[k]) + g0;
      float* zp = it.zeros[k] + g0;
      if constexpr (NH == 2) {
        __stcs(reinterpret_cast<float2*>(sp), make_float2(s[0], s[1]));
        __stcs(reinterpret_cast<float2*>(zp), make_float2(lo[0], lo[1]));
      } else {
        __stcs(sp, s[0]);
        __stcs(zp, lo[0]);
      }
    }
    if (k + 1 < p.n_stages) {  // the residual's range is the next stage's
#pragma unroll
      for (int h = 0; h < NH; ++h) {
        lo[h] = fminf(mn[h][0], mn[h][1]);
        hi[h] = fmaxf(mx[h][0], mx[h][1]);
        group_minmax<L>(lo[h], hi[h]);
      }
    }
  }
}

// One chunk of a lane on the symmetric grid (implicit zero-point 2); kF16:
// the scale is rounded to binary16, stored so, and quantized against.
template <int G, int LW, bool kF16>
__device__ __forceinline__ void tile_chunk_sym(const QuantizeBatch& p, const QuantizeItem& it, int64_t e0,
                                               bool valid, int lane, const uint4 (&raw)[Tile<LW>::kPieces]) {
  using T = Tile<LW>;
  constexpr int NH = G < LW ? LW / G : 1;
  constexpr int L = G > LW ? G / LW : 1;
  constexpr int PH = T::kPairs / NH;
  f32x2 v[T::kPairs];
#pragma unroll
  for (int j = 0; j < T::kPieces; ++j) {
    const uint32_t w4[4] = {raw[j].x, raw[j].y, raw[j].z, raw[j].w};
#pragma unroll
    for (int m = 0; m < 4; ++m) v[4 * j + m] = pack2u(w4[m] << 16, w4[m] & 0xffff0000u);
  }
  float amax[NH];
#pragma unroll
  for (int h = 0; h < NH; ++h) {
    float m0 = 0.0f, m1 = 0.0f;
#pragma unroll
    for (int i = h * PH; i < (h + 1) * PH; i += 2) {
      float a, b, c, d;
      unpack2(v[i], a, b);
      unpack2(v[i + 1], c, d);
      m0 = max3(m0, fabsf(a), fabsf(b));
      m1 = max3(m1, fabsf(c), fabsf(d));
    }
    amax[h] = group_max<L>(fmaxf(m0, m1));
  }
  const int64_t g0 = e0 / G;
  const bool writes_meta = valid && (L == 1 || (lane & (L - 1)) == 0);
  const bool force_exact = (p.flags & kDebugForceExact) != 0;

#if RRQ_TILE_UNROLL_STAGES
#pragma unroll
#else
#pragma unroll 1
#endif
  for (int k = 0; k < kMaxStages; ++k) {
    if (k >= p.n_stages) break;
    float s[NH], r_hi[NH], r_lo[NH];
    uint16_t s16[NH];
    bool fast = !force_exact;
#pragma unroll
    for (int h = 0; h < NH; ++h) {
      s[h] = div3(__fmul_rn(amax[h], 2.0f));  // 2 * amax is exact
      s16[h] = 0;
      if (kF16) {
        s16[h] = __half_as_ushort(__float2half_rn(s[h]));
        s[h] = __half2float(__ushort_as_half(s16[h]));
      }
      fast = fast && (kF16 || s[h] == 0.0f || corrected_quotient_safe(s[h]));
      recip2(s[h], r_hi[h], r_lo[h]);
      if (!(s[h] > 0.0f)) r_hi[h] = r_lo[h] = 0.0f;
    }
    uint32_t acc[T::kWords];
#pragma unroll
    for (int w = 0; w < T::kWords; ++w) acc[w] = 0u;
    float mx[NH][2];
#pragma unroll
    for (int h = 0; h < NH; ++h) mx[h][0] = mx[h][1] = 0.0f;
    const bool last = k + 1 == p.n_stages;  // its residual and range are never used
    if (fast && last) {
#pragma unroll
      for (int h = 0; h < NH; ++h) {
        const f32x2 RH = pack2(r_hi[h], r_hi[h]), RL = pack2(r_lo[h], r_lo[h]);
        const f32x2 C = pack2(kSymRound, kSymRound);
#pragma unroll
        for (int i = h * PH; i < (h + 1) * PH; ++i) {
          const f32x2 q = fma2(v[i], RH, mul2(v[i], RL));
          float qa, qb;
          unpack2(q, qa, qb);
          const f32x2 t = add2(pack2(fminf(qa, 1.0f), fminf(qb, 1.0f)), C);
          acc[i >> 3] = push_code(push_code(acc[i >> 3], static_cast<uint32_t>(t)), static_cast<uint32_t>(t >> 32));
        }
      }
    } else if (fast) {
#pragma unroll
      for (int h = 0; h < NH; ++h) {
        const f32x2 RH = pack2(r_hi[h], r_hi[h]), RL = pack2(r_lo[h], r_lo[h]), NS = pack2(-s[h], -s[h]);
        const f32x2 C = pack2(kSymRound, kSymRound);
#pragma unroll
        for (int i = h * PH; i < (h + 1) * PH; ++i) {
          const f32x2 q = fma2(v[i], RH, mul2(v[i], RL));  // v/s to 2^-45.3
          float qa, qb;
          unpack2(q, qa, qb);
          const f32x2 t = add2(pack2(fminf(qa, 1.0f), fminf(qb, 1.0f)), C);  // C + rhe, clamped
          v[i] = fma2(sub2(t, C), NS, v[i]);                                // v - (Q-2) s
          acc[i >> 3] = push_code(push_code(acc[i >> 3], static_cast<uint32_t>(t)), static_cast<uint32_t>(t >> 32));
          float a, b;
          unpack2(v[i], a, b);
          mx[h][i & 1] = max3(mx[h][i & 1], fabsf(a), fabsf(b));
        }
      }
    } else {
#pragma unroll
      for (int h = 0; h < NH; ++h) {
#pragma unroll
        for (int i = h * PH; i < (h + 1) * PH; ++i) {
          const ExactPair x = exact_pair_sym(v[i], s[h]);
          v[i] = x.w;
          acc[i >> 3] = push_code(push_code(acc[i >> 3], x.q0), x.q1);
          float a, b;
          unpack2(v[i], a, b);
          mx[h][i & 1] = max3(mx[h][i & 1], fabsf(a), fabsf(b));
        }
      }
    }
    if (valid) {
      uint8_t* cp = it.codes[k] + (e0 >> 2);
      if constexpr (T::kWords == 4)
        __stcs(reinterpret_cast<uint4*>(cp), make_uint4(acc[0], acc[1], acc[2], acc[3]));
      else
        __stcs(reinterpret_cast<uint2*>(cp), make_uint2(acc[0], acc[1]));
    }
    if (writes_meta) {
      if (kF16) {
        uint16_t* sp = static_cast<uint16_t*>(it.scales[k]) + g0;
        if constexpr (NH == 2)
          __stcs(reinterpret_cast<unsigned int*>(sp), static_cast<unsigned int>(s16[0]) | (static_cast<unsigned int>(s16[1]) << 16));
        else
          stcs_u16(sp, s16[0]);
      } else {
        float* sp = static_cast<float*>(it.scales[k]) + g0;
        if constexpr (NH == 2)
          __stcs(reinterpret_cast<float2*>(sp), make_float2(s[0], s[1]));
        else
          __stcs(sp, s[0]);
      }
    }
    if (k + 1 < p.n_stages) {
#pragma unroll
      for (int h = 0; h < NH; ++h) amax[h] = group_max<L>(fmaxf(mx[h][0], mx[h][1]));
    }
  }
}

// Persistent grid; warps take the chunks of all matrices of the launch in
// turn, each streaming its tiles through a private ring of kTileRing buffers.
template <int G, int F, int LW>
__global__ void __launch_bounds__(kTileThreads, RRQ_TILE_CTAS_PER_SM) quantize_tile_kernel(const __grid_constant__ QuantizeTileBatch p) {
  using T = Tile<LW>;
  extern __shared__ uint8_t smem_raw[];
  // 128-byte swizzled tiles: buffers on a 1024-byte boundary
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const QuantizeBatch& b = p.b;
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  uint8_t* ring = smem + warp * (kTileRing * T::kBytes);
  const uint32_t ring_s = smem_u32(ring);
  const uint32_t bar0 = smem_u32(smem + kTileWarps * kTileRing * T::kBytes) + warp * kTileRing * 8;

  const int64_t first = static_cast<int64_t>(blockIdx.x) * kTileWarps + warp;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kTileWarps;
  if (first >= b.total_chunks) return;  // warp-uniform: nothing issued, nothing to wait for

  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < kTileRing; ++i) mbar_init(bar0 + 8 * i, 1);
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
    const int row = static_cast<int>((chunk - b.item[m].chunk_begin) * 32);
    mbar_arrive_expect_tx(bar0 + 8 * slot, T::kBytes);
    tma_tile_load(ring_s + slot * T::kBytes, &p.w[m], 0, row, bar0 + 8 * slot);
  };
  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < kTileRing; ++i) {
      const int64_t c = first + i * stride;
      if (c < b.total_chunks) issue(c, i);
    }
  }

  // this lane's row of a tile: 16-byte piece j at piece j ^ (row bits)
  const uint32_t swz = (static_cast<uint32_t>(lane) >> T::kRowShift) & T::kSwz;
  uint32_t iter = 0;
  for (int64_t chunk = first; chunk < b.total_chunks; chunk += stride, ++iter) {
    const int slot = iter % kTileRing;
    const bool ready = mbar_wait(bar0 + 8 * slot, (iter / kTileRing) & 1, b.wait_limit_us);
    if (!__all_sync(kFullMask, ready)) {
      // Give up: record it, wait (bounded) for this warp's tiles in flight so
      // that none lands in freed shared memory, and leave.
      if (lane == 0) {
        atomicOr(b.status, kStatusTimeout);
        for (int j = 0; j < kTileRing; ++j) {
          if (chunk + j * stride >= b.total_chunks) break;
          const uint32_t jt = iter + j;
          mbar_wait(bar0 + 8 * (jt % kTileRing), (jt / kTileRing) & 1, kDrainLimitUs);
        }
      }
      __syncwarp();
      return;
    }
    const uint8_t* row = ring + slot * T::kBytes + lane * (LW * 2);
    uint4 raw[T::kPieces];
#pragma unroll
    for (int j = 0; j < T::kPieces; ++j) raw[j] = *reinterpret_cast<const uint4*>(row + ((j ^ swz) << 4));
    fence_proxy_async_smem();  // this lane's reads before the next tile's async write
    __syncwarp();
    if (lane == 0) {
      const int64_t next = chunk + kTileRing * stride;
      if (next < b.total_chunks) issue(next, slot);
    }
    const int m = item_of(chunk, m_work);
    const QuantizeItem& it = b.item[m];
    const int64_t e0 = (chunk - it.chunk_begin) * T::kChunk + static_cast<int64_t>(lane) * LW;
    const bool valid = e0 < it.n;
    if constexpr (F == kAsymF32)
      tile_chunk_asym<G, LW>(b, it, e0, valid, lane, raw);
    else
      tile_chunk_sym<G, LW, F == kSymF16>(b, it, e0, valid, lane, raw);
  }
}

template <int G, int F, int LW>
cudaError_t tile_launch_gf(const QuantizeTileBatch& p, cudaStream_t stream, int sms) {
  // resident CTAs per multiprocessor: the same for every device of this
  // build, asked once (an atomic: any thread may launch)
  static std::atomic<int> cached{0};
  int blocks_per_sm = cached.load(std::memory_order_relaxed);
  if (blocks_per_sm == 0) {
    int n = 0;
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, quantize_tile_kernel<G, F, LW>, kTileThreads,
                                                                  tile_smem_bytes<LW>());
    if (e != cudaSuccess) return e;
    blocks_per_sm = n < 1 ? 1 : n;
    cached.store(blocks_per_sm, std::memory_order_relaxed);
  }
  const int64_t want = (p.b.total_chunks + kTileWarps - 1) / kTileWarps;
  const int64_t cap = static_cast<int64_t>(sms) * blocks_per_sm;
  const int grid = static_cast<int>(want < cap ? want : cap);
  quantize_tile_kernel<G, F, LW><<<grid, kTileThreads, tile_smem_bytes<LW>(), stream>>>(p);
  return cudaGetLastError();
}

template <int F, int LW>
cudaError_t tile_launch_f(int group, const QuantizeTileBatch& p, cudaStream_t stream, int sms) {
  switch (group) {
    case 32: return tile_launch_gf<32, F, LW>(p, stream, sms);
    case 64: return tile_launch_gf<64, F, LW>(p, stream, sms);
    case 128: return tile_launch_gf<128, F, LW>(p, stream, sms);
    case 256: return tile_launch_gf<256, F, LW>(p, stream, sms);
    default: return cudaErrorInvalidValue;
  }
}

template <int F, int LW>
cudaError_t tile_prepare_f() {
  cudaError_t e;
  const cudaFuncAttribute a = cudaFuncAttributeMaxDynamicSharedMemorySize;
  if ((e = cudaFuncSetAttribute(quantize_tile_kernel<32, F, LW>, a, tile_smem_bytes<LW>()))) return e;
  if ((e = cudaFuncSetAttribute(quantize_tile_kernel<64, F, LW>, a, tile_smem_bytes<LW>()))) return e;
  if ((e = cudaFuncSetAttribute(quantize_tile_kernel<128, F, LW>, a, tile_smem_bytes<LW>()))) return e;
  return cudaFuncSetAttribute(quantize_tile_kernel<256, F, LW>, a, tile_smem_bytes<LW>());
}

}  // namespace
}  // namespace rrq
