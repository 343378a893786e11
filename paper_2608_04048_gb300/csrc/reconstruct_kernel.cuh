// RRQ prefix reconstruction (Section 3.2 Eq. 8; Appendix C): the bf16 weight
// at operating point k (k = 1..4 -> 2/4/6/8 bits) is
//     acc = L_0;  acc = fl(acc + L_i) for i = 1..k-1;  out = bf16_rne(acc)
// with L_i = fl(zero_i + fl(Q_i * scale_i)) the dequantized value of stage i.
//
// A warp owns a chunk of 1024 consecutive weights of one matrix, a lane owns
// 32 consecutive weights (one 8-byte code word per stage, one scale and one
// zero per stage).  The chunks of all matrices of a launch form one sequence
// taken in turn by the warps of a persistent grid.  Each lane copies its code
// words and metadata asynchronously (cp.async) into a per-warp ring of
// shared-memory buffers kRing - 1 chunks ahead of use, so that many chunks'
// loads are in flight without holding registers; the 2 KiB of bf16 output of
// a chunk is staged in shared memory and written by a 1-D bulk copy (TMA
// store), double-buffered per warp.
//
// fl(Q*s) is one fused multiply-add: code j of a byte stays in its bit field
// under the exponent of 2^(23-2j), so that the float t = 2^(23-2j) + Q
// exactly, and fma(t, s, -2^(23-2j) s) = RN(Q*s) because the scaling by a
// power of two is exact for s in [2^-100, 2^100] (asym_levels).  So the four
// codes of one byte need one shift per byte and one logic operation per code.
// Groups with a scale outside that range use the plain form RN((t - 2^23) s).
//
// Symmetric grid (implicit zero-point 2): L_i = (Q_i - 2) * s_i, exact in
// binary32, so acc + L_i is one fma(u, s, acc) with u = Q - 2 taken exactly
// from the same t (sym_offsets), for every scale; the base stage is the
// exact product u * s.  binary16 scales are read as the 4-byte word holding
// the lane's scale and its neighbour's (the copy is cut to 2 bytes at the end
// of an array with an odd number of groups) and widened exactly.
//
// Heterogeneous stage widths (kAsymBits): a lane copies the 4b bytes of its
// b-bit codes per stage, extracts each code by shift and mask and forms
// fl(zero + fl(Q s)) as fma(t - 2^23, s, 0) + zero; values are kept in natural
// order.
//
// This header holds the kernel template; reconstruct_asym_f32.cu,
// reconstruct_sym_f32.cu, reconstruct_sym_f16.cu and reconstruct_asym_bits.cu
// each instantiate one package format (they compile in parallel).
#pragma once

#include <atomic>

#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "rrq_device.cuh"

namespace rrq {
namespace {

constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;
constexpr int kRing = 4;               // chunks of inputs per warp in shared memory
constexpr float kTwo23 = 8388608.0f;   // bits 0x4B000000 | q encode 2^23 + q for 0 <= q < 2^23

// One stage of one chunk in shared memory: codes (8 B per lane, 16 B for the
// heterogeneous-width format), then scales 128 B, zeros 128 B.
template <int F>
__host__ __device__ constexpr int code_bytes() { return F == kAsymBits ? 512 : 256; }
template <int F>
__host__ __device__ constexpr int stage_bytes() { return code_bytes<F>() + 256; }
template <int K, int F>
__host__ __device__ constexpr int warp_smem_bytes() { return kRing * K * stage_bytes<F>() + 2 * kChunkBytes; }
template <int K, int F>
__host__ __device__ constexpr int smem_bytes() { return kWarps * warp_smem_bytes<K, F>(); }


// kAllPrefixes: write the reconstruction after every stage i < K (prefixes
// 1..K in one pass over the package) instead of only after stage K-1.
template <int G, int K, bool kAllPrefixes, int F>
__global__ void __launch_bounds__(kThreads, 2) reconstruct_kernel(const __grid_constant__ ReconstructBatch p) {
  constexpr bool kSym = F == kSymF32 || F == kSymF16;
  constexpr bool kF16 = F == kSymF16;
  extern __shared__ __align__(128) uint8_t smem[];
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  constexpr int kStageBytes = stage_bytes<F>();
  constexpr int kCB = code_bytes<F>();
  uint8_t* ring = smem + warp * warp_smem_bytes<K, F>();
  uint8_t* stage_buf = ring + kRing * K * kStageBytes;
  constexpr int kBufBytes = K * kStageBytes;

  const int64_t first = static_cast<int64_t>(blockIdx.x) * kWarps + warp;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kWarps;
  if (first >= p.total_chunks) return;

  // Slot j of a lane handles its 16-byte output piece (j + rot) & 3, so that
  // the shared-memory stores of a quarter warp hit distinct bank groups; the
  // code words are rotated right by 16*rot bits to match.
  const int rot = F == kAsymBits ? 0 : (lane >> 1) & 3;
  const uint32_t sel_lo = rot == 0 ? 0x3210u : rot == 1 ? 0x5432u : rot == 2 ? 0x7654u : 0x1076u;
  const uint32_t sel_hi = rot == 0 ? 0x7654u : rot == 1 ? 0x1076u : rot == 2 ? 0x3210u : 0x5432u;

  int m_load = 0, m_work = 0;
  auto item_of = [&](int64_t chunk, int& m) -> const ReconstructItem& {
    while (m + 1 < p.count && chunk >= p.item[m + 1].chunk_begin) ++m;
    return p.item[m];
  };

  // Copies this lane's inputs of `chunk` into ring buffer `buf` (one commit
  // group per call, empty past the end; lanes past a matrix's end get zeros).
  auto issue = [&](int64_t chunk, int buf) {
    if (chunk < p.total_chunks) {
      const ReconstructItem& it = item_of(chunk, m_load);
      const int64_t e = (chunk - it.chunk_begin) * kChunkElems + static_cast<int64_t>(lane) * kLaneElems;
      const bool valid = e < it.n;  // false only in the last chunk of a matrix
      // byte offsets shared by every stage's arrays (invalid lanes read nothing)
      const uint64_t off_code = valid ? static_cast<uint64_t>(e) >> 2 : 0;
      const uint64_t gi = static_cast<uint64_t>(e) / G;
      uint64_t off_meta = valid ? gi * 4 : 0;
      uint32_t n_scale = valid ? 4u : 0u;
      if (kF16) {  // the aligned 4-byte word holding this group's 2-byte scale
        off_meta = valid ? (gi * 2) & ~uint64_t{3} : 0;
        const uint64_t left = static_cast<uint64_t>(it.n / G) * 2 - off_meta;
        n_scale = valid ? (left < 4 ? 2u : 4u) : 0u;
      }
      const uint32_t n8 = valid ? 8u : 0u, n4 = valid ? 4u : 0u;
      const uint32_t base = smem_u32(ring + buf * K * kStageBytes) + lane * (F == kAsymBits ? 16 : 8);
      const uint32_t mbase = smem_u32(ring + buf * K * kStageBytes) + kCB + lane * 4;
#pragma unroll
      for (int i = 0; i < K; ++i) {
        if (F == kAsymBits) {  // 4b bytes of b-bit codes for the lane's 32 weights
          const int b = p.bits[i];
          const char* src = reinterpret_cast<const char*>(it.codes[i]) + (valid ? (static_cast<uint64_t>(e) >> 5) * 4 * b : 0);
          const uint32_t dst = base + i * kStageBytes;
          if (b == 4) cp_async_16(dst, src, valid ? 16u : 0u);
          else if (b == 2) cp_async_8(dst, src, n8);
          else {
            cp_async_4(dst, src, n4);
            if (b == 3) {
              cp_async_4(dst + 4, src + 4, n4);
              cp_async_4(dst + 8, src + 8, n4);
            }
          }
        } else {
          cp_async_8(base + i * kStageBytes, reinterpret_cast<const char*>(it.codes[i]) + off_code, n8);
        }
        cp_async_4(mbase + i * kStageBytes, reinterpret_cast<const char*>(it.scales[i]) + off_meta, n_scale);
        if (!kSym)
          cp_async_4(mbase + i * kStageBytes + 128, reinterpret_cast<const char*>(it.zeros[i]) + off_meta, n4);
      }
    }
    cp_async_commit();
  };

#pragma unroll
  for (int j = 0; j < kRing - 1; ++j) issue(first + j * stride, j);

  uint32_t iter = 0, n_store = 0;
  for (int64_t chunk = first; chunk < p.total_chunks; chunk += stride, ++iter) {
    issue(chunk + (kRing - 1) * stride, (iter + kRing - 1) % kRing);
    cp_async_wait<kRing - 1>();  // this lane's copies of `chunk` have landed

    const uint8_t* buf = ring + (iter % kRing) * kBufBytes;
    uint2 code[K];
    float scale[K], zero[K];
    bool ok = true;
#pragma unroll
    for (int i = 0; i < K; ++i) {
      code[i] = F == kAsymBits ? make_uint2(0u, 0u) : *reinterpret_cast<const uint2*>(buf + i * kStageBytes + lane * 8);
      if (kF16) {
        // group index parity of this lane: chunks start on an even group
        const uint32_t w = *reinterpret_cast<const uint32_t*>(buf + i * kStageBytes + kCB + lane * 4);
        const uint32_t h = ((lane / (G / 32)) & 1) ? (w >> 16) : (w & 0xffffu);
        scale[i] = __half2float(__ushort_as_half(static_cast<unsigned short>(h)));
      } else {
        scale[i] = *reinterpret_cast<const float*>(buf + i * kStageBytes + kCB + lane * 4);
      }
      zero[i] = kSym ? 0.0f : *reinterpret_cast<const float*>(buf + i * kStageBytes + kCB + 128 + lane * 4);
      ok = ok && (kSym || prescale_ok(scale[i]));  // symmetric levels need no condition
    }

    const bool all_ok = __all_sync(kFullMask, ok);
    const ReconstructItem& it = item_of(chunk, m_work);
    const int64_t c0 = (chunk - it.chunk_begin) * kChunkElems;

    // bf16 round-to-nearest-even of acc, staged in shared memory and written
    // by one bulk copy (two staging buffers per warp, used in turn)
    auto emit = [&](const f32x2 (&acc)[16], uint16_t* out) {
      uint32_t outw[16];
#pragma unroll
      for (int m = 0; m < 16; ++m) {
        float a, b;
        unpack2(acc[m], a, b);
        const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
        outw[m] = *reinterpret_cast<const uint32_t*>(&h);
      }
      const int bsel = n_store & 1;
      ++n_store;
      if (lane == 0) bulk_wait_read<1>();  // the store that last used this buffer has read it
      __syncwarp();
      uint4* dst = reinterpret_cast<uint4*>(stage_buf + bsel * kChunkBytes + lane * 64);
#pragma unroll
      for (int j = 0; j < 4; ++j)
        dst[(j + rot) & 3] = make_uint4(outw[4 * j], outw[4 * j + 1], outw[4 * j + 2], outw[4 * j + 3]);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        const int64_t left = it.n - c0;
        const uint32_t bytes = static_cast<uint32_t>((left < kChunkElems ? left : kChunkElems) * 2);
        bulk_store(out + c0, smem_u32(stage_buf + bsel * kChunkBytes), bytes);
        bulk_commit();
      }
    };

    f32x2 acc[16];
#pragma unroll
    for (int i = 0; i < K; ++i) {
      const uint32_t w0 = __byte_perm(code[i].x, code[i].y, sel_lo);
      const uint32_t w1 = __byte_perm(code[i].x, code[i].y, sel_hi);
      const f32x2 LO = pack2(zero[i], zero[i]);
      if (F == kAsymBits) {
        const uint4 w4 = *reinterpret_cast<const uint4*>(buf + i * kStageBytes + lane * 16);
        switch (p.bits[i]) {
          case 1: dequant_bits<1>(w4, scale[i], zero[i], i == 0, acc); break;
          case 3: dequant_bits<3>(w4, scale[i], zero[i], i == 0, acc); break;
          case 4: dequant_bits<4>(w4, scale[i], zero[i], i == 0, acc); break;
          default: dequant_bits<2>(w4, scale[i], zero[i], i == 0, acc); break;
        }
      } else if (kSym) {
        // u = Q - 2 and L = u s, both exact (sym_offsets)
        const f32x2 S = pack2(scale[i], scale[i]);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const uint32_t word = j < 4 ? w0 : w1;
          const uint32_t b = (j & 3) == 0 ? word : (word >> (8 * (j & 3)));
          f32x2 u01, u23;
          sym_offsets(b, u01, u23);
          acc[2 * j] = (i == 0) ? mul2(u01, S) : fma2(u01, S, acc[2 * j]);
          acc[2 * j + 1] = (i == 0) ? mul2(u23, S) : fma2(u23, S, acc[2 * j + 1]);
        }
      } else if (all_ok) {
        const StageConsts c = stage_consts(scale[i], zero[i]);
#pragma unroll
        for (int j = 0; j < 8; ++j) {  // byte j: elements 4j..4j+3 (pairs 2j, 2j+1)
          const uint32_t word = j < 4 ? w0 : w1;
          const uint32_t b = (j & 3) == 0 ? word : (word >> (8 * (j & 3)));
          f32x2 l01, l23;
          asym_levels(b, c, l01, l23);
          acc[2 * j] = (i == 0) ? l01 : add2(acc[2 * j], l01);
          acc[2 * j + 1] = (i == 0) ? l23 : add2(acc[2 * j + 1], l23);
        }
      } else {
        const f32x2 Z = pack2(0.0f, 0.0f), T23 = pack2(kTwo23, kTwo23);
        const f32x2 S = pack2(scale[i], scale[i]);
#pragma unroll
        for (int m = 0; m < 16; ++m) {
          const uint32_t word = m < 8 ? w0 : w1;
          const int sh = 4 * (m & 7);
          const f32x2 t = pack2u(magic23<3u>(word >> sh), magic23<3u>(word >> (sh + 2)));
          // RN(Q*s) through an fma with a zero addend (the compiler would fuse
          // a separate multiply into the following add)
          const f32x2 level = add2(LO, fma2(sub2(t, T23), S, Z));
          acc[m] = (i == 0) ? level : add2(acc[m], level);
        }
      }
      if (kAllPrefixes) emit(acc, it.out[i]);
    }
    if (!kAllPrefixes) emit(acc, it.out[0]);
  }
  cp_async_wait<0>();
  if (lane == 0) bulk_wait<0>();
}

template <int G, int K, bool A, int F>
cudaError_t launch_gk(const ReconstructBatch& p, cudaStream_t stream, int sms) {
  // resident CTAs per multiprocessor: the same for every device of this
  // build, asked once (an atomic: any thread may launch)
  static std::atomic<int> cached{0};
  int blocks_per_sm = cached.load(std::memory_order_relaxed);
  if (blocks_per_sm == 0) {
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
        &blocks_per_sm, reconstruct_kernel<G, K, A, F>, kThreads, smem_bytes<K, F>());
    if (e != cudaSuccess) return e;
    if (blocks_per_sm < 1) blocks_per_sm = 1;
    cached.store(blocks_per_sm, std::memory_order_relaxed);
  }
  const int64_t want = (p.total_chunks + kWarps - 1) / kWarps;
  const int64_t cap = static_cast<int64_t>(sms) * blocks_per_sm;
  const int grid = static_cast<int>(want < cap ? want : cap);
  reconstruct_kernel<G, K, A, F><<<grid, kThreads, smem_bytes<K, F>(), stream>>>(p);
  return cudaGetLastError();
}

template <int G, bool A, int F>
cudaError_t launch_g(int k, const ReconstructBatch& p, cudaStream_t stream, int sms) {
  switch (k) {
    case 1: return launch_gk<G, 1, A, F>(p, stream, sms);
    case 2: return launch_gk<G, 2, A, F>(p, stream, sms);
    case 3: return launch_gk<G, 3, A, F>(p, stream, sms);
    case 4: return launch_gk<G, 4, A, F>(p, stream, sms);
    default: return cudaErrorInvalidValue;
  }
}

template <int G, bool A, int F>
cudaError_t prepare_ga() {
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(reconstruct_kernel<G, 1, A, F>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes<1, F>()))) return e;
  if ((e = cudaFuncSetAttribute(reconstruct_kernel<G, 2, A, F>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes<2, F>()))) return e;
  if ((e = cudaFuncSetAttribute(reconstruct_kernel<G, 3, A, F>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes<3, F>()))) return e;
  return cudaFuncSetAttribute(reconstruct_kernel<G, 4, A, F>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes<4, F>());
}

template <int G, int F>
cudaError_t prepare_g() {
  cudaError_t e = prepare_ga<G, false, F>();
  return e != cudaSuccess ? e : prepare_ga<G, true, F>();
}

// Set-up and launch of one format (instantiated by one translation unit each).
template <int F>
cudaError_t prepare_format() {
  cudaError_t e;
  if ((e = prepare_g<32, F>())) return e;
  if ((e = prepare_g<64, F>())) return e;
  if ((e = prepare_g<128, F>())) return e;
  return prepare_g<256, F>();
}

template <int F>
cudaError_t launch_format(int group, int k, bool all_prefixes, const ReconstructBatch& p,
                          cudaStream_t stream, int sms) {
  if (all_prefixes) {
    switch (group) {
      case 32: return launch_g<32, true, F>(k, p, stream, sms);
      case 64: return launch_g<64, true, F>(k, p, stream, sms);
      case 128: return launch_g<128, true, F>(k, p, stream, sms);
      case 256: return launch_g<256, true, F>(k, p, stream, sms);
      default: return cudaErrorInvalidValue;
    }
  }
  switch (group) {
    case 32: return launch_g<32, false, F>(k, p, stream, sms);
    case 64: return launch_g<64, false, F>(k, p, stream, sms);
    case 128: return launch_g<128, false, F>(k, p, stream, sms);
    case 256: return launch_g<256, false, F>(k, p, stream, sms);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

}  // namespace rrq
