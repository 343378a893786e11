// Stage-wise product with the prefix weights (Appendix C): for the package's
// first k stages, Y[b][r] = sum_c W~[r][c] * A[b][c], where W~ is the binary32
// stage sum of the reconstruction (acc = L_0; acc = fl(acc + L_i)) before its
// bf16 rounding.  By linearity this is A W^_0 + sum_i A R^_i, computed here
// with the stages summed per weight first (one multiply per weight and token
// instead of one per stage), reading only the package -- k x (2 + 64/g) bits
// per weight -- and never a bf16 copy of the weights.  Aimed at decoding
// (1 to 8 activation rows), where the product is bound by weight movement.
//
// Work decomposition: the rows of all matrices of a launch form one sequence;
// warp w of the persistent grid takes rows w, w + W, ... (W warps in all) and
// walks each row in chunks of 1024 columns, lane l owning columns 32l..32l+31
// of a chunk.  Each lane copies its code words, scales and zeros of every
// stage asynchronously (cp.async) into a per-warp ring of shared-memory
// buffers, kRing - 1 chunks ahead, across row boundaries.  The lane forms its
// 32 prefix weights in binary32 exactly as the reconstruction does, reads its
// activations (bf16, L1-resident: every warp of an SM reads the same few KB),
// and accumulates packed fp32 fma's.  At the end of a row the warp reduces by
// butterfly shuffles and lane 0 stores Y: a fixed order, so results are
// deterministic, with no atomics and no workspace.
//
// Accuracy: every product W~ * a is exact inside its fma and each partial sum
// is rounded once, so |Y - exact| <= gamma_n * sum_c |W~ a| (n = cols) for any
// summation order; the parity tests use that bound.
#include <cuda_fp16.h>

#include "rrq_device.cuh"

namespace rrq {
namespace {

constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;
constexpr int kRing = 4;
constexpr int kStageBytes = 512;  // one stage of one chunk: codes 256 B | scales 128 B | zeros 128 B
constexpr int kWarpBytes = kRing * kMaxStages * kStageBytes;
constexpr int kSmemBytes = kWarps * kWarpBytes;
constexpr float kTwo23 = 8388608.0f;

__device__ __forceinline__ bool prescale_ok(float s) {
  return s == 0.0f || (s >= 0x1p-100f && s <= 0x1p+100f);
}

// A position in a warp's stream: global row index and chunk within the row.
struct Pos {
  int64_t row;
  int64_t ch;
};

template <int F, int B>
__global__ void __launch_bounds__(kThreads, 2) gemv_kernel(const __grid_constant__ GemvBatch p) {
  constexpr bool kSym = F != kAsymF32;
  constexpr bool kF16 = F == kSymF16;
  extern __shared__ __align__(128) uint8_t smem[];
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  uint8_t* ring = smem + warp * kWarpBytes;
  const int k = p.k;
  const int bufb = k * kStageBytes;

  const int64_t first = static_cast<int64_t>(blockIdx.x) * kWarps + warp;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kWarps;
  if (first >= p.total_rows) return;

  int m_issue = 0, m_work = 0, m_adv_i = 0, m_adv_w = 0;
  auto item_of = [&](int64_t row, int& m) -> const GemvItem& {
    while (m + 1 < p.count && row >= p.item[m + 1].row_begin) ++m;
    return p.item[m];
  };
  auto advance = [&](Pos& q, int& m) {
    if (q.row >= p.total_rows) return;
    const GemvItem& it = item_of(q.row, m);
    if (++q.ch * kChunkElems >= it.cols) {
      q.ch = 0;
      q.row += stride;
    }
  };
  // Copies this lane's package words of position q into ring buffer buf (one
  // commit group per call, empty past the end; lanes past the row's end get
  // zeros).
  auto issue = [&](const Pos& q, int buf) {
    if (q.row < p.total_rows) {
      const GemvItem& it = item_of(q.row, m_issue);
      const int64_t col = q.ch * kChunkElems + static_cast<int64_t>(lane) * kLaneElems;
      const bool valid = col < it.cols;
      const uint64_t e = static_cast<uint64_t>((q.row - it.row_begin) * it.cols + col);
      const uint64_t off_code = valid ? e >> 2 : 0;
      const uint64_t gi = e >> p.log2g;
      uint64_t off_meta = valid ? gi * 4 : 0;
      uint32_t n_scale = valid ? 4u : 0u;
      if (kF16) {
        off_meta = valid ? (gi * 2) & ~uint64_t{3} : 0;
        const uint64_t left = static_cast<uint64_t>((it.rows * it.cols) >> p.log2g) * 2 - off_meta;
        n_scale = valid ? (left < 4 ? 2u : 4u) : 0u;
      }
      const uint32_t n8 = valid ? 8u : 0u, n4 = valid ? 4u : 0u;
      const uint32_t base = smem_u32(ring + buf * bufb);
      for (int i = 0; i < k; ++i) {
        cp_async_8(base + i * kStageBytes + lane * 8, reinterpret_cast<const char*>(it.codes[i]) + off_code, n8);
        cp_async_4(base + i * kStageBytes + 256 + lane * 4,
                   reinterpret_cast<const char*>(it.scales[i]) + off_meta, n_scale);
        if (!kSym)
          cp_async_4(base + i * kStageBytes + 384 + lane * 4,
                     reinterpret_cast<const char*>(it.zeros[i]) + off_meta, n4);
      }
    }
    cp_async_commit();
  };

  Pos ip{first, 0}, wp{first, 0};
#pragma unroll
  for (int j = 0; j < kRing - 1; ++j) {
    issue(ip, j);
    advance(ip, m_adv_i);
  }

  f32x2 acc[B];
#pragma unroll
  for (int b = 0; b < B; ++b) acc[b] = pack2(0.0f, 0.0f);

  uint32_t iter = 0;
  while (wp.row < p.total_rows) {
    issue(ip, (iter + kRing - 1) % kRing);
    advance(ip, m_adv_i);
    cp_async_wait<kRing - 1>();  // this lane's copies of wp have landed

    const GemvItem& it = item_of(wp.row, m_work);
    const int64_t col = wp.ch * kChunkElems + static_cast<int64_t>(lane) * kLaneElems;
    const bool valid = col < it.cols;
    const uint8_t* buf = ring + (iter % kRing) * bufb;

    // prefix weights of this lane's 32 columns (pairs of consecutive columns)
    f32x2 w[16];
#pragma unroll 1
    for (int i = 0; i < k; ++i) {
      const uint2 code = *reinterpret_cast<const uint2*>(buf + i * kStageBytes + lane * 8);
      float s;
      if (kF16) {
        const uint32_t word = *reinterpret_cast<const uint32_t*>(buf + i * kStageBytes + 256 + lane * 4);
        const uint64_t gi = static_cast<uint64_t>((wp.row - it.row_begin) * it.cols + col) >> p.log2g;
        const uint32_t h = (gi & 1) ? (word >> 16) : (word & 0xffffu);
        s = __half2float(__ushort_as_half(static_cast<unsigned short>(h)));
      } else {
        s = *reinterpret_cast<const float*>(buf + i * kStageBytes + 256 + lane * 4);
      }
      const float z = kSym ? 0.0f : *reinterpret_cast<const float*>(buf + i * kStageBytes + 384 + lane * 4);
      const f32x2 Z = pack2(z, z);
      if (prescale_ok(s)) {
        // t = 2^23 + Q*4^j exactly; s*4^-j exact (see reconstruct_kernel.cuh)
        const f32x2 S01 = pack2(s, __fmul_rn(s, 0x1p-2f));
        const f32x2 S23 = pack2(__fmul_rn(s, 0x1p-4f), __fmul_rn(s, 0x1p-6f));
        const f32x2 C01 = pack2(__fmul_rn(s, -0x1p23f), __fmul_rn(s, -0x1p21f));
        const f32x2 C23 = pack2(__fmul_rn(s, -0x1p19f), __fmul_rn(s, -0x1p17f));
        const f32x2 K01 = pack2(kTwo23 + 2.0f, kTwo23 + 8.0f);
        const f32x2 K23 = pack2(kTwo23 + 32.0f, kTwo23 + 128.0f);
#pragma unroll
        for (int j = 0; j < 8; ++j) {  // byte j: columns 4j..4j+3 (pairs 2j, 2j+1)
          const uint32_t word = j < 4 ? code.x : code.y;
          const uint32_t b8 = (j & 3) == 0 ? word : (word >> (8 * (j & 3)));
          const f32x2 t01 = pack2u(0x4B000000u | (b8 & 0x03u), 0x4B000000u | (b8 & 0x0Cu));
          const f32x2 t23 = pack2u(0x4B000000u | (b8 & 0x30u), 0x4B000000u | (b8 & 0xC0u));
          f32x2 l01, l23;
          if (kSym) {  // (Q - 2) s, exact; summed by one fma
            const f32x2 u01 = sub2(t01, K01), u23 = sub2(t23, K23);
            w[2 * j] = (i == 0) ? mul2(u01, S01) : fma2(u01, S01, w[2 * j]);
            w[2 * j + 1] = (i == 0) ? mul2(u23, S23) : fma2(u23, S23, w[2 * j + 1]);
          } else {     // fl(zero + fl(Q s))
            l01 = add2(Z, fma2(t01, S01, C01));
            l23 = add2(Z, fma2(t23, S23, C23));
            w[2 * j] = (i == 0) ? l01 : add2(w[2 * j], l01);
            w[2 * j + 1] = (i == 0) ? l23 : add2(w[2 * j + 1], l23);
          }
        }
      } else {
        const f32x2 S = pack2(s, s), T = pack2(kTwo23, kTwo23), Z0 = pack2(0.0f, 0.0f);
        const f32x2 K2 = pack2(kTwo23 + 2.0f, kTwo23 + 2.0f);
#pragma unroll
        for (int m = 0; m < 16; ++m) {
          const uint32_t word = m < 8 ? code.x : code.y;
          const int sh = 4 * (m & 7);
          const f32x2 t = pack2u(0x4B000000u | ((word >> sh) & 3u), 0x4B000000u | ((word >> (sh + 2)) & 3u));
          if (kSym) {
            const f32x2 u = sub2(t, K2);
            w[m] = (i == 0) ? mul2(u, S) : fma2(u, S, w[m]);
          } else {
            const f32x2 level = add2(Z, fma2(sub2(t, T), S, Z0));
            w[m] = (i == 0) ? level : add2(w[m], level);
          }
        }
      }
    }

    // w . a for every activation row
    if (valid) {
#pragma unroll
      for (int b = 0; b < B; ++b) {
        const uint4* a = reinterpret_cast<const uint4*>(it.A + b * it.cols + col);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const uint4 a8 = __ldg(a + q);
          const uint32_t a4[4] = {a8.x, a8.y, a8.z, a8.w};
#pragma unroll
          for (int m = 0; m < 4; ++m)
            acc[b] = fma2(w[4 * q + m], pack2u(a4[m] << 16, a4[m] & 0xffff0000u), acc[b]);
        }
      }
    }

    if ((wp.ch + 1) * kChunkElems >= it.cols) {  // last chunk of the row: reduce and store
      const int64_t r = wp.row - it.row_begin;
#pragma unroll
      for (int b = 0; b < B; ++b) {
        float x, y;
        unpack2(acc[b], x, y);
        float t = __fadd_rn(x, y);
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) t = __fadd_rn(t, __shfl_xor_sync(kFullMask, t, off));
        if (lane == 0) it.Y[b * it.rows + r] = t;
        acc[b] = pack2(0.0f, 0.0f);
      }
    }
    advance(wp, m_adv_w);
    ++iter;
  }
  cp_async_wait<0>();
}

template <int F, int B>
cudaError_t launch_fb(const GemvBatch& p, cudaStream_t stream, int sms) {
  static int blocks_per_sm = 0;
  if (blocks_per_sm == 0) {
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&blocks_per_sm, gemv_kernel<F, B>,
                                                                  kThreads, kSmemBytes);
    if (e != cudaSuccess) return e;
    if (blocks_per_sm < 1) blocks_per_sm = 1;
  }
  const int64_t want = (p.total_rows + kWarps - 1) / kWarps;
  const int64_t cap = static_cast<int64_t>(sms) * blocks_per_sm;
  const int grid = static_cast<int>(want < cap ? want : cap);
  gemv_kernel<F, B><<<grid, kThreads, kSmemBytes, stream>>>(p);
  return cudaGetLastError();
}

template <int F>
cudaError_t launch_f(int batch, const GemvBatch& p, cudaStream_t stream, int sms) {
  switch (batch) {
    case 1: return launch_fb<F, 1>(p, stream, sms);
    case 2: return launch_fb<F, 2>(p, stream, sms);
    case 3: return launch_fb<F, 3>(p, stream, sms);
    case 4: return launch_fb<F, 4>(p, stream, sms);
    case 5: return launch_fb<F, 5>(p, stream, sms);
    case 6: return launch_fb<F, 6>(p, stream, sms);
    case 7: return launch_fb<F, 7>(p, stream, sms);
    case 8: return launch_fb<F, 8>(p, stream, sms);
    default: return cudaErrorInvalidValue;
  }
}

template <int F, int B>
cudaError_t prepare_fb() {
  return cudaFuncSetAttribute(gemv_kernel<F, B>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
}

template <int F>
cudaError_t prepare_f() {
  cudaError_t e;
  if ((e = prepare_fb<F, 1>())) return e;
  if ((e = prepare_fb<F, 2>())) return e;
  if ((e = prepare_fb<F, 3>())) return e;
  if ((e = prepare_fb<F, 4>())) return e;
  if ((e = prepare_fb<F, 5>())) return e;
  if ((e = prepare_fb<F, 6>())) return e;
  if ((e = prepare_fb<F, 7>())) return e;
  return prepare_fb<F, 8>();
}

}  // namespace

cudaError_t gemv_prepare() {
  cudaError_t e;
  if ((e = prepare_f<kAsymF32>())) return e;
  if ((e = prepare_f<kSymF32>())) return e;
  return prepare_f<kSymF16>();
}

cudaError_t gemv_launch(Format fmt, int batch, const GemvBatch& p, cudaStream_t stream, int sms) {
  switch (fmt) {
    case kAsymF32: return launch_f<kAsymF32>(batch, p, stream, sms);
    case kSymF32: return launch_f<kSymF32>(batch, p, stream, sms);
    case kSymF16: return launch_f<kSymF16>(batch, p, stream, sms);
  }
  return cudaErrorInvalidValue;
}

}  // namespace rrq
