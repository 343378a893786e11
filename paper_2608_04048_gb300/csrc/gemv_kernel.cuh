// Stage-wise product with the prefix weights (Appendix C): for the package's
// first k stages, Y[b][r] = sum_c W~[r][c] * A[b][c], where W~ is the binary32
// stage sum of the reconstruction (acc = L_0; acc = fl(acc + L_i)) before its
// bf16 rounding.  By linearity this is A W^_0 + sum_i A R^_i, computed here
// with the stages summed per weight first (one multiply per weight and token
// instead of one per stage), reading only the package -- k x (2 + 64/g) bits
// per weight -- and never a bf16 copy of the weights.  Aimed at decoding
// (1 to 8 activation rows), where the product is bound by weight movement.
//
// Work decomposition: the rows of every matrix are cut into blocks of 16
// rows; the blocks of all matrices of a launch form one sequence, cut into
// one contiguous range per CTA of a persistent grid with equal shares of
// rows x columns (so a CTA meets few matrices), each CTA taking its blocks in
// order with 16 warps, one row of the block per warp.  A CTA keeps the activations of its current matrix in shared memory
// as binary32 (converted once when the matrix changes, in a swizzled layout:
// 16-byte piece P of a row stored at P ^ ((P >> 3) & 7), so that the eight
// lanes of a quarter warp reading their piece q hit eight different bank
// groups).  A warp walks its row in chunks of 1024 columns, lane l owning
// columns 32l..32l+31; each lane copies its code words, scales and zeros of
// every stage asynchronously (cp.async) into a per-warp ring of shared-memory
// buffers, two chunks ahead across rows and blocks.  Per group of four
// columns the lane forms the binary32 prefix weights exactly as the
// reconstruction does and multiplies them with one 16-byte shared-memory read
// of activations per activation row (packed fp32 fma's).  At the end of a row
// the warp reduces by butterfly shuffles and lane 0 stores Y: a fixed order,
// so results are deterministic, with no atomics and no workspace.
//
// Accuracy: every product W~ * a is exact inside its fma and each partial sum
// is rounded once, so |Y - exact| <= gamma_n * sum_c |W~ a| (n = cols) for any
// summation order; the parity tests use the tighter count of this kernel's
// summation tree.
//
// This header holds the kernel template; gemv_asym_f32.cu, gemv_sym_f32.cu
// and gemv_sym_f16.cu each instantiate one package format.
#pragma once

#include <cuda_fp16.h>

#include "rrq_device.cuh"

namespace rrq {
namespace {

constexpr int kWarps = 16;
constexpr int kThreads = kWarps * 32;
constexpr int kRows = kGemvRows;       // rows per block (one per warp)
static_assert(kRows == kWarps, "one row of a block per warp");
// ring depth (chunks per warp in shared memory, two ahead of use)
template <int K>
__host__ __device__ constexpr int ring_depth() { return 3; }
// one stage of one chunk: codes (256 B at 2 bits, up to 512 B with per-stage
// widths: 16 B per lane) | scales 128 B | zeros 128 B
template <int F>
__host__ __device__ constexpr int code_area() { return F == kAsymBits ? 512 : 256; }
template <int F>
__host__ __device__ constexpr int stage_bytes() { return code_area<F>() + 256; }
constexpr int kMaxSmem = 227 * 1024;
constexpr float kTwo23 = 8388608.0f;

template <int F, int K>
__host__ __device__ constexpr int ring_bytes() { return kWarps * ring_depth<K>() * K * stage_bytes<F>(); }

// swizzled position of 16-byte activation piece P of a row
__device__ __forceinline__ uint32_t act_piece(uint32_t P) { return P ^ ((P >> 3) & 7u); }

// Where a warp is in its stream: block, chunk of the row, and the row's start.
struct Cursor {
  int64_t blk;   // global block index (>= total_blocks: past the end)
  int64_t e;     // element offset of the chunk's first column within its matrix
  int ch, nch;
  int m;
};

template <int F, int K, int B>
__global__ void __launch_bounds__(kThreads, 1)
gemv_kernel(const __grid_constant__ GemvBatch p, int nb, int act_floats) {
  constexpr bool kSym = F == kSymF32 || F == kSymF16;
  constexpr bool kF16 = F == kSymF16;
  constexpr int kStageBytes = stage_bytes<F>();
  constexpr int kCA = code_area<F>();  // scales at kCA, zeros at kCA + 128
  constexpr int kBuf = K * kStageBytes;
  constexpr int kRing = ring_depth<K>();
  extern __shared__ __align__(128) uint8_t smem[];
  float* act = reinterpret_cast<float*>(smem + ring_bytes<F, K>());  // [B][act_floats], swizzled pieces
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  uint8_t* ring = smem + warp * kRing * kBuf;
  const uint32_t ring_s = smem_u32(ring);
  const int lane_col = lane * kLaneElems;
  // byte offsets of this lane's eight activation pieces within a chunk
  uint32_t poff[8];
#pragma unroll
  for (int q = 0; q < 8; ++q) poff[q] = act_piece(static_cast<uint32_t>(lane * 8 + q)) * 16u;

  auto item_of = [&](int64_t blk, int& m) -> const GemvItem& {
    while (m + 1 < p.count && blk >= p.item[m + 1].blk_begin) ++m;
    return p.item[m];
  };
  const int64_t blk_end = p.cta_begin[blockIdx.x + 1];
  // position the cursor on the first valid row of this warp at or after blk
  auto start_block = [&](Cursor& c, int64_t blk) {
    for (; blk < blk_end; ++blk) {
      const GemvItem& it = item_of(blk, c.m);
      const int64_t r = (blk - it.blk_begin) * kRows + warp;
      if (r < it.rows) {
        c.blk = blk;
        c.ch = 0;
        c.e = r * it.cols;
        c.nch = static_cast<int>((it.cols + kChunkElems - 1) / kChunkElems);
        return;
      }
    }
    c.blk = blk_end;
  };
  auto advance = [&](Cursor& c) {
    if (c.blk >= blk_end) return;
    if (++c.ch < c.nch) c.e += kChunkElems;
    else start_block(c, c.blk + 1);
  };
  auto issue = [&](const Cursor& c, int buf) {
    if (c.blk < blk_end) {
      // every field read before the first copy (the copies clobber memory)
      const GemvItem& it = p.item[c.m];
      const char* cp[K];
      const char* sp[K];
      const char* zp[K];
#pragma unroll
      for (int i = 0; i < K; ++i) {
        cp[i] = reinterpret_cast<const char*>(it.codes[i]);
        sp[i] = reinterpret_cast<const char*>(it.scales[i]);
        zp[i] = kSym ? nullptr : reinterpret_cast<const char*>(it.zeros[i]);
      }
      const int64_t cols = it.cols;
      const int col = c.ch * kChunkElems + lane_col;
      const bool valid = col < cols;
      const uint64_t e = static_cast<uint64_t>(c.e) + lane_col;
      const uint64_t off_code = valid ? e >> 2 : 0;
      const uint64_t gi = e >> p.log2g;
      uint64_t off_meta = valid ? gi * 4 : 0;
      uint32_t n_scale = valid ? 4u : 0u;
      if (kF16) {  // the aligned 4-byte word holding this group's 2-byte scale
        off_meta = valid ? (gi * 2) & ~uint64_t{3} : 0;
        const uint64_t left = static_cast<uint64_t>((it.rows * cols) >> p.log2g) * 2 - off_meta;
        n_scale = valid ? (left < 4 ? 2u : 4u) : 0u;
      }
      const uint32_t n8 = valid ? 8u : 0u, n4 = valid ? 4u : 0u;
      const uint32_t base = ring_s + buf * kBuf;
#pragma unroll
      for (int i = 0; i < K; ++i) {
        if constexpr (F == kAsymBits) {  // 4b bytes of b-bit codes for the lane's 32 weights
          const int b = p.bits[i];
          const char* src = cp[i] + (valid ? (e >> 5) * 4 * static_cast<uint64_t>(b) : 0);
          const uint32_t dst = base + i * kStageBytes + lane * 16;
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
          cp_async_8(base + i * kStageBytes + lane * 8, cp[i] + off_code, n8);
        }
        cp_async_4(base + i * kStageBytes + kCA + lane * 4, sp[i] + off_meta, n_scale);
        if (!kSym) cp_async_4(base + i * kStageBytes + kCA + 128 + lane * 4, zp[i] + off_meta, n4);
      }
    }
    cp_async_commit();
  };

  Cursor ic{0, 0, 0, 0, 0};
  start_block(ic, p.cta_begin[blockIdx.x]);
#pragma unroll
  for (int j = 0; j < kRing - 1; ++j) {
    issue(ic, j);
    advance(ic);
  }

  int slot = 0, slot_issue = kRing - 1;  // ring buffer of this chunk / of the next copy
  int m_work = 0, m_act = -1;
  for (int64_t blk = p.cta_begin[blockIdx.x]; blk < blk_end; ++blk) {
    const GemvItem& it = item_of(blk, m_work);
    if (m_work != m_act) {
      // a new matrix: every warp has finished with the old activations
      __syncthreads();
      const int pieces = static_cast<int>(it.cols / 4);
      for (int b = 0; b < nb; ++b)
        for (int P = threadIdx.x; P < pieces; P += kThreads) {
          const uint2 a = __ldg(reinterpret_cast<const uint2*>(it.A + b * it.cols) + P);
          const float4 f = make_float4(__uint_as_float(a.x << 16), __uint_as_float(a.x & 0xffff0000u),
                                       __uint_as_float(a.y << 16), __uint_as_float(a.y & 0xffff0000u));
          reinterpret_cast<float4*>(act + b * act_floats)[act_piece(static_cast<uint32_t>(P))] = f;
        }
      __syncthreads();
      m_act = m_work;
    }
    const int64_t r = (blk - it.blk_begin) * kRows + warp;
    if (r >= it.rows) continue;  // this warp has no row in the matrix's last block
    const int cols = static_cast<int>(it.cols);
    const int nch = (cols + kChunkElems - 1) / kChunkElems;

    f32x2 acc[B];
#pragma unroll
    for (int b = 0; b < B; ++b) acc[b] = pack2(0.0f, 0.0f);

    for (int ch = 0; ch < nch; ++ch) {
      issue(ic, slot_issue);
      advance(ic);
      slot_issue = slot_issue == kRing - 1 ? 0 : slot_issue + 1;
      cp_async_wait<kRing - 1>();  // this lane's copies of this chunk have landed

      const int col = ch * kChunkElems + lane_col;
      const uint8_t* buf = ring + slot * kBuf;
      slot = slot == kRing - 1 ? 0 : slot + 1;
      uint2 code[K];
      float s[K], z[K];
      bool fast = true;
#pragma unroll
      for (int i = 0; i < K; ++i) {
        code[i] = F == kAsymBits ? make_uint2(0u, 0u) : *reinterpret_cast<const uint2*>(buf + i * kStageBytes + lane * 8);
        if (kF16) {
          const uint32_t word = *reinterpret_cast<const uint32_t*>(buf + i * kStageBytes + kCA + lane * 4);
          const uint64_t gi = static_cast<uint64_t>(r * cols + col) >> p.log2g;
          const uint32_t h = (gi & 1) ? (word >> 16) : (word & 0xffffu);
          s[i] = __half2float(__ushort_as_half(static_cast<unsigned short>(h)));
        } else {
          s[i] = *reinterpret_cast<const float*>(buf + i * kStageBytes + kCA + lane * 4);
          fast = fast && prescale_ok(s[i]);
        }
        z[i] = kSym ? 0.0f : *reinterpret_cast<const float*>(buf + i * kStageBytes + kCA + 128 + lane * 4);
      }
      if (col >= cols) continue;  // beyond the row's last column: nothing to add
      const uint8_t* abase = reinterpret_cast<const uint8_t*>(act) + static_cast<uint32_t>(ch) * (kChunkElems * 4);

      // four columns at a time: the k-stage prefix weights, then w . a
      auto dot = [&](int q, const f32x2& w01, const f32x2& w23) {
#pragma unroll
        for (int b = 0; b < B; ++b) {
          if (b < nb) {
            const float4 a = *reinterpret_cast<const float4*>(abase + b * act_floats * 4 + poff[q]);
            acc[b] = fma2(w01, pack2(a.x, a.y), acc[b]);
            acc[b] = fma2(w23, pack2(a.z, a.w), acc[b]);
          }
        }
      };
      if constexpr (F == kAsymBits) {
        // per-stage widths: the reconstruction's width-generic stage sum
        f32x2 w[16];
#pragma unroll
        for (int i = 0; i < K; ++i) {
          const uint4 w4 = *reinterpret_cast<const uint4*>(buf + i * kStageBytes + lane * 16);
          switch (p.bits[i]) {
            case 1: dequant_bits<1>(w4, s[i], z[i], i == 0, w); break;
            case 3: dequant_bits<3>(w4, s[i], z[i], i == 0, w); break;
            case 4: dequant_bits<4>(w4, s[i], z[i], i == 0, w); break;
            default: dequant_bits<2>(w4, s[i], z[i], i == 0, w); break;
          }
        }
#pragma unroll
        for (int q = 0; q < 8; ++q) dot(q, w[2 * q], w[2 * q + 1]);
      } else if (fast) {
        // t = 2^23 + Q*4^j exactly; s*4^-j exact (see reconstruct_kernel.cuh)
        f32x2 S01[K], S23[K], C01[K], C23[K], Z[K];
#pragma unroll
        for (int i = 0; i < K; ++i) {
          S01[i] = pack2(s[i], __fmul_rn(s[i], 0x1p-2f));
          S23[i] = pack2(__fmul_rn(s[i], 0x1p-4f), __fmul_rn(s[i], 0x1p-6f));
          C01[i] = pack2(__fmul_rn(s[i], -0x1p23f), __fmul_rn(s[i], -0x1p21f));
          C23[i] = pack2(__fmul_rn(s[i], -0x1p19f), __fmul_rn(s[i], -0x1p17f));
          Z[i] = pack2(z[i], z[i]);
        }
        const f32x2 K01 = pack2(kTwo23 + 2.0f, kTwo23 + 8.0f), K23 = pack2(kTwo23 + 32.0f, kTwo23 + 128.0f);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          f32x2 w01, w23;
#pragma unroll
          for (int i = 0; i < K; ++i) {
            const uint32_t word = q < 4 ? code[i].x : code[i].y;
            const uint32_t b8 = (q & 3) == 0 ? word : (word >> (8 * (q & 3)));
            const f32x2 t01 = pack2u(0x4B000000u | (b8 & 0x03u), 0x4B000000u | (b8 & 0x0Cu));
            const f32x2 t23 = pack2u(0x4B000000u | (b8 & 0x30u), 0x4B000000u | (b8 & 0xC0u));
            if (kSym) {  // (Q - 2) s, exact; summed by one fma
              const f32x2 u01 = sub2(t01, K01), u23 = sub2(t23, K23);
              w01 = (i == 0) ? mul2(u01, S01[i]) : fma2(u01, S01[i], w01);
              w23 = (i == 0) ? mul2(u23, S23[i]) : fma2(u23, S23[i], w23);
            } else {     // fl(zero + fl(Q s))
              const f32x2 l01 = add2(Z[i], fma2(t01, S01[i], C01[i]));
              const f32x2 l23 = add2(Z[i], fma2(t23, S23[i], C23[i]));
              w01 = (i == 0) ? l01 : add2(w01, l01);
              w23 = (i == 0) ? l23 : add2(w23, l23);
            }
          }
          dot(q, w01, w23);
        }
      } else {
        // a scale outside [2^-100, 2^100]: unscaled codes, plain (t - 2^23) s
        const f32x2 T = pack2(kTwo23, kTwo23), Z0 = pack2(0.0f, 0.0f), K2 = pack2(kTwo23 + 2.0f, kTwo23 + 2.0f);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          f32x2 w01, w23;
#pragma unroll
          for (int i = 0; i < K; ++i) {
            const uint32_t word = q < 4 ? code[i].x : code[i].y;
            const uint32_t b8 = (q & 3) == 0 ? word : (word >> (8 * (q & 3)));
            const f32x2 t01 = pack2u(0x4B000000u | (b8 & 3u), 0x4B000000u | ((b8 >> 2) & 3u));
            const f32x2 t23 = pack2u(0x4B000000u | ((b8 >> 4) & 3u), 0x4B000000u | ((b8 >> 6) & 3u));
            const f32x2 S = pack2(s[i], s[i]);
            if (kSym) {
              const f32x2 u01 = sub2(t01, K2), u23 = sub2(t23, K2);
              w01 = (i == 0) ? mul2(u01, S) : fma2(u01, S, w01);
              w23 = (i == 0) ? mul2(u23, S) : fma2(u23, S, w23);
            } else {
              const f32x2 Z = pack2(z[i], z[i]);
              const f32x2 l01 = add2(Z, fma2(sub2(t01, T), S, Z0));
              const f32x2 l23 = add2(Z, fma2(sub2(t23, T), S, Z0));
              w01 = (i == 0) ? l01 : add2(w01, l01);
              w23 = (i == 0) ? l23 : add2(w23, l23);
            }
          }
          dot(q, w01, w23);
        }
      }
    }

    // end of the row: reduce over the warp in a fixed order and store
#pragma unroll
    for (int b = 0; b < B; ++b) {
      float x, y;
      unpack2(acc[b], x, y);
      float t = __fadd_rn(x, y);
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) t = __fadd_rn(t, __shfl_xor_sync(kFullMask, t, off));
      if (lane == 0 && b < nb) it.Y[b * it.rows + r] = t;
    }
  }
  cp_async_wait<0>();
}

// activation rows a launch can hold for matrices of up to max_cols columns
inline int64_t act_floats_of(int64_t max_cols) {
  return ((max_cols + kChunkElems - 1) / kChunkElems) * kChunkElems;
}
template <int F, int K>
int tokens_per_launch(int64_t max_cols) {
  const int64_t t = (kMaxSmem - ring_bytes<F, K>()) / (act_floats_of(max_cols) * 4);
  return static_cast<int>(t < kMaxGemvBatch ? t : kMaxGemvBatch);
}

template <int F, int K, int B>
cudaError_t launch_fkb(const GemvBatch& p, int nb, int64_t max_cols, cudaStream_t stream, int sms) {
  static int attr_bytes = 0;  // largest dynamic shared memory enabled so far (same for every device)
  const int act_floats = static_cast<int>(act_floats_of(max_cols));
  const int smem = ring_bytes<F, K>() + nb * act_floats * 4;
  if (smem > attr_bytes) {
    cudaError_t e = cudaFuncSetAttribute(gemv_kernel<F, K, B>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    attr_bytes = smem;
  }
  gemv_kernel<F, K, B><<<p.grid, kThreads, smem, stream>>>(p, nb, act_floats);
  return cudaGetLastError();
}

template <int F, int K>
cudaError_t launch_fk(int nb, int64_t max_cols, const GemvBatch& p, cudaStream_t stream, int sms) {
  if (nb <= 1) return launch_fkb<F, K, 1>(p, nb, max_cols, stream, sms);
  if (nb <= 2) return launch_fkb<F, K, 2>(p, nb, max_cols, stream, sms);
  if (nb <= 4) return launch_fkb<F, K, 4>(p, nb, max_cols, stream, sms);
  return launch_fkb<F, K, 8>(p, nb, max_cols, stream, sms);
}

// Launch of one format (instantiated by one translation unit each).
template <int F>
cudaError_t launch_format(int k, int nb, int64_t max_cols, const GemvBatch& p, cudaStream_t stream, int sms) {
  switch (k) {
    case 1: return launch_fk<F, 1>(nb, max_cols, p, stream, sms);
    case 2: return launch_fk<F, 2>(nb, max_cols, p, stream, sms);
    case 3: return launch_fk<F, 3>(nb, max_cols, p, stream, sms);
    case 4: return launch_fk<F, 4>(nb, max_cols, p, stream, sms);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace
}  // namespace rrq
