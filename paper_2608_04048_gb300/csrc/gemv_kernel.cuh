// Stage-wise product with the prefix weights (Appendix C): for the package's
// first k stages, Y[b][r] = sum_c W~[r][c] * A[b][c], where W~ is the binary32
// stage sum of the reconstruction (acc = L_0; acc = fl(acc + L_i)) before its
// bf16 rounding.  By linearity this is A W^_0 + sum_i A R^_i, computed here
// with the stages summed per weight first (one multiply per weight and token
// instead of one per stage), reading only the package -- k x (2 + 64/g) bits
// per weight -- and never a bf16 copy of the weights.  Aimed at decoding
// (1 to 8 activation rows), where the product moves little data per weight
// and its cost is the instructions that form each weight.
//
// Work decomposition: the rows of every matrix are cut into blocks of 16
// rows; the blocks of all matrices of a launch form one sequence, cut into
// one contiguous range per CTA of a persistent grid (as many CTAs as fit on
// the multiprocessors) with equal shares of rows x columns, so that a CTA
// meets few matrices.  The CTA's 16 warps take one row of each block each.
// A warp walks its row in windows of 32 x lc columns, lane l owning the lc
// columns lc*l .. lc*l + lc-1 of the window: lc = 128 at k = 1, and at k = 2
// with up to 2 activation rows (64 otherwise, where registers are scarcer),
// never more than the group, so that a lane's columns share one group (the row length
// is a multiple of the group, so a lane's columns are all in the row or all
// past its end).  Per stage the lane loads lc/4 bytes of codes (16-byte
// loads; 8 bytes for 32 columns) and one scale and zero, all into registers
// one window ahead, across rows, blocks and matrices.
//
// The CTA keeps the activations of its current matrix in shared memory as
// binary32, converted once per matrix, stored transposed within each window:
// the 16-byte piece j (columns 4j..4j+3 of a lane's columns) of lane l sits at
// (window, j, l), so the 32 lanes reading their piece j touch 512 contiguous
// bytes (no bank conflict) at an offset that is a constant per j.  Per four
// columns a lane forms the binary32 prefix weights exactly as the
// reconstruction does and multiplies them with one 16-byte read of
// activations per activation row (packed fp32 fma's).  At the end of a row
// the warp reduces by butterfly shuffles and lane 0 stores Y: a fixed order,
// so results are deterministic, with no atomics and no workspace.
//
// Accuracy: every product W~ * a is exact inside its fma and each partial sum
// is rounded once.  A lane's two accumulators (even and odd columns of each
// pair) each take at most 64 products per 4096 columns of the row (rounded
// up), then the pair and 5 butterfly steps, so |Y - exact| <=
// (64 ceil(cols/4096) + 6) * 2^-24 * sum_c |W~ a| to first order.
//
// This header holds the kernel template; gemv_asym_f32.cu, gemv_sym_f32.cu,
// gemv_sym_f16.cu and gemv_asym_bits.cu each instantiate one package format.
#pragma once

#include <cuda_fp16.h>

#include "rrq.h"  // RRQ_MAX_GEMV_COLS
#include "rrq_device.cuh"

namespace rrq {
namespace {

constexpr int kWarps = 16;
constexpr int kThreads = kWarps * 32;
constexpr int kRows = kGemvRows;       // rows per block (one per warp)
static_assert(kRows == kWarps, "one row of a block per warp");
constexpr int kWinCols = 4096;         // columns of the widest warp window (activation padding)

// Columns a lane owns in a window at most: 128 at k = 1, and at k = 2 with 1
// or 2 activation rows (more weights per window's fixed cost), else 64
// (registers).
template <int F, int K, int B>
__host__ __device__ constexpr int lane_cols_max() {
  return (F != kAsymBits && (K == 1 || (K == 2 && B <= 2))) ? 128 : 64;
}
constexpr int kMaxSmem = 227 * 1024;
constexpr float kTwo23 = 8388608.0f;

// Read-once package loads: no L1 allocation, read-only path.
__device__ __forceinline__ uint4 ld_nc16(const void* p) {
  uint4 v;
  asm("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
      : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}
__device__ __forceinline__ uint2 ld_nc8(const void* p) {
  uint2 v;
  asm("ld.global.nc.L1::no_allocate.v2.u32 {%0,%1}, [%2];" : "=r"(v.x), "=r"(v.y) : "l"(p));
  return v;
}
__device__ __forceinline__ uint32_t ld_nc4(const void* p) {
  uint32_t v;
  asm("ld.global.nc.L1::no_allocate.u32 %0, [%1];" : "=r"(v) : "l"(p));
  return v;
}
__device__ __forceinline__ uint32_t ld_nc2(const void* p) {
  unsigned short v;
  asm("ld.global.nc.L1::no_allocate.u16 %0, [%1];" : "=h"(v) : "l"(p));
  return v;
}

// A lane's package data of one window: per stage the codes of its 64 (or 32)
// columns (16 bytes at 2 bits; up to 32 bytes with per-stage widths), and the
// raw scale and zero of their group.
template <int F, int K, int B>
struct Window {
  static constexpr int kVecs = F == kAsymBits ? 2 : lane_cols_max<F, K, B>() / 64;
  uint4 code[K][kVecs];
  uint32_t s[K];  // binary32 bits, or binary16 bits in the low half
  float z[K];
};

// Where a warp is in its sequence of windows.
struct Pos {
  int64_t blk;   // global block index (>= the CTA's end: no window)
  int64_t rowe;  // element offset of the row's first column within its matrix
  int m;         // matrix (item) index
  int ch, nch;   // window of the row, windows per row
};

// Named barrier 1 over the whole CTA, in its non-aligned form: warps reach
// it from different places of the loop (each warp passes the same matrix
// changes in the same order, so the arrivals always pair up).
__device__ __forceinline__ void cta_barrier() {
  asm volatile("barrier.sync 1, %0;" ::"n"(kThreads) : "memory");
}

template <int F, int K, int B>
__global__ void __launch_bounds__(kThreads, (K == 1 && B == 1 && F != kAsymBits) ? 2 : 1)
gemv_kernel(const __grid_constant__ GemvBatch p, int nb, int act_floats) {
  constexpr bool kSym = F == kSymF32 || F == kSymF16;
  constexpr bool kF16 = F == kSymF16;
  constexpr bool kBits = F == kAsymBits;
  extern __shared__ __align__(16) float4 act4[];  // [B][act_floats / 4] pieces, transposed per window
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int64_t blk_begin = p.cta_begin[blockIdx.x];
  const int64_t blk_end = p.cta_begin[blockIdx.x + 1];
  if (blk_begin >= blk_end) return;  // the whole CTA: no barrier is reached
  const int log2g = p.log2g;
  constexpr int kLCM = lane_cols_max<F, K, B>();
  // columns of a lane in a window: within one group
  const int lc = (1 << log2g) < kLCM ? (1 << log2g) : kLCM;
  const int wcols = 32 * lc;                          // columns of a window
  const int lsh = lc == 32 ? 3 : (lc == 64 ? 4 : 5);  // log2 of a lane's 16-byte pieces per window
  const int wsh = lsh + 7;                            // log2 of wcols
  const int nh = lc >> 5;                             // 32-column parts of a lane's window
  const int act_pieces = act_floats / 4;

  auto item_index = [&](int64_t blk, int m) {
    while (m + 1 < p.count && blk >= p.item[m + 1].blk_begin) ++m;
    return m;
  };
  // activations of matrix m, bf16 -> binary32 (exact), piece P of window w,
  // lane l, piece j of the lane stored at (w * lc/4 + j) * 32 + l
  auto load_acts = [&](int m) {
    const GemvItem& it = p.item[m];
    const int pieces = static_cast<int>(it.cols / 4);
    for (int b = 0; b < nb; ++b) {
      const uint2* src = reinterpret_cast<const uint2*>(it.A + b * it.cols);
      float4* dst = act4 + b * act_pieces;
      for (int P = threadIdx.x; P < pieces; P += kThreads) {
        const uint2 a = __ldg(src + P);
        dst[(((P >> (lsh + 5)) << lsh) + (P & ((1 << lsh) - 1))) * 32 + ((P >> lsh) & 31)] =
            make_float4(__uint_as_float(a.x << 16), __uint_as_float(a.x & 0xffff0000u),
                        __uint_as_float(a.y << 16), __uint_as_float(a.y & 0xffff0000u));
      }
    }
  };
  const int m_first = item_index(blk_begin, 0);
  const int m_last = item_index(blk_end - 1, m_first);
  load_acts(m_first);
  cta_barrier();
  int m_act = m_first;
  // every warp passes every matrix change of the CTA's range, in order:
  // all warps done with the old activations, load, all loaded
  auto switch_to = [&](int m) {
    while (m_act < m) {
      cta_barrier();
      load_acts(++m_act);
      cta_barrier();
    }
  };

  // the first row of this warp at or after block blk
  auto seek = [&](Pos& c, int64_t blk) {
    for (; blk < blk_end; ++blk) {
      c.m = item_index(blk, c.m);
      const GemvItem& it = p.item[c.m];
      const int64_t r = (blk - it.blk_begin) * kRows + warp;
      if (r < it.rows) {
        c.blk = blk;
        c.rowe = r * it.cols;
        c.ch = 0;
        c.nch = static_cast<int>((it.cols + wcols - 1) >> wsh);
        return;
      }
    }
    c.blk = blk_end;
  };

  // this lane's package data of window c, into registers
  auto load = [&](const Pos& c, Window<F, K, B>& w) {
    if (c.blk >= blk_end) return;
    const GemvItem& it = p.item[c.m];
    const int64_t col = static_cast<int64_t>(c.ch) * wcols + lane * lc;
    if (col >= it.cols) return;  // beyond the row: never used
    const uint64_t e = static_cast<uint64_t>(c.rowe + col);
    const uint64_t g0 = e >> log2g;
#pragma unroll
    for (int i = 0; i < K; ++i) {
      if constexpr (kBits) {  // 8b bytes for 64 codes of width b, 4-byte aligned
        const int b = p.bits[i];
        const int words = nh * b;
        const uint32_t* src = reinterpret_cast<const uint32_t*>(it.codes[i]) + (e >> 5) * b;
        uint32_t wd[8];
#pragma unroll
        for (int t = 0; t < 8; ++t) wd[t] = t < words ? ld_nc4(src + t) : 0u;
        w.code[i][0] = make_uint4(wd[0], wd[1], wd[2], wd[3]);
        w.code[i][kBits ? 1 : 0] = make_uint4(wd[4], wd[5], wd[6], wd[7]);
      } else {
        const uint8_t* src = it.codes[i] + (e >> 2);
        if (lc >= 64) {
          w.code[i][0] = ld_nc16(src);
          if constexpr (Window<F, K, B>::kVecs > 1)
            if (lc == 128) w.code[i][Window<F, K, B>::kVecs - 1] = ld_nc16(src + 16);
        } else {
          const uint2 v = ld_nc8(src);
          w.code[i][0] = make_uint4(v.x, v.y, 0u, 0u);
        }
      }
      if constexpr (kF16) w.s[i] = ld_nc2(static_cast<const uint16_t*>(it.scales[i]) + g0);
      else w.s[i] = ld_nc4(static_cast<const uint32_t*>(it.scales[i]) + g0);
      if constexpr (!kSym) w.z[i] = __uint_as_float(ld_nc4(it.zeros[i] + g0));
    }
  };

  f32x2 acc[B];
#pragma unroll
  for (int b = 0; b < B; ++b) acc[b] = pack2(0.0f, 0.0f);

  // the k-stage prefix weights of a lane's window and their products with
  // the activations, four columns at a time
  auto window_dot = [&](const Pos& c, const Window<F, K, B>& w) {
    const GemvItem& it = p.item[c.m];
    const int64_t col = static_cast<int64_t>(c.ch) * wcols + lane * lc;
    if (col >= it.cols) return;  // beyond the row: nothing to add
    const float4* ap = act4 + ((c.ch << lsh) << 5) + lane;  // piece j of row b: ap[b * act_pieces + j * 32]
    auto dot = [&](int j, const f32x2& w01, const f32x2& w23) {
#pragma unroll
      for (int b = 0; b < B; ++b) {
        if (b < nb) {
          const float4 a = ap[b * act_pieces + j * 32];
          acc[b] = fma2(w01, pack2(a.x, a.y), acc[b]);
          acc[b] = fma2(w23, pack2(a.z, a.w), acc[b]);
        }
      }
    };
    if constexpr (kBits) {
      // per-stage widths: the reconstruction's width-generic stage sum
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        if (h >= nh) break;
        f32x2 v[16];
#pragma unroll
        for (int i = 0; i < K; ++i) {
          const float s = __uint_as_float(w.s[i]), z = w.z[i];
          const uint4 c0 = w.code[i][0], c1 = w.code[i][Window<F, K, B>::kVecs - 1];
          switch (p.bits[i]) {  // half h: words [h b, h b + b) of the window's 2b
            case 1: dequant_bits<1>(make_uint4(h ? c0.y : c0.x, 0u, 0u, 0u), s, z, i == 0, v); break;
            case 3:
              dequant_bits<3>(h ? make_uint4(c0.w, c1.x, c1.y, 0u) : make_uint4(c0.x, c0.y, c0.z, 0u), s, z, i == 0, v);
              break;
            case 4: dequant_bits<4>(h ? c1 : c0, s, z, i == 0, v); break;
            default:
              dequant_bits<2>(h ? make_uint4(c0.z, c0.w, 0u, 0u) : make_uint4(c0.x, c0.y, 0u, 0u), s, z, i == 0, v);
              break;
          }
        }
#pragma unroll
        for (int q = 0; q < 8; ++q) dot(8 * h + q, v[2 * q], v[2 * q + 1]);
      }
    } else {
      // the stage levels of each byte's four codes (asym_levels, sym_offsets)
      StageConsts c[K];
      bool fast = true;
#pragma unroll
      for (int i = 0; i < K; ++i) {
        const float s = kF16 ? __half2float(__ushort_as_half(static_cast<unsigned short>(w.s[i])))
                             : __uint_as_float(w.s[i]);
        if (!kSym) fast = fast && prescale_ok(s);  // symmetric levels need no condition
        c[i] = stage_consts(s, kSym ? 0.0f : w.z[i]);
      }
#pragma unroll
      for (int h = 0; h < kLCM / 32; ++h) {
        if (h >= nh) break;
        if (fast) {
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            f32x2 w01, w23;
#pragma unroll
            for (int i = 0; i < K; ++i) {
              const uint4 cw = w.code[i][h >> 1];
              const uint32_t word = (h & 1) == 0 ? (q < 4 ? cw.x : cw.y) : (q < 4 ? cw.z : cw.w);
              const uint32_t b8 = (q & 3) == 0 ? word : (word >> (8 * (q & 3)));
              if (kSym) {  // (Q - 2) s, exact; summed by one fma
                f32x2 u01, u23;
                sym_offsets(b8, u01, u23);
                w01 = (i == 0) ? mul2(u01, c[i].S) : fma2(u01, c[i].S, w01);
                w23 = (i == 0) ? mul2(u23, c[i].S) : fma2(u23, c[i].S, w23);
              } else {     // fl(zero + fl(Q s))
                f32x2 l01, l23;
                asym_levels(b8, c[i], l01, l23);
                w01 = (i == 0) ? l01 : add2(w01, l01);
                w23 = (i == 0) ? l23 : add2(w23, l23);
              }
            }
            dot(8 * h + q, w01, w23);
          }
        } else if constexpr (!kSym) {
          // an asymmetric scale outside [2^-100, 2^100]: unscaled codes,
          // fl(Q s) as a plain (t - 2^23) s
          const f32x2 T = pack2(kTwo23, kTwo23), Z0 = pack2(0.0f, 0.0f);
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            f32x2 w01, w23;
#pragma unroll
            for (int i = 0; i < K; ++i) {
              const uint4 cw = w.code[i][h >> 1];
              const uint32_t word = (h & 1) == 0 ? (q < 4 ? cw.x : cw.y) : (q < 4 ? cw.z : cw.w);
              const uint32_t b8 = (q & 3) == 0 ? word : (word >> (8 * (q & 3)));
              const f32x2 t01 = pack2u(magic23<3u>(b8), magic23<3u>(b8 >> 2));
              const f32x2 t23 = pack2u(magic23<3u>(b8 >> 4), magic23<3u>(b8 >> 6));
              const f32x2 l01 = add2(c[i].Z, fma2(sub2(t01, T), c[i].S, Z0));
              const f32x2 l23 = add2(c[i].Z, fma2(sub2(t23, T), c[i].S, Z0));
              w01 = (i == 0) ? l01 : add2(w01, l01);
              w23 = (i == 0) ? l23 : add2(w23, l23);
            }
            dot(8 * h + q, w01, w23);
          }
        }
      }
    }
  };

  // end of a row: reduce over the warp in a fixed order and store
  auto finish_row = [&](const Pos& c) {
    const GemvItem& it = p.item[c.m];
    const int64_t r = (c.blk - it.blk_begin) * kRows + warp;
#pragma unroll
    for (int b = 0; b < B; ++b) {
      float x, y;
      unpack2(acc[b], x, y);
      float t = __fadd_rn(x, y);
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) t = __fadd_rn(t, __shfl_xor_sync(kFullMask, t, off));
      if (lane == 0 && b < nb) it.Y[b * it.rows + r] = t;
      acc[b] = pack2(0.0f, 0.0f);
    }
  };

  // two windows in registers, loaded one ahead of use
  Pos pa{0, 0, m_first, 0, 0}, pb{0, 0, m_first, 0, 0};
  Window<F, K, B> wa{}, wb{};
  seek(pa, blk_begin);
  load(pa, wa);
  auto step = [&](const Pos& pc, const Window<F, K, B>& wc, Pos& pn, Window<F, K, B>& wn) -> bool {
    if (pc.blk >= blk_end) return false;
    pn = pc;
    if (++pn.ch >= pn.nch) seek(pn, pc.blk + 1);
    load(pn, wn);
    switch_to(pc.m);
    window_dot(pc, wc);
    if (pc.ch == pc.nch - 1) finish_row(pc);
    return true;
  };
  while (step(pa, wa, pb, wb) && step(pb, wb, pa, wa)) {
  }
  switch_to(m_last);
}

// activation floats per row a launch keeps for matrices of up to max_cols columns
constexpr int64_t act_floats_of(int64_t max_cols) {
  return ((max_cols + kWinCols - 1) / kWinCols) * kWinCols;
}
static_assert(act_floats_of(RRQ_MAX_GEMV_COLS) * 4 <= kMaxSmem &&
                  act_floats_of(RRQ_MAX_GEMV_COLS + 32) * 4 > kMaxSmem,
              "RRQ_MAX_GEMV_COLS is the widest row one activation row of a launch holds");
// activation rows one launch takes: as many as shared memory holds, and at
// most 4 at k = 4 (with 8 rows the k = 4 kernel runs out of registers; two
// launches of 4 are faster)
constexpr int max_rows_per_launch(int k) { return k == 4 ? 4 : kMaxGemvBatch; }
inline int tokens_per_launch(int64_t max_cols, int k) {
  const int64_t t = kMaxSmem / (act_floats_of(max_cols) * 4);
  return static_cast<int>(t < max_rows_per_launch(k) ? t : max_rows_per_launch(k));
}

template <int F, int K, int B>
cudaError_t launch_fkb(GemvBatch& p, int nb, int64_t max_cols, cudaStream_t stream, int sms) {
  // the kernel's dynamic shared memory limit is raised once per device
  // (prepare_format); the resident CTAs are asked for at this launch's size
  const int act_floats = static_cast<int>(act_floats_of(max_cols));
  const int smem = nb * act_floats * 4;
  int occ = 0;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, gemv_kernel<F, K, B>, kThreads, smem);
  if (e != cudaSuccess) return e;
  int64_t grid = static_cast<int64_t>(sms) * (occ < 1 ? 1 : occ);
  if (grid > kMaxGemvGrid) grid = kMaxGemvGrid;
  if (grid > p.total_blocks) grid = p.total_blocks;
  gemv_split(p, static_cast<int>(grid));
  gemv_kernel<F, K, B><<<p.grid, kThreads, smem, stream>>>(p, nb, act_floats);
  return cudaGetLastError();
}

template <int F, int K, int B>
cudaError_t prepare_fkb() {
  return cudaFuncSetAttribute(gemv_kernel<F, K, B>, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmem);
}

template <int F, int K>
cudaError_t prepare_fk() {
  cudaError_t e;
  if ((e = prepare_fkb<F, K, 1>())) return e;
  if ((e = prepare_fkb<F, K, 2>())) return e;
  if ((e = prepare_fkb<F, K, 4>())) return e;
  if constexpr (max_rows_per_launch(K) > 4) return prepare_fkb<F, K, 8>();
  return cudaSuccess;
}

// Once per device: every kernel of one format may take up to kMaxSmem bytes.
template <int F>
cudaError_t prepare_format() {
  cudaError_t e;
  if ((e = prepare_fk<F, 1>())) return e;
  if ((e = prepare_fk<F, 2>())) return e;
  if ((e = prepare_fk<F, 3>())) return e;
  return prepare_fk<F, 4>();
}

template <int F, int K>
cudaError_t launch_fk(int nb, int64_t max_cols, GemvBatch& p, cudaStream_t stream, int sms) {
  if (nb > max_rows_per_launch(K)) return cudaErrorInvalidValue;
  if (nb <= 1) return launch_fkb<F, K, 1>(p, nb, max_cols, stream, sms);
  if (nb <= 2) return launch_fkb<F, K, 2>(p, nb, max_cols, stream, sms);
  if (nb <= 4) return launch_fkb<F, K, 4>(p, nb, max_cols, stream, sms);
  if constexpr (max_rows_per_launch(K) > 4) return launch_fkb<F, K, 8>(p, nb, max_cols, stream, sms);
  return cudaErrorInvalidValue;
}

// Launch of one format (instantiated by one translation unit each).
template <int F>
cudaError_t launch_format(int k, int nb, int64_t max_cols, GemvBatch& p, cudaStream_t stream, int sms) {
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
