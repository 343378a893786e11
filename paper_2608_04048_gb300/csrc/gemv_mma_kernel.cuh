// Stage-wise product for decoding on the tensor cores, in the per-group
// factored form of Appendix C's A W~ = A W_0 + sum_k A R_k.  Within one group
// g of one stage k every weight is lo + Q s (asymmetric grid) or (Q - 2) s
// (symmetric), so
//     sum_{c in g} w_c a_c = s_kg * D_kg + lo_kg * S_g      (asymmetric)
//                          = s_kg * (D_kg - 2 S_g)          (symmetric)
// with D_kg = sum_{c in g} Q_c a_c over the integer codes and S_g = sum_{c in g}
// a_c.  The kernel forms D_kg with bf16 MMAs (mma.sync m16n8k16, binary32
// accumulation), the codes entering as the exact bf16 values 0..3, and sums
// the groups' terms per row.  It never forms the binary32 prefix weights W~;
// the result differs from A W~ by the rounding of the stage levels and of
// the sums (bounded below).
//
// Layout.  A CTA of 16 warps takes a contiguous range of 16-row blocks
// (gemv_split), matrix by matrix; a warp takes whole blocks (w, w + 16, ...
// of the CTA's blocks of a matrix).  Where some CTA holds fewer than 16
// blocks (a launch over few rows, such as the matrices of one layer), groups
// of P warps share each block instead, each warp taking every P-th item, and
// the group adds its parts of the rows' sums in warp order.  A block is walked stage by stage, each
// stage in spans of kSpan = max(512, G) columns: the item (block, stage,
// span) is 16 rows x kSpan/4 contiguous bytes of codes per row -- whole
// 128-byte lines, so that each DRAM page opened for a row serves a whole
// line, not the 32 bytes of one group -- and the rows' scales and zeros of
// the span's groups.  The warp's lanes copy items with cp.async into a ring
// of D slots of the warp's own in shared memory, D - 1 items ahead of the one
// it multiplies (rows padded so that the fragment reads below hit distinct
// banks).  Within a group, lane l (t = l % 4, rq = l / 4) takes the codes of
// rows rq and rq + 8 of the block for the columns [t G/4, (t + 1) G/4) of the
// group: G/64 words of 16 codes per row.  One MMA takes, for each lane, the
// codes at bit offset 2e (e = 0..3) of the four bytes of one word: bytes 0
// and 2 (one register: the code field masked in place under the bf16
// exponent of 128, i.e. 128 + 4^e Q, brought to Q by one exact bf16x2 fma)
// as k = 2t, 2t + 1, bytes 1 and 3 as k = 2t + 8, 2t + 9.  The permutation of
// K this implies is applied to the activations: per matrix the CTA writes
// them once, as bf16, into shared memory in exactly the B-fragment order of
// every MMA (each lane then reads 8 bytes per MMA), with the group sums S_g
// next to them.  Activation rows n >= nb of the launch are zero in B.  The
// accumulator rows are the block's rows and its columns the activation rows:
// lane l holds rows rq, rq + 8 for activation rows 2t, 2t + 1.
//
// Accuracy (binary32, round to nearest; the tensor cores' accumulation is
// assumed to round each k16 step once, as for the prefill product): the
// result differs from the oracle's binary64 sum of A W~ by at most
//     d * 2^-24 * sum_c sum_k (|lo_k| + 3 s_k) |a_c|     (asymmetric)
//     d * 2^-24 * sum_c sum_k 2 s_k |a_c|                 (symmetric)
// with d = (k + 1) + G/16 + 8 + 2k groups + 18: the stage levels and their
// sum that W~ rounds (k + 1), the G/16 MMA steps of D, the sum S_g (a sum of
// 8 then a tree over G/8, at most 8 roundings at G = 256), two fma per group
// and stage into the row's sum, and slack (18, which also covers the P - 1 <=
// 15 additions of a group's parts: each part holds fewer of the row's terms).
#pragma once

#include <cuda_bf16.h>

#include "gemv_kernel.cuh"

namespace rrq {
namespace {

constexpr int kMmaWarps = 16;
constexpr int kMmaThreads = kMmaWarps * 32;
constexpr int kMmaRingMax = 4;  // slots of a warp's ring at most
constexpr int kMmaSmemMax = kMaxSmem - 128;  // dynamic shared memory (the kernel has 32 static bytes)

// The item geometry for groups of G columns and spans of S columns (512
// or 1024, at least G): kL = S / G groups per item; a slot row holds the
// span's codes (S / 4 bytes) and a pad that puts the rows rq = 0..7 (G = 64:
// 4-byte reads), 0..3 (G = 128: 8-byte) or 0..1 (G = 256: 16-byte reads) of
// one read phase on distinct banks.
__host__ __device__ constexpr int mma_pitch(int G, int S) { return S / 4 + (G == 64 ? 16 : G == 128 ? 32 : 64); }
// one ring slot: 16 rows of codes, then the 16 x kL scales (binary32, or the
// aligned binary16 pair holding the scale) and, on the asymmetric grid, the
// 16 x kL zeros
__host__ __device__ constexpr int mma_slot_bytes(bool sym, int G, int S) {
  return kGemvRows * mma_pitch(G, S) + (sym ? 1 : 2) * kGemvRows * (S / G) * 4;
}

// shared memory of the per-matrix tables: per activation row, B fragments
// (cols bf16, two MMAs' fragments of a lane in 16 bytes) and 64 bytes of pad
// (rows 2 apart start on other banks), then per row the group sums (cols / G
// floats, rounded up to 4); the whole rounded up to 128 bytes
__host__ __device__ constexpr int64_t mma_brow_bytes(int64_t cols) { return cols * 2 + 64; }
__host__ __device__ constexpr int64_t mma_srow_floats(int64_t cols, int G) { return (cols / G + 3) / 4 * 4; }
__host__ __device__ constexpr int64_t mma_table_bytes(int64_t cols, int nb, int G) {
  return (nb * mma_brow_bytes(cols) + nb * mma_srow_floats(cols, G) * 4 + 127) / 128 * 128;
}
// ring slots a launch gives each warp: up to kMmaRingMax within what the
// tables leave of the shared memory (0 if not even 2 fit)
__host__ __device__ constexpr int mma_ring_slots(bool sym, int G, int S, int64_t table_bytes, int64_t smem_max) {
  const int64_t fit = (smem_max - table_bytes) / (kMmaWarps * static_cast<int64_t>(mma_slot_bytes(sym, G, S)));
  const int64_t d = fit < kMmaRingMax ? fit : kMmaRingMax;
  return d < 2 ? 0 : static_cast<int>(d);
}

// named barrier `id` over `count` threads (whole warps)
__device__ __forceinline__ void named_barrier(int id, int count) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// wait until at most n (< kMmaRingMax) of this thread's cp.async groups are pending
__device__ __forceinline__ void cp_async_wait_n(int n) {
  if (n <= 1) cp_async_wait<1>();
  else if (n == 2) cp_async_wait<2>();
  else cp_async_wait<3>();
}

__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// The code field at bit 2f (f <= 2) of a half, masked with the exponent bits
// clear, is the bf16 subnormal 4^f Q 2^-133 (exact: the tensor cores take
// subnormal bf16 operands as they are).  Register r of MMA e takes bytes 0, 2
// (r = 0) or 1, 3 (r = 1) of the lane's word at code offset e from the word or
// its shifts by 6 and 12; frag_f gives its f.  The B fragment of that register
// carries b 2^(k - 2f), so that each product is Q b 2^(k - 133).
__host__ __device__ constexpr int frag_f(int e, int r) {
  return r == 0 ? (e == 3 ? 0 : e) : (e == 2 ? 0 : e == 3 ? 1 : e + 1);
}
template <int E>
__device__ __forceinline__ void a_frag(uint32_t w0, uint32_t w1, uint32_t x6_0, uint32_t x6_1, uint32_t x12_0,
                                       uint32_t x12_1, uint32_t (&a)[4]) {
  constexpr uint32_t M0 = 0x00030003u, M1 = 0x000C000Cu, M2 = 0x00300030u;  // f = 0, 1, 2 in both halves
  if constexpr (E == 0) {         // bytes 0, 2 bits 0-1 (w);  bytes 1, 3 bits 0-1 (w >> 6, f = 1)
    a[0] = w0 & M0; a[1] = w1 & M0; a[2] = x6_0 & M1; a[3] = x6_1 & M1;
  } else if constexpr (E == 1) {  // bits 2-3 (w, f = 1);      bits 2-3 (w >> 6, f = 2)
    a[0] = w0 & M1; a[1] = w1 & M1; a[2] = x6_0 & M2; a[3] = x6_1 & M2;
  } else if constexpr (E == 2) {  // bits 4-5 (w, f = 2);      bits 4-5 (w >> 12, f = 0)
    a[0] = w0 & M2; a[1] = w1 & M2; a[2] = x12_0 & M0; a[3] = x12_1 & M0;
  } else {                        // bits 6-7 (w >> 6, f = 0); bits 6-7 (w >> 12, f = 1)
    a[0] = x6_0 & M0; a[1] = x6_1 & M0; a[2] = x12_0 & M1; a[3] = x12_1 & M1;
  }
}

// N consecutive 4-byte words of shared memory (N = 2: 8-byte aligned; N = 4:
// 16-byte aligned) into registers, one read
template <int N, typename T>
__device__ __forceinline__ void lds_vec(const void* p, T (&v)[N]) {
  static_assert(sizeof(T) == 4 && (N == 2 || N == 4), "two or four words");
  if constexpr (N == 2) {
    const uint2 x = *reinterpret_cast<const uint2*>(p);
    v[0] = __builtin_bit_cast(T, x.x); v[1] = __builtin_bit_cast(T, x.y);
  } else {
    const uint4 x = *reinterpret_cast<const uint4*>(p);
    v[0] = __builtin_bit_cast(T, x.x); v[1] = __builtin_bit_cast(T, x.y);
    v[2] = __builtin_bit_cast(T, x.z); v[3] = __builtin_bit_cast(T, x.w);
  }
}

// kGrp: blocks shared by groups of P > 1 warps (else P = 1, compiled out)
template <int F, int K, int G, int S, bool kGrp>
__global__ void __launch_bounds__(kMmaThreads, 1)
gemv_mma_kernel(const __grid_constant__ GemvBatch p, int nb, int ring_off, int D, int P_arg, int red_off) {
  const int P = kGrp ? P_arg : 1;
  constexpr bool kSym = F == kSymF32 || F == kSymF16;
  constexpr bool kF16 = F == kSymF16;
  constexpr int W = G / 64;  // words of 16 codes per lane, row and group
  constexpr int kSpan = S, kL = S / G, kPitch = mma_pitch(G, S);
  constexpr int kP = S / 64;                   // 16-byte pieces of a row's codes in a span
  constexpr int kCopies = kGemvRows * kP / 32;  // pieces a lane copies per item
  static_assert(S % G == 0 && kP <= 32, "a span is whole groups, a row at most one warp's pieces");
  constexpr int kCodes = kGemvRows * kPitch;   // a slot's codes
  constexpr int kSlot = mma_slot_bytes(kSym, G, S);
  extern __shared__ __align__(16) uint8_t smem[];
  const int lane = threadIdx.x & 31;
  // the warp index by broadcast: the compiler then treats it, and the item
  // and copy addresses derived from it, as warp-uniform
  const int warp = __shfl_sync(kFullMask, static_cast<int>(threadIdx.x >> 5), 0);
  const int t = lane & 3, rq = lane >> 2;
  const int64_t blk_begin = p.cta_begin[blockIdx.x];
  const int64_t blk_end = p.cta_begin[blockIdx.x + 1];
  if (blk_begin >= blk_end) return;  // the whole CTA: no barrier is reached

  int m_cur = -1;
  int64_t cols = 0, ngroups = 0;
  uint4* btab = nullptr;
  float* stab = nullptr;
  int64_t srow = 0;  // floats per row of the group sums

  // B fragments and group sums of matrix m, per activation row n: for column
  // c of group g, the lane quarter t = (c % G) / (G/4), word w, byte b and
  // offset e of its code give MMA i = (g W + w) 4 + e, register b & 1, half
  // b >> 1 of the fragment (n, i, t), stored at 16-byte unit (n, i / 2, t),
  // 8-byte half i % 2, and holding a_c 2^(k_n - 2f); S_g 2^(k_n - 133) of row
  // n at (n, g).  k_n = 253 - (the largest exponent field of the row's bf16
  // activations) keeps every scaled activation below 2^127; the row sums are
  // formed in the domain scaled by 2^(k_n - 133) and scaled back at the
  // store.  A lane reads activation row min(rq, nb - 1) of B and the sums of
  // rows min(2t, nb - 1), min(2t + 1, nb - 1): accumulator columns n >= nb
  // repeat a real row and are never stored.
  __shared__ int emax_s[kMaxGemvBatch];
  const uint4* bt_lane = nullptr;
  const float *sa_lane = nullptr, *sb_lane = nullptr;
  int back0 = 0, back1 = 0;  // 133 - k of the lane's output columns 2t, 2t + 1
  auto build_tables = [&](int m) {
    const GemvItem& it = p.item[m];
    cols = it.cols;
    ngroups = cols / G;
    const int64_t brow = mma_brow_bytes(cols) / 16;  // 16-byte units per B row
    srow = mma_srow_floats(cols, G);
    btab = reinterpret_cast<uint4*>(smem);
    stab = reinterpret_cast<float*>(smem + nb * mma_brow_bytes(cols));
    if (threadIdx.x < nb) emax_s[threadIdx.x] = 0;
    __syncthreads();
    // The activations in 16-byte chunks of 8 columns, chunk q = n cols/8 +
    // (column / 8) at thread q % 512: a group's G/8 chunks are consecutive
    // lanes of one warp, in one row (cols / 8 is a multiple of G / 8).
    // Pass 1: the row's largest exponent field, and S_g
    // as the sums of 8 consecutive activations (left to right) added by a
    // tree over the G / 8 (lane q + h into lane q, h = G/16 .. 1).
    const int64_t cpr = cols / 8;  // chunks per row
    const int64_t nch = cpr * nb;
    for (int64_t q0 = threadIdx.x - lane; q0 < nch; q0 += kMmaThreads) {  // warp-uniform
      const int64_t q = q0 + lane;
      const bool ok = q < nch;
      const int n = static_cast<int>((ok ? q : q0) / cpr);
      uint4 v = make_uint4(0u, 0u, 0u, 0u);
      if (ok) v = *reinterpret_cast<const uint4*>(it.A + static_cast<int64_t>(n) * cols + (q - n * cpr) * 8);
      const uint32_t h[8] = {v.x & 0xFFFFu, v.x >> 16, v.y & 0xFFFFu, v.y >> 16,
                             v.z & 0xFFFFu, v.z >> 16, v.w & 0xFFFFu, v.w >> 16};
      int e = 0;
      float sum = __uint_as_float(h[0] << 16);
#pragma unroll
      for (int i = 0; i < 8; ++i) e = max(e, static_cast<int>((h[i] >> 7) & 0xFF));
#pragma unroll
      for (int i = 1; i < 8; ++i) sum = __fadd_rn(sum, __uint_as_float(h[i] << 16));
#pragma unroll
      for (int hh = G / 16; hh >= 1; hh >>= 1) {
        sum = __fadd_rn(sum, __shfl_down_sync(kFullMask, sum, hh, G / 8));
        e = max(e, __shfl_down_sync(kFullMask, e, hh, G / 8));
      }
      if (ok && (lane % (G / 8)) == 0) {  // the group's first chunk
        atomicMax(&emax_s[n], e);
        stab[n * srow + (q - n * cpr) / (G / 8)] = sum;
      }
    }
    __syncthreads();
    // Pass 2: the B fragments a_c 2^(k_n - 2f), and S_g 2^(k_n - 133).
    uint16_t* bh = reinterpret_cast<uint16_t*>(btab);
    for (int64_t q = threadIdx.x; q < nch; q += kMmaThreads) {
      const int n = static_cast<int>(q / cpr);
      const int64_t c0 = (q - n * cpr) * 8;
      const int kn = 253 - emax_s[n];
      const uint4 v = *reinterpret_cast<const uint4*>(it.A + static_cast<int64_t>(n) * cols + c0);
      const uint32_t h[8] = {v.x & 0xFFFFu, v.x >> 16, v.y & 0xFFFFu, v.y >> 16,
                             v.z & 0xFFFFu, v.z >> 16, v.w & 0xFFFFu, v.w >> 16};
      const int64_t g = c0 / G;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int cg = static_cast<int>((c0 + i) % G);
        const int tq = cg / (G / 4), u = cg % (G / 4);
        const int w = u >> 4, vv = u & 15, b = vv >> 2, e = vv & 3;
        const int64_t mi = (g * W + w) * 4 + e;
        const float x = scalbnf(__uint_as_float(h[i] << 16), kn - 2 * frag_f(e, b & 1));
        bh[(n * brow + (mi >> 1) * 4 + tq) * 8 + (mi & 1) * 4 + (b & 1) * 2 + (b >> 1)] =
            __bfloat16_as_ushort(__float2bfloat16_rn(x));
      }
      if (c0 % G == 0) stab[n * srow + g] = scalbnf(stab[n * srow + g], kn - 133);
    }
    __syncthreads();
    const int bn = rq < nb ? rq : nb - 1;
    const int n0 = 2 * t < nb ? 2 * t : nb - 1, n1 = 2 * t + 1 < nb ? 2 * t + 1 : nb - 1;
    bt_lane = btab + bn * brow + t;
    sa_lane = stab + n0 * srow;
    sb_lane = stab + n1 * srow;
    back0 = emax_s[n0] - 120;
    back1 = emax_s[n1] - 120;
  };

  // This warp's ring: item j of its current matrix in slot j % D.
  uint8_t* const ring = smem + ring_off + static_cast<int64_t>(warp) * D * kSlot;
  const uint32_t ring_s = smem_u32(ring);

  // The lanes' copies of item (block from row r0, stage k, span sp): piece i
  // of a lane is the 16 bytes at part lane % kP of row lane / kP + (32 / kP) i
  // of the span's codes (a warp's copy instruction covers whole rows of S / 4
  // bytes); entry i (e = lane + 32 i < 16 kL) is the scale (and zero) of row
  // lane / kL + (32 / kL) i, group lane % kL of the span.  The lane keeps its
  // first piece and entry per (block, stage); rows past the matrix are not
  // copied (their sums are never stored), nor groups past the row's end.
  constexpr int kEntries = (kGemvRows * kL + 31) / 32;
  static_assert(32 % kL == 0, "a lane's entries are one group of rows 32 / kL apart");
  const uint8_t* cbase = nullptr;  // the lane's first piece in span 0
  const void* sbase = nullptr;     // its first entry's scale (binary32 or binary16) in group 0
  const float* zbase = nullptr;    // and zero
  int64_t xbase = 0;               // element index of the first entry in group 0
  int vrows = 0;                   // rows of the block in the matrix
  auto set_stage = [&](const GemvItem& it, int64_t r0, int k) {
    vrows = it.rows - r0 < kGemvRows ? static_cast<int>(it.rows - r0) : kGemvRows;
    cbase = it.codes[k] + (r0 + lane / kP) * (cols / 4) + (lane % kP) * 16;
    xbase = (r0 + lane / kL) * ngroups + lane % kL;
    sbase = it.scales[k];
    zbase = it.zeros[k];
  };
  auto issue = [&](const GemvItem& it, int sp, uint32_t dst) {
    const int64_t g0 = static_cast<int64_t>(sp) * kL;
    const int lg = ngroups - g0 < kL ? static_cast<int>(ngroups - g0) : kL;  // groups of this span
    const uint8_t* src = cbase + g0 * (G / 4);
    const int64_t cstep = (32 / kP) * (cols / 4);  // bytes between a lane's pieces
#pragma unroll
    for (int i = 0; i < kCopies; ++i, src += cstep) {
      const int row = lane / kP + (32 / kP) * i;
      if (row < vrows && (lg == kL || (lane % kP) * 16 < lg * (G / 4)))
        cp_async_16(dst + row * kPitch + (lane % kP) * 16, src, 16);
    }
    int64_t x = xbase + g0;
#pragma unroll
    for (int i = 0; i < kEntries; ++i, x += (32 / kL) * ngroups) {
      const int e = lane + 32 * i;
      const int row = lane / kL + (32 / kL) * i;
      if (e < kGemvRows * kL && row < vrows && (lg == kL || lane % kL < lg)) {
        const uint32_t md = dst + kCodes + e * 4;
        if constexpr (kF16) {  // the 4-byte aligned pair holding the scale (2 bytes at the array's end)
          const int64_t xa = x & ~static_cast<int64_t>(1);
          cp_async_4(md, static_cast<const uint16_t*>(sbase) + xa, xa + 1 < it.rows * ngroups ? 4u : 2u);
        } else {
          cp_async_4(md, static_cast<const float*>(sbase) + x, 4);
          if constexpr (!kSym) cp_async_4(md + kGemvRows * kL * 4, zbase + x, 4);
        }
      }
    }
  };

  // The CTA's range, matrix by matrix: the tables are built for a matrix,
  // then each warp (P = 1), or each group of P warps, takes whole blocks of
  // it (blocks q, q + 16/P, ... for group q).  A block is walked item by item
  // (item i: stage i / nspan, span i % nspan); warp j of a group takes items
  // j, j + P, ..., D - 1 items in flight.  With P > 1 the group's warps sum
  // their parts of a block's rows in shared memory, in warp order, behind
  // named barrier 1 + q.
  const int ngrp = kMmaWarps / P;
  const int grp = warp / P, wj = warp % P;
  // the item in slot `sl`: span sp of rows r0 (= block row + rq), r0 + 8 of a
  // stage, into the row sums y (rows r0 (0, 1) and r0 + 8 (2, 3); activation
  // rows 2t, 2t + 1)
  auto item = [&](float (&y)[4], const uint8_t* sl, int64_t r0, int sp) {
    const uint32_t* ssl = reinterpret_cast<const uint32_t*>(sl + kCodes);  // [16][kL]
    const float* zsl = reinterpret_cast<const float*>(sl + kCodes) + kGemvRows * kL;
    const int64_t g0 = static_cast<int64_t>(sp) * kL;
    const int lg = ngroups - g0 < kL ? static_cast<int>(ngroups - g0) : kL;
    // one group of the item: D by G/16 MMAs, then the row sums with the
    // rows' scales s0, s1, offsets o0, o1 (lo, or -2 s) and the sums sa, sb
    auto group = [&](int gi, float s0, float s1, float o0, float o1, float sa, float sb) {
      const int64_t g = g0 + gi;
      // the lane's W words of rows rq and rq + 8 (one read each)
      uint32_t c0[W], c1[W];
      const uint8_t* cb = sl + gi * (G / 4) + t * (G / 16);
      if constexpr (W == 1) {
        c0[0] = *reinterpret_cast<const uint32_t*>(cb + rq * kPitch);
        c1[0] = *reinterpret_cast<const uint32_t*>(cb + (rq + 8) * kPitch);
      } else if constexpr (W == 2) {
        const uint2 x0 = *reinterpret_cast<const uint2*>(cb + rq * kPitch);
        const uint2 x1 = *reinterpret_cast<const uint2*>(cb + (rq + 8) * kPitch);
        c0[0] = x0.x; c0[1] = x0.y;
        c1[0] = x1.x; c1[1] = x1.y;
      } else {
        const uint4 x0 = *reinterpret_cast<const uint4*>(cb + rq * kPitch);
        const uint4 x1 = *reinterpret_cast<const uint4*>(cb + (rq + 8) * kPitch);
        c0[0] = x0.x; c0[1] = x0.y; c0[2] = x0.z; c0[3] = x0.w;
        c1[0] = x1.x; c1[1] = x1.y; c1[2] = x1.z; c1[3] = x1.w;
      }
      float d[4] = {0.0f, 0.0f, 0.0f, 0.0f};
      const uint4* bt = bt_lane + g * (W * 2 * 4);  // 16-byte units: MMA pairs x 4 lanes
#pragma unroll
      for (int w = 0; w < W; ++w) {
        const uint32_t x6_0 = c0[w] >> 6, x6_1 = c1[w] >> 6, x12_0 = c0[w] >> 12, x12_1 = c1[w] >> 12;
#pragma unroll
        for (int h = 0; h < 2; ++h) {  // MMAs e = 2h, 2h + 1: one 16-byte read of B
          const uint4 b = bt[(w * 2 + h) * 4];
          uint32_t a[4];
          if (h == 0) a_frag<0>(c0[w], c1[w], x6_0, x6_1, x12_0, x12_1, a);
          else a_frag<2>(c0[w], c1[w], x6_0, x6_1, x12_0, x12_1, a);
          mma_bf16_16816(d, a, b.x, b.y);
          if (h == 0) a_frag<1>(c0[w], c1[w], x6_0, x6_1, x12_0, x12_1, a);
          else a_frag<3>(c0[w], c1[w], x6_0, x6_1, x12_0, x12_1, a);
          mma_bf16_16816(d, a, b.z, b.w);
        }
      }
      // y += s D + lo S (asymmetric), s D - 2 s S (symmetric)
      y[0] = __fmaf_rn(o0, sa, __fmaf_rn(s0, d[0], y[0]));
      y[1] = __fmaf_rn(o0, sb, __fmaf_rn(s0, d[1], y[1]));
      y[2] = __fmaf_rn(o1, sa, __fmaf_rn(s1, d[2], y[2]));
      y[3] = __fmaf_rn(o1, sb, __fmaf_rn(s1, d[3], y[3]));
    };
    // a row's scale from its raw 4-byte word (binary16: the half holding element x)
    auto scale_of = [&](uint32_t u, int64_t x) -> float {
      if constexpr (kF16) {
        return __half2float(__ushort_as_half(static_cast<unsigned short>((x & 1) ? u >> 16 : u & 0xFFFFu)));
      } else {
        return __uint_as_float(u);
      }
    };
    const int64_t x0 = r0 * ngroups + g0, x1 = x0 + 8 * ngroups;  // scale element of rows rq, rq + 8 at g0
    if (lg == kL) {  // a whole span: C groups' scales, zeros and sums per read; their MMA chains interleave
      constexpr int C = kL < 4 ? kL : 4;
#pragma unroll
      for (int h = 0; h < kL; h += C) {
        uint32_t u0[C], u1[C];
        float z0[C], z1[C], sa[C], sb[C];
        lds_vec<C>(ssl + rq * kL + h, u0);
        lds_vec<C>(ssl + (rq + 8) * kL + h, u1);
        lds_vec<C>(sa_lane + g0 + h, sa);
        lds_vec<C>(sb_lane + g0 + h, sb);
        if constexpr (!kSym) {
          lds_vec<C>(zsl + rq * kL + h, z0);
          lds_vec<C>(zsl + (rq + 8) * kL + h, z1);
        }
#pragma unroll
        for (int i = 0; i < C; ++i) {
          const float s0 = scale_of(u0[i], x0 + h + i), s1 = scale_of(u1[i], x1 + h + i);
          group(h + i, s0, s1, kSym ? -2.0f * s0 : z0[i], kSym ? -2.0f * s1 : z1[i], sa[i], sb[i]);
        }
      }
    } else {
      for (int gi = 0; gi < lg; ++gi) {
        const float s0 = scale_of(ssl[rq * kL + gi], x0 + gi), s1 = scale_of(ssl[(rq + 8) * kL + gi], x1 + gi);
        const float o0 = kSym ? -2.0f * s0 : zsl[rq * kL + gi], o1 = kSym ? -2.0f * s1 : zsl[(rq + 8) * kL + gi];
        group(gi, s0, s1, o0, o1, sa_lane[g0 + gi], sb_lane[g0 + gi]);
      }
    }
  };
  auto store = [&](const float (&y)[4], const GemvItem& it, int64_t r0) {
    const int64_t r1 = r0 + 8;
    const int n0 = 2 * t, n1 = 2 * t + 1;
    if (r0 < it.rows) {
      if (n0 < nb) it.Y[static_cast<int64_t>(n0) * it.rows + r0] = scalbnf(y[0], back0);
      if (n1 < nb) it.Y[static_cast<int64_t>(n1) * it.rows + r0] = scalbnf(y[1], back1);
    }
    if (r1 < it.rows) {
      if (n0 < nb) it.Y[static_cast<int64_t>(n0) * it.rows + r1] = scalbnf(y[2], back0);
      if (n1 < nb) it.Y[static_cast<int64_t>(n1) * it.rows + r1] = scalbnf(y[3], back1);
    }
  };
  int m = 0;
  while (m + 1 < p.count && blk_begin >= p.item[m + 1].blk_begin) ++m;
  for (int64_t seg = blk_begin; seg < blk_end; ++m) {
    const GemvItem& it = p.item[m];
    const int64_t seg_end = m + 1 < p.count && p.item[m + 1].blk_begin < blk_end ? p.item[m + 1].blk_begin : blk_end;
    if (m_cur >= 0) __syncthreads();  // every warp is done with the old tables
    build_tables(m);
    m_cur = m;
    __syncthreads();
    const int nspan = static_cast<int>((cols + kSpan - 1) / kSpan);
    const int ipb = K * nspan;                                                    // items per block
    const int nblk = static_cast<int>((seg_end - seg - grp + ngrp - 1) / ngrp);  // may be <= 0
    const int64_t row_step = static_cast<int64_t>(ngrp) * kGemvRows;
    const int64_t r_first = (seg + grp - it.blk_begin) * kGemvRows;
    if constexpr (!kGrp) {
      // one warp per block: cursors (first row of the block, stage, span) of
      // the next item to copy and of the item to multiply
      const int items = nblk > 0 ? nblk * ipb : 0;
      int64_t ir = r_first;
      int is = 0, ik = 0, left = items;
      auto issue_next = [&](int s_dst) {
        if (left > 0) {
          if (is == 0) set_stage(it, ir, ik);
          issue(it, is, ring_s + s_dst * kSlot);
          --left;
          if (++is == nspan) {
            is = 0;
            if (++ik == K) ik = 0, ir += row_step;
          }
        }
        cp_async_commit();
      };
      for (int j = 0; j + 1 < D; ++j) issue_next(j);  // items 0 .. D - 2 (empty groups past the end)
      float y[4] = {0.0f, 0.0f, 0.0f, 0.0f};
      int slot = 0;  // j % D
      int64_t cr = r_first;
      int cs = 0, ck = 0;
      for (int j = 0; j < items; ++j) {
        // item j + D - 1 into the slot item j - 1 used (every lane is past it)
        issue_next(slot == 0 ? D - 1 : slot - 1);
        cp_async_wait_n(D - 1);  // this lane's copies of item j are done
        __syncwarp();            // and every lane's
        item(y, ring + slot * kSlot, cr + rq, cs);
        __syncwarp();  // every lane is done with the slot before it is refilled
        slot = slot + 1 == D ? 0 : slot + 1;
        if (++cs == nspan) {
          cs = 0;
          if (++ck == K) {  // the block's rows are complete: store and start over
            ck = 0;
            store(y, it, cr + rq);
            y[0] = y[1] = y[2] = y[3] = 0.0f;
            cr += row_step;
          }
        }
      }
    } else {
      // groups of P warps: cursors (first row of the block, stage, span) of
      // this warp's next item to copy and item to multiply; the block ends
      // when the stage passes K
      const int per = ipb > wj ? (ipb - wj + P - 1) / P : 0;  // this warp's items of a block
      struct Cur {
        int64_t r;
        int k, s;
      };
      const int k_first = wj / nspan, s_first = wj % nspan;
      auto advance = [&](Cur& c) {  // true if the stage or block changed
        c.s += P;
        if (c.s < nspan) return false;
        do c.s -= nspan, ++c.k;
        while (c.s >= nspan);
        if (c.k >= K) c.k = k_first, c.s = s_first, c.r += row_step;
        return true;
      };
      Cur ic{r_first, k_first, s_first};
      int left = nblk > 0 ? nblk * per : 0;
      bool fresh = true;  // the copy pointers are for another stage or block
      auto issue_next = [&](int s_dst) {
        if (left > 0) {
          if (fresh) set_stage(it, ic.r, ic.k);
          issue(it, ic.s, ring_s + s_dst * kSlot);
          --left;
          fresh = advance(ic);
        }
        cp_async_commit();
      };
      for (int j = 0; j + 1 < D; ++j) issue_next(j);
      int slot = 0;
      Cur cc{r_first, k_first, s_first};
      float* red = reinterpret_cast<float*>(smem + red_off);  // [16 warps][32 lanes][4]
      for (int b = 0; b < nblk; ++b) {
        float y[4] = {0.0f, 0.0f, 0.0f, 0.0f};
        const int64_t r0 = cc.r + rq;
        for (int u = 0; u < per; ++u) {
          issue_next(slot == 0 ? D - 1 : slot - 1);
          cp_async_wait_n(D - 1);
          __syncwarp();
          item(y, ring + slot * kSlot, cc.r + rq, cc.s);
          __syncwarp();
          slot = slot + 1 == D ? 0 : slot + 1;
          advance(cc);
        }
        // the block's rows are complete: sum the group's parts in warp order and store
        if (wj > 0) {
#pragma unroll
          for (int q = 0; q < 4; ++q) red[(warp * 32 + lane) * 4 + q] = y[q];
        }
        named_barrier(1 + grp, P * 32);
        if (wj == 0) {
          for (int j = 1; j < P; ++j)
#pragma unroll
            for (int q = 0; q < 4; ++q) y[q] = __fadd_rn(y[q], red[((warp + j) * 32 + lane) * 4 + q]);
          store(y, it, r0);
        }
        named_barrier(1 + grp, P * 32);  // the parts are read before the next block's
      }
    }
    cp_async_wait<0>();  // the empty groups of the last items
    seg = seg_end;
  }
}

// the group partial sums of a launch with more than one warp per block
constexpr int kMmaRedBytes = kMmaWarps * 32 * 4 * 4;

// activation rows one launch of the tensor-core form holds for matrices of up
// to max_cols columns, with a ring of at least 2 slots of 512-column spans a
// warp and the partial sums (0 if not even one row fits)
inline int mma_rows_per_launch(bool sym, int64_t max_cols, int group) {
  const int span = group > 512 ? group : 512;
  for (int nb = kMaxGemvBatch; nb >= 1; --nb)
    if (mma_ring_slots(sym, group, span, mma_table_bytes(max_cols, nb, group) + kMmaRedBytes, kMmaSmemMax) >= 2)
      return nb;
  return 0;
}

// Warps per block: 1 while every CTA holds at least 16 blocks; else the
// smallest CTA's blocks (rounded down to a power of two) times P make 16, so
// that each group of P warps has a block (launches over few rows, e.g. the
// matrices of one layer).
inline int mma_warps_per_block(const GemvBatch& p) {
  int64_t least = p.total_blocks;
  for (int c = 0; c < p.grid; ++c) {
    const int64_t n = p.cta_begin[c + 1] - p.cta_begin[c];
    if (n < least) least = n;
  }
  int P = 1;
  while (P < kMmaWarps && least * P < kMmaWarps) P *= 2;
  return P;
}

template <int F, int K, int G, int S>
cudaError_t mma_launch_kgs(GemvBatch& p, int nb, int64_t tables, int P, cudaStream_t stream, int D) {
  constexpr bool kSym = F == kSymF32 || F == kSymF16;
  const int64_t ring = static_cast<int64_t>(kMmaWarps) * D * mma_slot_bytes(kSym, G, S);
  const int red = P > 1 ? kMmaRedBytes : 0;
  const int smem = static_cast<int>(tables + ring + red);
  const int ring_off = static_cast<int>(tables), red_off = static_cast<int>(tables + ring);
  if (P > 1)
    gemv_mma_kernel<F, K, G, S, true><<<p.grid, kMmaThreads, smem, stream>>>(p, nb, ring_off, D, P, red_off);
  else
    gemv_mma_kernel<F, K, G, S, false><<<p.grid, kMmaThreads, smem, stream>>>(p, nb, ring_off, D, 1, red_off);
  return cudaGetLastError();
}

// spans of 1024 columns where groups of 128 or more leave room for a ring of
// at least 2 of them (half the per-item costs), else 512 (G = 64: 512 only)
template <int F, int K, int G>
cudaError_t mma_launch_kg(GemvBatch& p, int nb, int64_t max_cols, cudaStream_t stream, int sms) {
  constexpr bool kSym = F == kSymF32 || F == kSymF16;
  int64_t grid = sms;  // one 16-warp CTA per multiprocessor
  if (grid > kMaxGemvGrid) grid = kMaxGemvGrid;
  if (grid > p.total_blocks) grid = p.total_blocks;
  gemv_split(p, static_cast<int>(grid));
  const int P = mma_warps_per_block(p);
  const int64_t tables = mma_table_bytes(max_cols, nb, G);
  const int64_t fixed = tables + (P > 1 ? kMmaRedBytes : 0);
  if constexpr (G >= 128) {
    const int d = mma_ring_slots(kSym, G, 1024, fixed, kMmaSmemMax);
    if (d >= 2) return mma_launch_kgs<F, K, G, 1024>(p, nb, tables, P, stream, d);
  }
  constexpr int S0 = G > 512 ? G : 512;
  const int d = mma_ring_slots(kSym, G, S0, fixed, kMmaSmemMax);
  if (d < 2) return cudaErrorInvalidValue;  // the caller sizes nb by mma_rows_per_launch
  return mma_launch_kgs<F, K, G, S0>(p, nb, tables, P, stream, d);
}

template <int F, int K>
cudaError_t mma_launch_k(int group, GemvBatch& p, int nb, int64_t max_cols, cudaStream_t stream, int sms) {
  switch (group) {
    case 64: return mma_launch_kg<F, K, 64>(p, nb, max_cols, stream, sms);
    case 128: return mma_launch_kg<F, K, 128>(p, nb, max_cols, stream, sms);
    case 256: return mma_launch_kg<F, K, 256>(p, nb, max_cols, stream, sms);
    default: return cudaErrorInvalidValue;
  }
}

template <int F>
cudaError_t mma_launch_format(int group, int k, int nb, int64_t max_cols, GemvBatch& p, cudaStream_t stream, int sms) {
  switch (k) {
    case 1: return mma_launch_k<F, 1>(group, p, nb, max_cols, stream, sms);
    case 2: return mma_launch_k<F, 2>(group, p, nb, max_cols, stream, sms);
    case 3: return mma_launch_k<F, 3>(group, p, nb, max_cols, stream, sms);
    case 4: return mma_launch_k<F, 4>(group, p, nb, max_cols, stream, sms);
    default: return cudaErrorInvalidValue;
  }
}

template <int F, int K, int G, int S>
cudaError_t mma_prepare_kgs() {
  cudaError_t e;
  const cudaFuncAttribute a = cudaFuncAttributeMaxDynamicSharedMemorySize;
  if ((e = cudaFuncSetAttribute(gemv_mma_kernel<F, K, G, S, false>, a, kMmaSmemMax))) return e;
  return cudaFuncSetAttribute(gemv_mma_kernel<F, K, G, S, true>, a, kMmaSmemMax);
}

template <int F, int K>
cudaError_t mma_prepare_k() {
  cudaError_t e;
  if ((e = mma_prepare_kgs<F, K, 64, 512>())) return e;
  if ((e = mma_prepare_kgs<F, K, 128, 512>())) return e;
  if ((e = mma_prepare_kgs<F, K, 128, 1024>())) return e;
  if ((e = mma_prepare_kgs<F, K, 256, 512>())) return e;
  return mma_prepare_kgs<F, K, 256, 1024>();
}

template <int F>
cudaError_t mma_prepare_format() {
  cudaError_t e;
  if ((e = mma_prepare_k<F, 1>())) return e;
  if ((e = mma_prepare_k<F, 2>())) return e;
  if ((e = mma_prepare_k<F, 3>())) return e;
  return mma_prepare_k<F, 4>();
}

}  // namespace
}  // namespace rrq
