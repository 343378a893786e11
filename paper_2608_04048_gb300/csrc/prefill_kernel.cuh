// Prefill form of the stage-wise product (Appendix C, A W~_(t) = A W^_0 +
// sum_k A R^_k, for many activation rows) on the fifth-generation tensor
// cores:
//
//     Y[t][r] = sum_c A[t][c] * bf16(W~_k)[r][c]
//
// with bf16(W~_k) the prefix-k reconstruction (Eq. 8: acc = L_0; acc =
// fl(acc + L_i); bf16 round to nearest-even), formed from the package inside
// the kernel and never written to memory.  The tensor cores take bf16
// operands, so the weight is the reconstruction exactly as rrq_reconstruct
// returns it; products are accumulated in binary32 in tensor memory.
//
// One CTA computes a tile of 128 weight rows x 512 tokens: two accumulators
// of tcgen05.mma.cta_group::1.kind::f16 shape M = 128, N = 256 (K = 16 per
// instruction), which fill the 512 columns of tensor memory.  CS CTAs (1, 2
// or 4) with the same 128 rows and consecutive token tiles form a cluster
// that shares the weight tiles: each CTA forms 128/CS of the rows and sends
// them to the others, so a weight tile formed from the package serves
// 512 x CS tokens.  The K range is walked in stages of 64 columns:
//   - warp 8 loads the activation tile of a stage (512 tokens x 64 columns,
//     bf16, two 2-D TMA boxes, 128-byte swizzle) into a 2-deep ring;
//   - warp 10 loads the stage's codes of this CTA's rows (one 2-D TMA box of
//     16 bytes x 128/CS rows per package stage) into a 4-deep ring;
//   - warps 0-7 take the codes from that ring (or load them themselves when
//     a matrix's code rows are not 16-byte multiples, and for packages with
//     per-stage widths: b words per 32 weights, formed by the
//     reconstruction's width-generic routine) and the scales and
//     zeros as 16-byte blocks a block ahead, form this CTA's rows of the bf16
//     weight tile in registers and store them in the K-major
//     128-byte-swizzled layout into a 3-deep ring;
//   - in a cluster, warp 11 then copies those rows (contiguous in the
//     swizzled tile) into the same slot of every other CTA with one bulk
//     copy each, which completes there as transaction bytes of the slot's
//     "full" barrier; no thread issues a cluster-scope release;
//   - one thread of warp 9 issues the MMAs of the stage and commits them to
//     the activation ring's "empty" barrier and, multicast, to the weight
//     ring's "empty" barrier of every CTA of the cluster, so that no CTA
//     overwrites a slot before all have read it;
//   - after the last stage warps 0-7 read the accumulators (tcgen05.ld, one
//     TMEM lane = one weight row) and store Y with coalesced binary32 stores.
// Every wait is bounded in wall time; on expiry the kernel sets the status
// word, drains its own copies and MMAs (bounded) and frees its tensor memory;
// the CTAs of a cluster meet at a cluster barrier before any of them leaves.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "rrq_device.cuh"

#ifndef PF_PRODUCERS_CS4
#define PF_PRODUCERS_CS4 4
#endif
#ifndef PF_PRODUCERS_CS2
#define PF_PRODUCERS_CS2 4
#endif

namespace rrq {
namespace {

constexpr int kPfWStages = 3;                        // weight-tile ring depth
constexpr int kPfCStages = 4;                        // code-tile ring depth
constexpr int kPfAStages = 2;                        // activation-tile ring depth
constexpr int kPfWTileBytes = kPrefillBM * 128;      // 128 rows x 64 bf16 (16 KiB)
constexpr int kPfAHalfBytes = kPrefillMmaN * 128;    // 256 tokens x 64 bf16 (32 KiB)
constexpr int kPfATileBytes = 2 * kPfAHalfBytes;     // 512 tokens (64 KiB)
constexpr int kPfCTileBytes = kPrefillBM * 16;       // one package stage's codes of a stage (2 KiB)
constexpr int kPfCStageBytes = kMaxStages * kPfCTileBytes;
constexpr int kPfDqWarps = 8;                        // the epilogue (and weight tiles, below)
constexpr int kPfTmaWarp = 8;
constexpr int kPfMmaWarp = 9;
constexpr int kPfCodeWarp = 10;
constexpr int kPfShareWarp = 11;                     // clusters: sends this CTA's rows to the others
constexpr int kPfThreads = 12 * 32;
constexpr uint32_t kPfTmemCols = kPrefillBN;         // two binary32 accumulators, 128 lanes x 256 columns each
constexpr int kPfCOffset = kPfWStages * kPfWTileBytes + kPfAStages * kPfATileBytes;
constexpr int kPfBarOffset = kPfCOffset + kPfCStages * kPfCStageBytes;
// full_w, empty_w per weight stage; full_a, empty_a per activation stage;
// full_c, empty_c per code stage; acc_full; drain; share_done per weight stage
constexpr int kPfBars = 2 * kPfWStages + 2 * kPfAStages + 2 * kPfCStages + 2 + kPfWStages;
// after the barriers: the TMEM address (16 bytes), then for clusters the
// stages each CTA sent to this one [4] and the stages this CTA's MMA thread
// consumed (32 bytes), and alignment slack
constexpr int kPfSmemBytes = kPfBarOffset + 8 * kPfBars + 16 + 32 + 1024;

// Instruction descriptor of tcgen05.mma .kind::f16: D binary32 (bits 4-5),
// A and B bf16 (bits 7-9, 10-12), both K-major (bits 15, 16 clear),
// N >> 3 at bits 17-22, M >> 4 at bits 24-28.
constexpr uint32_t kPfIdesc = (1u << 4) | (1u << 7) | (1u << 10) |
                              (static_cast<uint32_t>(kPrefillMmaN >> 3) << 17) |
                              (static_cast<uint32_t>(kPrefillBM >> 4) << 24);

// Shared-memory matrix descriptor of a K-major tile with 128-byte swizzle:
// rows 128 bytes apart, 8-row groups 1024 bytes apart (stride byte offset),
// the tile base 1024-byte aligned (base offset 0), descriptor version 1,
// layout type 2 (128-byte swizzle) in bits 61-63.  The leading byte offset
// is not used by this layout (one swizzle row spans the MMA's K).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  return static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4) | (static_cast<uint64_t>(1) << 16) |
         (static_cast<uint64_t>(1024 >> 4) << 32) | (static_cast<uint64_t>(1) << 46) |
         (static_cast<uint64_t>(2) << 61);
}

__device__ __forceinline__ void tmem_alloc(uint32_t slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(slot), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// D (tensor memory) = A B^T (+ D if acc != 0), A and B from shared memory.
__device__ __forceinline__ void mma_bf16(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d),
      "l"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}
// Arrives on `bar` once every MMA issued so far by this thread has completed.
__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}
// Counts `bytes` of the barrier's current phase as arrived without a copy
// (settles an expectation that no copy will meet).
__device__ __forceinline__ void mbar_complete_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.complete_tx.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
// 32-bit store into the shared memory of a CTA of the cluster (address from
// cluster_addr).
__device__ __forceinline__ void st_cluster_u32(uint32_t addr, uint32_t v) {
  asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}
// Cluster forms: the address of the same shared-memory offset in CTA `rank`
// of the cluster, an MMA commit that arrives on the barrier at the same
// offset in every CTA of `mask`, and the cluster-wide barrier.
__device__ __forceinline__ uint32_t cluster_addr(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}
__device__ __forceinline__ void mma_commit_multicast(uint32_t bar, uint16_t mask) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(bar),
      "h"(mask)
      : "memory");
}
// shared -> shared bulk copy into CTA dst's memory (cluster addresses of the
// destination and of its barrier), completing there as transaction bytes
__device__ __forceinline__ void bulk_copy_cluster(uint32_t dst, uint32_t src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "r"(src), "r"(bytes), "r"(bar)
               : "memory");
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// 2-D tiled TMA load: box at (x = column, y = row) of `map`, completing on `bar`.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
// 32 consecutive binary32 columns of this thread's tensor-memory lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
        "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]),
        "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]),
        "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Bounded wait that sleeps in the barrier (rrq_device.cuh).
__device__ __forceinline__ bool pf_wait(uint32_t bar, uint32_t parity, uint32_t limit_us) {
  return mbar_wait_sleep(bar, parity, limit_us);
}

// Package words of the 32 consecutive weights (one group) a thread forms in
// one stage.
template <int K>
struct PkgWords {
  uint2 cw[K];   // stage-i codes, LSB first, 2 bits each
  uint4 cb[K];   // per-stage widths: stage-i codes, b 32-bit words (b = the stage's width)
  float sc[K];   // stage-i scale
  float zr[K];   // stage-i zero (asymmetric grid)
};

// Scales (and zeros) of 16 consecutive bytes of one row: 4 binary32 or 8
// binary16 groups, loaded as one vector per package stage.
template <int K>
struct ScaleBlock {
  uint4 s[K];
  uint4 z[K];
};

template <int F>
__host__ __device__ constexpr int groups_per_block() { return F == kSymF16 ? 8 : 4; }

template <int F, int K>
__device__ __forceinline__ void load_block(const PrefillItem& it, int64_t b, ScaleBlock<K>& sb) {
#pragma unroll
  for (int i = 0; i < K; ++i) {
    sb.s[i] = __ldg(static_cast<const uint4*>(it.scales[i]) + b);
    if constexpr (F == kAsymF32 || F == kAsymBits) sb.z[i] = __ldg(reinterpret_cast<const uint4*>(it.zeros[i]) + b);
  }
}

__device__ __forceinline__ uint32_t pick_word(const uint4& v, int j) {
  return (j & 2) ? ((j & 1) ? v.w : v.z) : ((j & 1) ? v.y : v.x);
}

// stage-i scale and zero of group gi (0 .. groups_per_block - 1) of a block
template <int F, int K>
__device__ __forceinline__ void from_block(const ScaleBlock<K>& sb, int gi, PkgWords<K>& w) {
#pragma unroll
  for (int i = 0; i < K; ++i) {
    if constexpr (F == kSymF16) {
      const uint32_t word = pick_word(sb.s[i], gi >> 1);
      w.sc[i] = __half2float(__ushort_as_half(static_cast<unsigned short>((gi & 1) ? (word >> 16) : (word & 0xffffu))));
    } else {
      w.sc[i] = __uint_as_float(pick_word(sb.s[i], gi));
    }
    w.zr[i] = (F == kAsymF32 || F == kAsymBits) ? __uint_as_float(pick_word(sb.z[i], gi)) : 0.0f;
  }
}

// stage-i scale and zero of group g, one scalar load each
template <int F, int K>
__device__ __forceinline__ void load_scales(const PrefillItem& it, int64_t g, PkgWords<K>& w) {
#pragma unroll
  for (int i = 0; i < K; ++i) {
    if constexpr (F == kSymF16)
      w.sc[i] = __half2float(__ushort_as_half(__ldg(static_cast<const unsigned short*>(it.scales[i]) + g)));
    else
      w.sc[i] = __ldg(static_cast<const float*>(it.scales[i]) + g);
    w.zr[i] = (F == kAsymF32 || F == kAsymBits) ? __ldg(it.zeros[i] + g) : 0.0f;
  }
}

// bf16 prefix-k weights of the first NW (8, 16 or 32) of those weights: acc =
// L_0; acc = fl(acc + L_i);
// bf16 nearest-even.  L_i = fl(zero + fl(Q s)) (asymmetric) or (Q - 2) s
// (symmetric, exact).  Two evaluations of fl(Q s), both exact to the same
// bits: with prescale_ok(s) each code stays in its bit field (value 4^j Q
// for the j-th code of a byte) and one fma with s / 4^j and -2^23 s / 4^j
// rounds Q s once; otherwise the code is shifted down and fma(Q, s, 0).
// (The decode product and the reconstruction use the other placement of the
// same trick, asym_levels: one exponent per code position and one scale.  In
// this kernel the form here measured 1 % faster at k = 2..4.)
template <int F, int K, int NW>
__device__ __forceinline__ void prefix_weights_bf16(const PkgWords<K>& w, uint32_t (&h)[NW / 2]) {
  constexpr bool kSym = F == kSymF32 || F == kSymF16;
  constexpr float kT23 = 8388608.0f;
  f32x2 acc[NW / 2];
#pragma unroll
  for (int i = 0; i < K; ++i) {
    const float s = w.sc[i];
    if (prescale_ok(s)) {
      const f32x2 S01 = pack2(s, __fmul_rn(s, 0x1p-2f)), S23 = pack2(__fmul_rn(s, 0x1p-4f), __fmul_rn(s, 0x1p-6f));
      const f32x2 LO = pack2(w.zr[i], w.zr[i]);
      const f32x2 C01 = pack2(__fmul_rn(s, -0x1p23f), __fmul_rn(s, -0x1p21f));
      const f32x2 C23 = pack2(__fmul_rn(s, -0x1p19f), __fmul_rn(s, -0x1p17f));
      const f32x2 K01 = pack2(kT23 + 2.0f, kT23 + 8.0f), K23 = pack2(kT23 + 32.0f, kT23 + 128.0f);
#pragma unroll
      for (int j = 0; j < NW / 4; ++j) {  // byte j: weights 4j..4j+3 (pairs 2j, 2j+1)
        const uint32_t word = j < 4 ? w.cw[i].x : w.cw[i].y;
        const uint32_t b = (j & 3) == 0 ? word : (word >> (8 * (j & 3)));
        const f32x2 t01 = pack2u(magic23<0x03u>(b), magic23<0x0Cu>(b));
        const f32x2 t23 = pack2u(magic23<0x30u>(b), magic23<0xC0u>(b));
        if constexpr (kSym) {  // 4^j (Q - 2), exact; times s / 4^j exact
          const f32x2 u01 = sub2(t01, K01), u23 = sub2(t23, K23);
          acc[2 * j] = (i == 0) ? mul2(u01, S01) : fma2(u01, S01, acc[2 * j]);
          acc[2 * j + 1] = (i == 0) ? mul2(u23, S23) : fma2(u23, S23, acc[2 * j + 1]);
        } else {
          const f32x2 l01 = add2(LO, fma2(t01, S01, C01));
          const f32x2 l23 = add2(LO, fma2(t23, S23, C23));
          acc[2 * j] = (i == 0) ? l01 : add2(acc[2 * j], l01);
          acc[2 * j + 1] = (i == 0) ? l23 : add2(acc[2 * j + 1], l23);
        }
      }
    } else {
      const f32x2 S = pack2(s, s);
      const f32x2 LO = pack2(w.zr[i], w.zr[i]), Z = pack2(0.0f, 0.0f);
      const f32x2 T23 = pack2(kT23, kT23), K2 = pack2(kT23 + 2.0f, kT23 + 2.0f);
#pragma unroll
      for (int m = 0; m < NW / 2; ++m) {
        const uint32_t word = m < 8 ? w.cw[i].x : w.cw[i].y;
        const int sh = 4 * (m & 7);
        const f32x2 t = pack2u(magic23<3u>(word >> sh), magic23<3u>(word >> (sh + 2)));
        if constexpr (kSym) {
          const f32x2 u = sub2(t, K2);  // Q - 2, exact
          acc[m] = (i == 0) ? mul2(u, S) : fma2(u, S, acc[m]);
        } else {
          // fl(zero + fl(Q s)): the product rounded on its own (fma, zero addend)
          const f32x2 level = add2(LO, fma2(sub2(t, T23), S, Z));
          acc[m] = (i == 0) ? level : add2(acc[m], level);
        }
      }
    }
  }
#pragma unroll
  for (int m = 0; m < NW / 2; ++m) {
    float a, b;
    unpack2(acc[m], a, b);
    const __nv_bfloat162 x = __floats2bfloat162_rn(a, b);
    h[m] = *reinterpret_cast<const uint32_t*>(&x);
  }
}

// Warps (of 0-7) that form weight tiles: fewer when a CTA forms few rows,
// so that each thread's fixed cost per stage covers more weights.
template <int CS>
__host__ __device__ constexpr int producer_warps() { return CS == 4 ? PF_PRODUCERS_CS4 : PF_PRODUCERS_CS2; }

template <int F, int K, int CS>
__global__ void __launch_bounds__(kPfThreads, 1) prefill_kernel(const __grid_constant__ PrefillBatch p) {
  constexpr int kRows = kPrefillBM / CS;  // rows of the tile this CTA forms for the cluster
  constexpr int kProd = CS == 1 ? kPfDqWarps : producer_warps<CS>();
  constexpr int kNW = kRows * kPrefillBK / (kProd * 32);  // weights a thread forms per stage
  static_assert(kNW == 8 || kNW == 16 || kNW == 32, "weights per producer thread");
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_s = smem_u32(smem_raw);
  const uint32_t base_s = (raw_s + 1023u) & ~1023u;  // swizzled tiles need 1024-byte alignment
  uint8_t* const base = smem_raw + (base_s - raw_s);
  const uint32_t w_s = base_s;                                // weight tiles
  const uint32_t a_s = base_s + kPfWStages * kPfWTileBytes;   // activation tiles
  const uint32_t bar_s = base_s + kPfBarOffset;
  const uint32_t c_s = base_s + kPfCOffset;                  // code tiles
  const uint32_t acc_full = bar_s + 8 * (2 * kPfWStages + 2 * kPfAStages + 2 * kPfCStages);
  const uint32_t drain = acc_full + 8;
  const uint32_t slot_s = bar_s + 8 * kPfBars;  // (after share_done)
  const volatile uint32_t* slot = reinterpret_cast<const volatile uint32_t*>(base + kPfBarOffset + 8 * kPfBars);
  // clusters: sent_in[d] = stages CTA d sent into this CTA's weight ring
  // (written by d's share warp at its end), sent_in[4] = stages this CTA's
  // MMA thread consumed
  volatile uint32_t* const sent_in = reinterpret_cast<volatile uint32_t*>(base + kPfBarOffset + 8 * kPfBars + 16);
  const uint32_t sent_in_s = slot_s + 16;
  auto full_w = [&](int s) { return bar_s + 8 * s; };
  auto empty_w = [&](int s) { return bar_s + 8 * (kPfWStages + s); };
  auto full_a = [&](int s) { return bar_s + 8 * (2 * kPfWStages + s); };
  auto empty_a = [&](int s) { return bar_s + 8 * (2 * kPfWStages + kPfAStages + s); };
  auto full_c = [&](int s) { return bar_s + 8 * (2 * kPfWStages + 2 * kPfAStages + s); };
  auto empty_c = [&](int s) { return bar_s + 8 * (2 * kPfWStages + 2 * kPfAStages + kPfCStages + s); };
  auto share_done = [&](int s) { return drain + 8 + 8 * s; };
  const bool codes_tma = p.codes_tma != 0;

  // warp index and tensor-memory address by broadcast: the compiler then
  // treats the copy and MMA operands derived from them as warp-uniform
  const int warp = __shfl_sync(kFullMask, static_cast<int>(threadIdx.x >> 5), 0);
  const int lane = threadIdx.x & 31;

  // this CTA's tile: clusters in token-tile-major order, rank = token tile
  // within the cluster
  const int64_t tile = blockIdx.x;
  int mi = 0;
  while (mi + 1 < p.count && tile >= p.item[mi + 1].tile_begin) ++mi;
  const PrefillItem& it = p.item[mi];
  const int64_t j = tile - it.tile_begin;
  const int rank = static_cast<int>(j % CS);
  const int64_t cj = j / CS;
  const int64_t row0 = (cj % it.row_tiles) * kPrefillBM;
  const int64_t t0 = ((cj / it.row_tiles) * CS + rank) * kPrefillBN;
  const bool active = t0 < p.tokens;              // (padding CTAs only form weights)
  const bool two = t0 + kPrefillMmaN < p.tokens;  // the second accumulator has tokens
  const int nk = static_cast<int>((it.cols + kPrefillBK - 1) / kPrefillBK);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kPfWStages; ++s) {
      // one CTA: the producer warps; a cluster: one arrival that expects the
      // other CTAs' rows as transaction bytes (this CTA's own rows are ready
      // before it)
      mbar_init(full_w(s), CS == 1 ? kProd : 1);
      mbar_init(empty_w(s), CS);              // every MMA thread of the cluster
      mbar_init(share_done(s), kProd);
    }
    for (int s = 0; s < kPfAStages; ++s) {
      mbar_init(full_a(s), 1);
      mbar_init(empty_a(s), 1);
    }
    for (int s = 0; s < kPfCStages; ++s) {
      mbar_init(full_c(s), 1);
      mbar_init(empty_c(s), kProd);
    }
    mbar_init(acc_full, 1);
    mbar_init(drain, 1);
    for (int d = 0; d < 5; ++d) sent_in[d] = 0u;
    fence_mbarrier_init();
  }
  if (warp == kPfMmaWarp) {
    tmem_alloc(slot_s, kPfTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = __shfl_sync(kFullMask, *slot, 0);
  if constexpr (CS > 1) cluster_sync();  // every CTA's barriers exist before any remote access

  if (warp == kPfTmaWarp) {
    if (lane == 0 && active) {
      bool ok = true;
      int issued = 0;
      for (int kb = 0; kb < nk; ++kb) {
        const int s = kb % kPfAStages;
        if (kb >= kPfAStages && !pf_wait(empty_a(s), ((kb / kPfAStages) - 1) & 1, p.wait_limit_us)) {
          ok = false;
          break;
        }
        const uint32_t dst = a_s + s * kPfATileBytes;
        mbar_arrive_expect_tx(full_a(s), two ? kPfATileBytes : kPfAHalfBytes);
        tma_load_2d(dst, &p.act[mi], kb * kPrefillBK, static_cast<int>(t0), full_a(s));
        if (two)
          tma_load_2d(dst + kPfAHalfBytes, &p.act[mi], kb * kPrefillBK, static_cast<int>(t0 + kPrefillMmaN), full_a(s));
        ++issued;
      }
      if (!ok) {  // let this thread's copies land before the CTA can leave
        atomicOr(p.status, kStatusTimeout);
        for (int kb = issued > kPfAStages ? issued - kPfAStages : 0; kb < issued; ++kb)
          mbar_wait(full_a(kb % kPfAStages), (kb / kPfAStages) & 1, kDrainLimitUs);
      }
    }
    __syncwarp();
  } else if (warp == kPfCodeWarp) {
    if (lane == 0 && codes_tma) {
      bool ok = true;
      int issued = 0;
      for (int kb = 0; kb < nk; ++kb) {
        const int s = kb % kPfCStages;
        if (kb >= kPfCStages && !pf_wait(empty_c(s), ((kb / kPfCStages) - 1) & 1, p.wait_limit_us)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(full_c(s), K * kRows * 16);
#pragma unroll
        for (int i = 0; i < K; ++i)
          tma_load_2d(c_s + s * kPfCStageBytes + i * kPfCTileBytes, &p.codes[mi][i], kb * 16,
                      static_cast<int>(row0 + rank * kRows), full_c(s));
        ++issued;
      }
      if (!ok) {  // let this thread's copies land before the CTA can leave
        atomicOr(p.status, kStatusTimeout);
        for (int kb = issued > kPfCStages ? issued - kPfCStages : 0; kb < issued; ++kb)
          mbar_wait(full_c(kb % kPfCStages), (kb / kPfCStages) & 1, kDrainLimitUs);
      }
    }
    __syncwarp();
  } else if (warp == kPfMmaWarp) {
    if (lane == 0) {
      bool ok = true;
      int consumed = 0;  // weight stages whose full barrier this thread passed
      for (int kb = 0; kb < nk; ++kb) {
        const int sw = kb % kPfWStages, sa = kb % kPfAStages;
        if ((active && !pf_wait(full_a(sa), (kb / kPfAStages) & 1, p.wait_limit_us)) ||
            !pf_wait(full_w(sw), (kb / kPfWStages) & 1, p.wait_limit_us)) {
          ok = false;
          break;
        }
        consumed = kb + 1;
        tc_fence_after();
        if (active) {
          const uint32_t wa = w_s + sw * kPfWTileBytes, aa = a_s + sa * kPfATileBytes;
#pragma unroll
          for (int kk = 0; kk < kPrefillBK / 16; ++kk) {  // K = 16 per MMA: 32 bytes along the swizzle row
            const uint64_t wd = sw128_desc(wa + 32 * kk);
            mma_bf16(tmem, wd, sw128_desc(aa + 32 * kk), kPfIdesc, (kb | kk) != 0);
            if (two)
              mma_bf16(tmem + kPrefillMmaN, wd, sw128_desc(aa + kPfAHalfBytes + 32 * kk), kPfIdesc, (kb | kk) != 0);
          }
        }
        // the weight slot is free in every CTA of the cluster once all their MMAs read it
        if constexpr (CS > 1) mma_commit_multicast(empty_w(sw), static_cast<uint16_t>((1u << CS) - 1u));
        else mma_commit(empty_w(sw));
        if (active) mma_commit(empty_a(sa));
      }
      if constexpr (CS > 1) sent_in[4] = static_cast<uint32_t>(consumed);
      if (ok) {
        if (active) mma_commit(acc_full);
      } else {  // no MMA may be in flight when the tensor memory is freed
        atomicOr(p.status, kStatusTimeout);
        mma_commit(drain);
        mbar_wait(drain, 0, kDrainLimitUs);
      }
    }
    __syncwarp();
  } else if (warp == kPfShareWarp) {
    // clusters: once this CTA's producer warps have written their rows of a
    // stage, send them to the same slot of every other CTA (one bulk copy
    // each, counted there as transaction bytes) and expect the others' rows
    if constexpr (CS > 1) {
      if (lane == 0) {
        constexpr uint32_t kBytes = kRows * 128;  // contiguous rows of the swizzled tile
        uint32_t sent = 0;
        for (int kb = 0; kb < nk; ++kb) {
          const int s = kb % kPfWStages;
          if (!pf_wait(share_done(s), (kb / kPfWStages) & 1, p.wait_limit_us)) {
            atomicOr(p.status, kStatusTimeout);
            break;
          }
          const uint32_t src = w_s + s * kPfWTileBytes + rank * kBytes;
#pragma unroll
          for (int d = 0; d < CS; ++d)
            if (d != rank) bulk_copy_cluster(cluster_addr(src, d), src, kBytes, cluster_addr(full_w(s), d));
          mbar_arrive_expect_tx(full_w(s), (CS - 1) * kBytes);
          sent = static_cast<uint32_t>(kb + 1);
        }
        // every CTA learns how many stages went into it (read after the
        // first of the two final cluster barriers)
#pragma unroll
        for (int d = 0; d < CS; ++d) st_cluster_u32(cluster_addr(sent_in_s + 4 * rank, d), sent);
      }
    }
    __syncwarp();
  } else {  // warps 0-7: weight tiles, then the epilogue
    // thread -> (row of this CTA's share, kNW-column chunk of a stage)
    const int chunk = threadIdx.x / kRows;
    const int rl = threadIdx.x % kRows;
    const int tr = rank * kRows + rl;  // row in the tile
    const int64_t r = row0 + tr;
    bool ok = true;
    const bool producer = warp < kProd;
    const bool blocked = p.scale_blocks != 0;
    constexpr int kSB = groups_per_block<F>();
    ScaleBlock<K> bc, bn;     // scale blocks in use and the next one (in flight)
    int64_t blk_cur = -1, blk_nxt = -1;
    for (int kb = 0; producer && kb < nk; ++kb) {
      const int s = kb % kPfWStages;
      const int64_t c0 = static_cast<int64_t>(kb) * kPrefillBK + kNW * chunk;
      const bool valid = r < it.rows && c0 < it.cols;
      PkgWords<K> cur;
#pragma unroll
      for (int i = 0; i < K; ++i) {
        cur.cw[i] = make_uint2(0u, 0u);
        cur.cb[i] = make_uint4(0u, 0u, 0u, 0u);
        cur.sc[i] = 0.0f;
        cur.zr[i] = 0.0f;
      }
      if (valid) {
        const int64_t e = r * it.cols + c0;
        const int64_t g = e >> p.log2g;
        if (blocked) {  // rows hold whole blocks, so a block never leaves its row
          const int64_t blk = g / kSB;
          if (blk != blk_cur) {
            if (blk == blk_nxt) bc = bn;
            else load_block<F, K>(it, blk, bc);
            blk_cur = blk;
            blk_nxt = -1;
            if (((blk + 1) * kSB << p.log2g) < (r + 1) * it.cols) {  // prefetch the row's next block
              load_block<F, K>(it, blk + 1, bn);
              blk_nxt = blk + 1;
            }
          }
          from_block<F, K>(bc, static_cast<int>(g % kSB), cur);
        } else {
          load_scales<F, K>(it, g, cur);
        }
        if constexpr (F == kAsymBits) {  // 32 weights of width b: b words at word b * (e / 32)
#pragma unroll
          for (int i = 0; i < K; ++i) {
            const int b = p.bits[i];
            const uint32_t* wp = reinterpret_cast<const uint32_t*>(it.codes[i]) + (e >> 5) * b;
            cur.cb[i].x = __ldg(wp);
            if (b > 1) cur.cb[i].y = __ldg(wp + 1);
            if (b > 2) cur.cb[i].z = __ldg(wp + 2);
            if (b > 3) cur.cb[i].w = __ldg(wp + 3);
          }
        } else if (!codes_tma) {  // kNW codes: kNW / 4 bytes (8-aligned for 32, 4 for 16, 2 for 8)
#pragma unroll
          for (int i = 0; i < K; ++i) {
            const uint8_t* cp = it.codes[i] + (e >> 2);
            if constexpr (kNW == 32) cur.cw[i] = __ldg(reinterpret_cast<const uint2*>(cp));
            else if constexpr (kNW == 16) cur.cw[i].x = __ldg(reinterpret_cast<const unsigned int*>(cp));
            else cur.cw[i].x = __ldg(reinterpret_cast<const unsigned short*>(cp));
          }
        }
      }
      if (codes_tma) {  // this stage's codes from the ring; the slot is free once read
        const int sc = kb % kPfCStages;
        const bool got = pf_wait(full_c(sc), (kb / kPfCStages) & 1, p.wait_limit_us);
        if (!__all_sync(kFullMask, got)) {
          ok = false;
          break;
        }
        const uint8_t* ct = base + kPfCOffset + sc * kPfCStageBytes + rl * 16 + chunk * (kNW / 4);
#pragma unroll
        for (int i = 0; i < K; ++i) {
          if constexpr (kNW == 32) cur.cw[i] = *reinterpret_cast<const uint2*>(ct + i * kPfCTileBytes);
          else if constexpr (kNW == 16) cur.cw[i].x = *reinterpret_cast<const uint32_t*>(ct + i * kPfCTileBytes);
          else cur.cw[i].x = *reinterpret_cast<const uint16_t*>(ct + i * kPfCTileBytes);
        }
        // every lane's reads before the next copy (async proxy) into the slot
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(empty_c(sc));
      }
      // the MMAs of this stage's previous round (in every CTA of the
      // cluster) have read its weight tile
      bool ready = true;
      if (kb >= kPfWStages) ready = pf_wait(empty_w(s), ((kb / kPfWStages) - 1) & 1, p.wait_limit_us);
      if (!__all_sync(kFullMask, ready)) {
        ok = false;
        break;
      }
      uint32_t h[kNW / 2];
      if (valid) {
        if constexpr (F == kAsymBits) {
          static_assert(kNW == 32, "per-stage widths take whole 32-weight words");
          f32x2 acc[16];
#pragma unroll
          for (int i = 0; i < K; ++i) {
            switch (p.bits[i]) {
              case 1: dequant_bits<1>(cur.cb[i], cur.sc[i], cur.zr[i], i == 0, acc); break;
              case 3: dequant_bits<3>(cur.cb[i], cur.sc[i], cur.zr[i], i == 0, acc); break;
              case 4: dequant_bits<4>(cur.cb[i], cur.sc[i], cur.zr[i], i == 0, acc); break;
              default: dequant_bits<2>(cur.cb[i], cur.sc[i], cur.zr[i], i == 0, acc); break;
            }
          }
#pragma unroll
          for (int m = 0; m < 16; ++m) {
            float a, b;
            unpack2(acc[m], a, b);
            const __nv_bfloat162 x = __floats2bfloat162_rn(a, b);
            h[m] = *reinterpret_cast<const uint32_t*>(&x);
          }
        } else {
          prefix_weights_bf16<F, K, kNW>(cur, h);
        }
      } else {
#pragma unroll
        for (int m = 0; m < kNW / 2; ++m) h[m] = 0u;
      }
      // K-major, 128-byte swizzle: 16-byte piece c of tile row tr at piece
      // c ^ (tr % 8), in this stage's slot (the share warp copies this CTA's
      // rows to the others)
      uint8_t* const wrow = base + s * kPfWTileBytes + (tr >> 3) * 1024 + (tr & 7) * 128;
#pragma unroll
      for (int q = 0; q < kNW / 8; ++q) {
        const int piece = (chunk * (kNW / 8) + q) ^ (tr & 7);
        *reinterpret_cast<uint4*>(wrow + 16 * piece) = make_uint4(h[4 * q], h[4 * q + 1], h[4 * q + 2], h[4 * q + 3]);
      }
      fence_proxy_async_smem();  // visible to the async proxy (tensor cores, bulk copies)
      __syncwarp();
      if (lane == 0) mbar_arrive(CS == 1 ? full_w(s) : share_done(s));
    }
    if constexpr (CS > 1) {
      // the other CTAs' last commits to this CTA's weight-ring barriers have
      // landed before it can leave
      if (ok && producer) {
        for (int sl = 0; sl < kPfWStages && sl < nk; ++sl) {
          const int last = sl + ((nk - 1 - sl) / kPfWStages) * kPfWStages;
          if (!pf_wait(empty_w(sl), (last / kPfWStages) & 1, p.wait_limit_us)) ok = false;
        }
      }
    }
    bool have = false;
    if (ok && active) have = pf_wait(acc_full, 0, p.wait_limit_us);
    have = __all_sync(kFullMask, have);
    if (!have && (active || !__all_sync(kFullMask, ok)) && lane == 0) atomicOr(p.status, kStatusTimeout);
    tc_fence_after();
    const int quarter = warp & 3;  // TMEM lanes 32 * quarter .. + 31 of this warp
    const int acc_i = warp >> 2;   // accumulator: tokens t0 + 256 * acc_i ..
    if (have && active && (acc_i == 0 || two)) {
      const int64_t row = row0 + 32 * quarter + lane;
#pragma unroll 1
      for (int c = 0; c < kPrefillMmaN / 32; ++c) {
        const int col = acc_i * kPrefillMmaN + 32 * c;
        uint32_t v[32];
        tmem_ld32(tmem + (static_cast<uint32_t>(32 * quarter) << 16) + static_cast<uint32_t>(col), v);
        const int64_t tb = t0 + col;
        if (row < it.rows) {
          float* y = it.Y + tb * it.rows + row;
#pragma unroll
          for (int q = 0; q < 32; ++q)
            if (tb + q < p.tokens) y[q * it.rows] = __uint_as_float(v[q]);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if constexpr (CS > 1) {
    cluster_sync();  // every CTA's sent counts are in place
    // After a timeout, the other CTAs may have sent weight rows into stages
    // this CTA's MMA thread never consumed; their bulk copies complete on
    // this CTA's full barriers.  Settle each such stage's expected bytes to
    // what was actually sent (this CTA's share warp expected every other
    // CTA's rows for the stages it sent itself), then wait (bounded) for
    // the phase, so that no copy lands after this CTA has left.  Pending
    // stages span fewer than kPfWStages (a CTA sends stage kb only after
    // every MMA thread of the cluster consumed kb - kPfWStages), so each
    // slot has at most one open phase.
    if (threadIdx.x == 0 && sent_in[4] < static_cast<uint32_t>(nk)) {
      constexpr uint32_t kBytes = kRows * 128;
      const uint32_t own = sent_in[rank];
      uint32_t most = own;
      for (int d = 0; d < CS; ++d) most = sent_in[d] > most ? sent_in[d] : most;
      for (uint32_t kb = sent_in[4]; kb < most; ++kb) {
        uint32_t m = 0;  // other CTAs that sent stage kb
        for (int d = 0; d < CS; ++d) m += (d != rank && sent_in[d] > kb) ? 1u : 0u;
        const uint32_t bar = full_w(static_cast<int>(kb % kPfWStages));
        if (kb < own) {
          if (m < CS - 1) mbar_complete_tx(bar, (CS - 1 - m) * kBytes);
        } else {
          if (m == 0) continue;  // nothing was sent into this stage
          mbar_arrive_expect_tx(bar, m * kBytes);
        }
        mbar_wait(bar, (kb / kPfWStages) & 1, kDrainLimitUs);
      }
    }
    cluster_sync();  // no CTA leaves while another may still write into it
  }
  if (warp == kPfMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kPfTmemCols);
  }
}

template <int F, int K, int CS>
cudaError_t prefill_launch_kc(const PrefillBatch& p, cudaStream_t stream) {
  // (per launch: the attribute belongs to the current device)
  cudaError_t e =
      cudaFuncSetAttribute(prefill_kernel<F, K, CS>, cudaFuncAttributeMaxDynamicSharedMemorySize, kPfSmemBytes);
  if (e != cudaSuccess) return e;
  if constexpr (CS == 1) {
    prefill_kernel<F, K, 1><<<static_cast<unsigned>(p.total_tiles), kPfThreads, kPfSmemBytes, stream>>>(p);
    return cudaGetLastError();
  } else {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(p.total_tiles), 1, 1);  // a multiple of CS
    cfg.blockDim = dim3(kPfThreads, 1, 1);
    cfg.dynamicSmemBytes = kPfSmemBytes;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CS;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, prefill_kernel<F, K, CS>, p);
  }
}

template <int F, int K>
cudaError_t prefill_launch_k(const PrefillBatch& p, cudaStream_t stream) {
  if constexpr (F == kAsymBits) {  // one CTA per cluster (the host asks for no more)
    return p.cluster == 1 ? prefill_launch_kc<F, K, 1>(p, stream) : cudaErrorInvalidValue;
  } else {
    switch (p.cluster) {
      case 1: return prefill_launch_kc<F, K, 1>(p, stream);
      case 2: return prefill_launch_kc<F, K, 2>(p, stream);
      case 4: return prefill_launch_kc<F, K, 4>(p, stream);
      default: return cudaErrorInvalidValue;
    }
  }
}

template <int F>
cudaError_t prefill_launch_f(int k, const PrefillBatch& p, cudaStream_t stream) {
  switch (k) {
    case 1: return prefill_launch_k<F, 1>(p, stream);
    case 2: return prefill_launch_k<F, 2>(p, stream);
    case 3: return prefill_launch_k<F, 3>(p, stream);
    case 4: return prefill_launch_k<F, 4>(p, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace
}  // namespace rrq
