// RRQ package construction: one fused sm_103a kernel computes every stage of
// Algorithm 1 for a batch of bf16 weight matrices (without a base checkpoint,
// or from a given base stage).
//
// Per stage k (Section 3.1 Eq. 1-3 applied to x for k = 0 and to the running
// residual for k >= 1, Section 3.2 Eq. 4-7), for every group:
//     lo = min v, hi = max v                     (-0 ordered before +0)
//     s  = fl(fl(hi - lo) / 3)                   2-bit grid: 3 steps
//     Q  = s == 0 ? 0 : clamp(rhe(fl(fl(v - lo) / s)), 0, 3)
//     v' = fl(v - fl(lo + fl(Q * s)))            residual, kept in registers
// Codes are packed 4 per byte (element c at bits 2*(c%4) of byte c/4); the
// per-group scale s and zero lo are stored as binary32.
//
// Work decomposition: a warp owns a chunk of 1024 consecutive weights of one
// matrix at a time (2 KiB of bf16), a lane owns 32 consecutive weights, and
// the group/32 consecutive lanes that hold one group reduce with shuffles.
// The chunks of all matrices of a launch form one sequence that the warps of
// a persistent grid take in turn, so small matrices share the machine.  Each
// warp streams its chunks through a private ring of shared-memory buffers
// filled by 1-D bulk copies (TMA) completing on mbarriers.
//
// Scale.  s = RN((hi - lo) / 3) is computed as q = RN(D * RN(1/3)), then one
// fused correction q + RN(D - 3q) * RN(1/3) (Markstein's step); this equals
// the IEEE quotient for every binary32 D (checked exhaustively over all
// significands).
//
// Code.  rhe(fl(d / s)) from a two-float reciprocal r_hi + r_lo = 1/s
// (rcp.approx and a Newton step give r_hi; r_lo = RN(RN(1 - s*r_hi) * r_hi)),
// relative error <= 2^-45.6: q = RN(d*r_hi + RN(d*r_lo)) (one multiply, one
// fma) where the value before the last rounding is within x * 2^-45.3 of
// x = d/s.  rhe(fl(x)) changes only where x crosses B1 = 0.5 + 2^-25,
// B2 = 1.5 - 2^-24 or B3 = 2.5 + 2^-23 (the binary32 rounding boundaries next
// to the ties 0.5, 1.5, 2.5), and rhe(RN(y)) changes at the same points, so
// rhe(q) equals rhe(fl(d/s)) unless some float d lies within that error of
// B_q * s.  In units of the last bit of B_q * s (an exact product of a 24-bit
// and a 25/26-bit integer) the error is below 10 units.  How close a float can
// come to B_q * s depends only on the significand m of s: within 64 units only
// for m < 2^23 + 64, |m - 3*2^22| < 64 or m > 2^24 - 64 (about 1 scale in
// 30,000).  Those groups, and scales outside [2^-90, 2^90], take the
// per-element IEEE-division path.  Results are bit-identical to the definition
// above in every case.
//
// Rounding to an integer uses t = RN(q + 2^23) = 2^23 + rhe(q) (the code is
// the low bits of t), and the dequantized step fl(Q*s) is one fused
// multiply-add fma(t, s, -2^23*s) with a single rounding.  (Separate packed
// multiply and add instructions are not used for it: the compiler fuses them
// into one fma even with -fmad=false.)
//
// Symmetric grid (the paper's "symmetric" configuration, Table 4 and
// Appendix G; implicit zero-point 2, no zero stored):
//     amax = max |v|,  s = fl(fl(2 amax) / 3)  [binary16-rounded if stored so]
//     Q  = s == 0 ? 2 : clamp(rhe(fl(v / s)) + 2, 0, 3)
//     v' = fl(v - (Q - 2) s)                   (Q - 2) s is exact
// The code uses the same two-float quotient q ~ v/s; min(q, 1) applies the
// upper clamp (rhe(x) >= 1 already means Q = 3; |x| <= 2.25 keeps the lower
// end at Q >= 0), t = RN(min(q, 1) + C) with C = 1.5 * 2^23 + 2 gives
// C + rhe (C is even), whose low two bits are Q, and u = t - C = Q - 2 exactly;
// the residual is one fma(u, -s, v) = RN(v - (Q - 2) s).  The boundaries that
// matter are +-B1 and -B2 (the same magnitudes as above), so binary32 scales
// use the same significand test.  A binary16 scale has at most 11 significant
// bits: then B_q * s has more than 24 significant bits with an odd top part,
// no float d equals it, and the distance from any float to it is at least one
// unit of 2^(exponent(s) - 48 + 13), far above the quotient's error -- every
// binary16 scale takes the fast path.
//
// Algorithm 1 with a base checkpoint (kBase): stage 0 of the package is given.
// Each lane loads its 8-byte base code word, base scale (and zero) one chunk
// ahead, dequantizes stage 0 in registers with the grid's level formula,
// starts the running residual at fl(x - L_0) and computes stages 1.. only.
//
// Heterogeneous stage widths (kAsymBits): stage k has b_k in 1..4 bits, 2^b - 1
// steps.  The band test above covers the 2-bit boundaries only; for any
// width the kernel instead checks each element: with q the two-float
// quotient, if q is farther than 2^-17 from every half-integer (while
// ulp(q) <= 2^-20 for q < 16 and |q - x| < 2^-40), x, RN(x) and q round to the
// same integer and the fast code is exact; the few elements within the margin
// (and groups with a scale outside [2^-90, 2^90]) take the IEEE-division
// path.  Codes are packed least significant bit first, element c at bits
// b*c.., so a lane's 32 weights fill b words; for this format the lane reads
// its shared-memory pieces in natural order.
//
// Build with prefixes (kModeEmit): the stage levels the build computes are
// exactly the values the reconstruction sums (fl(lo + fl(Q s)), or (Q-2) s),
// so the kernel also keeps the binary32 prefix sums acc = L_0,
// acc = fl(acc + L_k) in registers and writes the bf16 reconstruction after
// every stage -- the package and its 2/4/6/8-bit weights in one pass over W,
// bit-identical to rrq_reconstruct on the package.
//
// This header holds the kernel template; quantize.cu instantiates the build
// without a base checkpoint, quantize_base.cu the build from one,
// quantize_emit.cu the build that also writes every prefix.
#pragma once

#include <atomic>

#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "rrq_device.cuh"

namespace rrq {
namespace {

#ifndef RRQ_QUANTIZE_CTAS_PER_SM
#define RRQ_QUANTIZE_CTAS_PER_SM 3
#endif
#ifndef RRQ_QUANTIZE_RING
#define RRQ_QUANTIZE_RING 4
#endif
constexpr int kWarps = 8;                  // warps per CTA
constexpr int kThreads = kWarps * 32;
constexpr int kRing = RRQ_QUANTIZE_RING;   // bulk-copy buffers per warp
constexpr int kSmemBytes = kWarps * kRing * kChunkBytes + kWarps * kRing * 8;
// plus, when the prefixes are written, two 2 KiB output staging buffers per warp
template <int M>
__host__ __device__ constexpr int smem_bytes();
constexpr float kTwo23 = 8388608.0f;       // RN(x + 2^23) = 2^23 + rhe(x) for 0 <= x < 2^22
constexpr float kThird = 0x1.555556p-2f;   // RN(1/3)
constexpr float kSymRound = 12582914.0f;   // 1.5 * 2^23 + 2: RN(x + C) = C + rhe(x), low bits 2 + rhe(x)

// RN(D / 3) for finite D >= 0 (exhaustively equal to IEEE division).
__device__ __forceinline__ float div3(float D) {
  const float q = __fmul_rn(D, kThird);
  const float e = __fmaf_rn(-q, 3.0f, D);
  return __fmaf_rn(e, kThird, q);
}

// 1/s as r_hi + r_lo with relative error below 2^-45.6 (s in [2^-90, 2^90]):
// r_hi from rcp.approx and one Newton step (relative error ~2^-23),
// r_lo = RN(1 - s*r_hi) * r_hi carries the rest.
__device__ __forceinline__ void recip2(float s, float& r_hi, float& r_lo) {
  float r0;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r0) : "f"(s));
  const float e0 = __fmaf_rn(-s, r0, 1.0f);
  r_hi = __fmaf_rn(r0, e0, r0);
  const float e1 = __fmaf_rn(-s, r_hi, 1.0f);
  r_lo = __fmul_rn(e1, r_hi);
}

// Per-element IEEE-division path: code and residual of one value.
__device__ __forceinline__ int exact_code(float v, float lo, float s) {
  if (s == 0.0f) return 0;
  const float d = __fsub_rn(v, lo);
  const float u = __fdiv_rn(d, s);
  int q = __float2int_rn(u);  // round half to even
  q = q < 0 ? 0 : q;
  return q > 3 ? 3 : q;
}
struct ExactPair {
  f32x2 w;         // residuals
  f32x2 l;         // stage levels
  uint32_t q0, q1;
};

// What a launch computes.
enum Mode : int {
  kModeBuild = 0,  // every stage from W (Algorithm 1, no base checkpoint)
  kModeBase = 1,   // stage 0 given, stages 1.. from R_0 = W - W_0
  kModeEmit = 2,   // every stage from W, plus the bf16 reconstruction after every stage
};
__device__ __noinline__ ExactPair exact_pair(f32x2 v, float lo, float s) {
  float a, b;
  unpack2(v, a, b);
  const int qa = exact_code(a, lo, s), qb = exact_code(b, lo, s);
  const float la = __fadd_rn(lo, __fmul_rn(__int2float_rn(qa), s));
  const float lb = __fadd_rn(lo, __fmul_rn(__int2float_rn(qb), s));
  return {pack2(__fsub_rn(a, la), __fsub_rn(b, lb)), pack2(la, lb), static_cast<uint32_t>(qa),
          static_cast<uint32_t>(qb)};
}

// Symmetric grid, per-element IEEE-division path.
__device__ __forceinline__ int exact_code_sym(float v, float s) {
  if (s == 0.0f) return 2;
  int q = __float2int_rn(__fdiv_rn(v, s)) + 2;  // round half to even, zero-point 2
  q = q < 0 ? 0 : q;
  return q > 3 ? 3 : q;
}
__device__ __noinline__ ExactPair exact_pair_sym(f32x2 v, float s) {
  float a, b;
  unpack2(v, a, b);
  const int qa = exact_code_sym(a, s), qb = exact_code_sym(b, s);
  const float la = __fmul_rn(__int2float_rn(qa - 2), s), lb = __fmul_rn(__int2float_rn(qb - 2), s);
  return {pack2(__fsub_rn(a, la), __fsub_rn(b, lb)), pack2(la, lb), static_cast<uint32_t>(qa),
          static_cast<uint32_t>(qb)};
}

// Scales for which the corrected quotient is proven exact (see the file
// comment): significand away from the three near-boundary bands, exponent in
// [2^-90, 2^90].
__device__ __forceinline__ bool corrected_quotient_safe(float s) {
  const uint32_t bits = __float_as_uint(s);
  const uint32_t e = bits >> 23;  // s > 0: no sign bit
  // exponent field in [127-90, 127+89]
  const bool range_ok = (e - (127u - 90u)) < 180u;
  // significand field f = m - 2^23 within 64 of 0, 2^22 or 2^23 (mod 2^22)
  const bool band = (((bits & 0x7fffffu) + 64u) & 0x3fffffu) < 128u;
  return range_ok && !band;
}

// Appends the 2-bit code in the low bits of t to acc from the top: after
// eight calls the codes of elements 0..7 sit at bits 16..31, element 0 lowest.
__device__ __forceinline__ uint32_t push_code(uint32_t acc, uint32_t t) {
  return __funnelshift_r(acc, t, 2);
}

// b-bit stages: the per-element IEEE-division path for m = 2^b - 1 steps.
__device__ __noinline__ ExactPair exact_pair_bits(f32x2 v, float lo, float s, int m) {
  float a, b;
  unpack2(v, a, b);
  int qa = 0, qb = 0;
  if (s != 0.0f) {
    qa = __float2int_rn(__fdiv_rn(__fsub_rn(a, lo), s));  // round half to even
    qb = __float2int_rn(__fdiv_rn(__fsub_rn(b, lo), s));
    qa = qa < 0 ? 0 : (qa > m ? m : qa);
    qb = qb < 0 ? 0 : (qb > m ? m : qb);
  }
  const float la = __fadd_rn(lo, __fmul_rn(__int2float_rn(qa), s));
  const float lb = __fadd_rn(lo, __fmul_rn(__int2float_rn(qb), s));
  return {pack2(__fsub_rn(a, la), __fsub_rn(b, lb)), pack2(la, lb), static_cast<uint32_t>(qa),
          static_cast<uint32_t>(qb)};
}

constexpr float kTieMargin = 0.5f - 0x1p-17f;  // |q - rhe(q)| beyond this: near a half-integer

// One b-bit stage of a lane's 32 values (natural order): codes into words
// (element j at bits B*j), residuals in place, min/max of the new residuals.
template <int B>
__device__ __forceinline__ void stage_bits(f32x2 (&v)[16], float lo, float s, bool fast,
                                           uint32_t (&words)[4], float& mn, float& mx) {
  constexpr int M = (1 << B) - 1;
  constexpr uint32_t kMask = static_cast<uint32_t>(M);
#pragma unroll
  for (int w = 0; w < 4; ++w) words[w] = 0u;
  float mn0 = __int_as_float(0x7f800000), mn1 = mn0, mx0 = -mn0, mx1 = mx0;
  auto place = [&](int j, uint32_t code) {  // element j's code at bits B*j
    const int bit = B * j, w = bit >> 5, sh = bit & 31;
    words[w] |= code << sh;
    if (sh + B > 32) words[w + 1] |= code >> (32 - sh);
  };
  float r_hi = 0.0f, r_lo = 0.0f;
  if (fast && s > 0.0f) recip2(s, r_hi, r_lo);
  const float c = __fmul_rn(-kTwo23, s);
  const f32x2 LO = pack2(lo, lo), RH = pack2(r_hi, r_hi), RL = pack2(r_lo, r_lo), S = pack2(s, s);
  const f32x2 T23 = pack2(kTwo23, kTwo23), C = pack2(c, c);
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    uint32_t ca, cb;
    bool exact = !fast;
    f32x2 t = T23;
    if (fast) {
      const f32x2 d = sub2(v[i], LO);
      const f32x2 q = fma2(d, RH, mul2(d, RL));  // d/s to 2^-45.3
      t = add2(q, T23);                          // 2^23 + rhe(q)
      float fa, fb;
      unpack2(sub2(q, sub2(t, T23)), fa, fb);    // q - rhe(q), exact
      exact = fabsf(fa) > kTieMargin || fabsf(fb) > kTieMargin;
    }
    if (exact) {
      const ExactPair x = exact_pair_bits(v[i], lo, s, M);
      v[i] = x.w;
      ca = x.q0;
      cb = x.q1;
    } else {
      v[i] = sub2(v[i], add2(LO, fma2(t, S, C)));  // v - fl(lo + fl(Q s))
      ca = static_cast<uint32_t>(t) & kMask;
      cb = static_cast<uint32_t>(t >> 32) & kMask;
    }
    place(2 * i, ca);
    place(2 * i + 1, cb);
    float a, b;
    unpack2(v[i], a, b);
    if (i & 1) {
      mn1 = min3(mn1, a, b);
      mx1 = max3(mx1, a, b);
    } else {
      mn0 = min3(mn0, a, b);
      mx0 = max3(mx0, a, b);
    }
  }
  mn = fminf(mn0, mn1);
  mx = fmaxf(mx0, mx1);
}

template <int B>
__device__ __forceinline__ void store_words(uint8_t* codes, int64_t e0, const uint32_t (&w)[4]) {
  uint8_t* dst = codes + (e0 >> 5) * (4 * B);  // 4B bytes per 32 weights
  if (B == 4) {
    __stcs(reinterpret_cast<uint4*>(dst), make_uint4(w[0], w[1], w[2], w[3]));
  } else if (B == 2) {
    __stcs(reinterpret_cast<uint2*>(dst), make_uint2(w[0], w[1]));
  } else {
#pragma unroll
    for (int j = 0; j < B; ++j) __stcs(reinterpret_cast<unsigned int*>(dst) + j, w[j]);
  }
}

// Asymmetric grid with per-stage widths (values in natural order).  kBase:
// stage 0 is given (Algorithm 1 with a base checkpoint): the lane reads its
// bits[0] code words and the group's scale and zero, and the stages start
// from R_0 = fl(x - fl(zero + fl(Q s))).
template <int G, bool kBase>
__device__ __forceinline__ void quantize_chunk_bits(const QuantizeBatch& p, const QuantizeItem& it,
                                                    int64_t e0, int lane, uint4 (&raw)[4]) {
  constexpr int L = G / 32;  // lanes per group
  const bool valid = e0 < it.n;
  if (!valid) {
#pragma unroll
    for (int j = 0; j < 4; ++j) raw[j] = make_uint4(0u, 0u, 0u, 0u);
  }
  f32x2 v[16];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const uint32_t w4[4] = {raw[j].x, raw[j].y, raw[j].z, raw[j].w};
#pragma unroll
    for (int m = 0; m < 4; ++m) v[4 * j + m] = pack2u(w4[m] << 16, w4[m] & 0xffff0000u);
  }
  if constexpr (kBase) {
    if (valid) {
      const int b0 = p.bits[0];
      const uint32_t* wp = reinterpret_cast<const uint32_t*>(it.codes[0]) + (e0 >> 5) * b0;
      uint4 w = make_uint4(__ldg(wp), 0u, 0u, 0u);
      if (b0 > 1) w.y = __ldg(wp + 1);
      if (b0 > 2) w.z = __ldg(wp + 2);
      if (b0 > 3) w.w = __ldg(wp + 3);
      const float s0 = __ldg(static_cast<const float*>(it.scales[0]) + e0 / G);
      const float z0 = __ldg(it.zeros[0] + e0 / G);
      f32x2 l0[16];  // the base levels fl(zero + fl(Q s))
      switch (b0) {
        case 1: dequant_bits<1>(w, s0, z0, true, l0); break;
        case 3: dequant_bits<3>(w, s0, z0, true, l0); break;
        case 4: dequant_bits<4>(w, s0, z0, true, l0); break;
        default: dequant_bits<2>(w, s0, z0, true, l0); break;
      }
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] = sub2(v[i], l0[i]);  // R_0 = W - W_0
    }
  }
  float lo, hi;
  lane_minmax(v, lo, hi);
  group_minmax<L>(lo, hi);

#pragma unroll 1
  for (int k = kBase ? 1 : 0; k < p.n_stages; ++k) {
    if (__any_sync(kFullMask, lo == 0.0f)) {  // a zero minimum is -0 if the group holds a -0
      uint32_t neg = 0;
      if (lo == 0.0f) {
#pragma unroll
        for (int i = 0; i < 16; ++i)
          neg |= (static_cast<uint32_t>(v[i]) == 0x80000000u) |
                 (static_cast<uint32_t>(v[i] >> 32) == 0x80000000u);
      }
      neg = group_or<L>(neg);
      if (lo == 0.0f) lo = neg ? -0.0f : 0.0f;
    }
    const int b = p.bits[k];
    const float range = __fsub_rn(hi, lo);
    const float s = b == 2 ? div3(range) : b == 1 ? range : __fdiv_rn(range, static_cast<float>((1 << b) - 1));
    const uint32_t e = __float_as_uint(s) >> 23;
    const bool fast = !(p.flags & kDebugForceExact) && (s == 0.0f || (e - (127u - 90u)) < 180u);
    uint32_t words[4];
    float mn, mx;
    switch (b) {
      case 1: stage_bits<1>(v, lo, s, fast, words, mn, mx); break;
      case 3: stage_bits<3>(v, lo, s, fast, words, mn, mx); break;
      case 4: stage_bits<4>(v, lo, s, fast, words, mn, mx); break;
      default: stage_bits<2>(v, lo, s, fast, words, mn, mx); break;
    }
    if (valid) {
      switch (b) {
        case 1: store_words<1>(it.codes[k], e0, words); break;
        case 3: store_words<3>(it.codes[k], e0, words); break;
        case 4: store_words<4>(it.codes[k], e0, words); break;
        default: store_words<2>(it.codes[k], e0, words); break;
      }
      if ((lane & (L - 1)) == 0) {
        __stcs(static_cast<float*>(it.scales[k]) + e0 / G, s);
        __stcs(it.zeros[k] + e0 / G, lo);
      }
    }
    if (k + 1 < p.n_stages) {
      lo = mn;
      hi = mx;
      group_minmax<L>(lo, hi);
    }
  }
}

// Stores the packed codes of stage k of this lane's 32 weights: acc[m] holds
// the codes of slots 4m..4m+3 in its high half, in slot order.
__device__ __forceinline__ void store_codes(uint8_t* codes, int64_t e0, const uint32_t (&acc)[4],
                                            uint32_t sel_lo, uint32_t sel_hi) {
  const uint32_t c0 = __byte_perm(acc[0], acc[1], 0x7632);
  const uint32_t c1 = __byte_perm(acc[2], acc[3], 0x7632);
  const uint2 out = make_uint2(__byte_perm(c0, c1, sel_lo), __byte_perm(c0, c1, sel_hi));
  __stcs(reinterpret_cast<uint2*>(codes + (e0 >> 2)), out);
}

// A lane's stage-0 words of a given base checkpoint: its 32 codes (8 bytes),
// its group's scale and zero.
struct BaseWords {
  uint2 code;
  float scale;
  float zero;
};

template <int G, int F>
__device__ __forceinline__ BaseWords load_base(const QuantizeItem& it, int64_t e0) {
  BaseWords b{make_uint2(0u, 0u), 0.0f, 0.0f};
  if (e0 < it.n) {
    b.code = __ldg(reinterpret_cast<const uint2*>(it.codes[0] + (e0 >> 2)));
    if (F == kSymF16)
      b.scale = __half2float(__ldg(static_cast<const __half*>(it.scales[0]) + e0 / G));
    else
      b.scale = __ldg(static_cast<const float*>(it.scales[0]) + e0 / G);
    if (F == kAsymF32) b.zero = __ldg(it.zeros[0] + e0 / G);
  }
  return b;
}

// v <- fl(v - L_0) for the given base stage.  The code word is rotated so
// that slot j's 8 codes sit at bits 16j (the lane reads its pieces rotated).
template <int F>
__device__ __forceinline__ void subtract_base(f32x2 (&v)[16], const BaseWords& b, uint32_t ld_lo,
                                              uint32_t ld_hi) {
  const uint32_t w0 = __byte_perm(b.code.x, b.code.y, ld_lo);
  const uint32_t w1 = __byte_perm(b.code.x, b.code.y, ld_hi);
  const float s = b.scale;
  if (F == kAsymF32) {
    // fl(Q s) = fma(2^23 + Q, s, -2^23 s) when 2^23 s is exact, else
    // fma(t - 2^23, s, 0); then fl(zero + fl(Q s)) and fl(v - L_0)
    const bool scaled_ok = s == 0.0f || (fabsf(s) >= 0x1p-100f && fabsf(s) <= 0x1p+100f);
    const f32x2 S = pack2(s, s), Z = pack2(b.zero, b.zero), T23 = pack2(kTwo23, kTwo23);
    const float c = __fmul_rn(-kTwo23, s);
    const f32x2 C = pack2(c, c), Z0 = pack2(0.0f, 0.0f);
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const uint32_t word = i < 8 ? w0 : w1;
      const int sh = 4 * (i & 7);
      const f32x2 t = pack2u(magic23<3u>(word >> sh), magic23<3u>(word >> (sh + 2)));
      const f32x2 qs = scaled_ok ? fma2(t, S, C) : fma2(sub2(t, T23), S, Z0);
      v[i] = sub2(v[i], add2(Z, qs));
    }
  } else {
    // (Q - 2) s is exact: fl(v - (Q-2) s) is one fma
    const f32x2 NS = pack2(-s, -s), K2 = pack2(kTwo23 + 2.0f, kTwo23 + 2.0f);
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const uint32_t word = i < 8 ? w0 : w1;
      const int sh = 4 * (i & 7);
      const f32x2 t = pack2u(magic23<3u>(word >> sh), magic23<3u>(word >> (sh + 2)));
      v[i] = fma2(sub2(t, K2), NS, v[i]);
    }
  }
}

// Output staging of the build with prefixes: two 2 KiB buffers per warp used
// in turn; every lane writes its 32 bf16 values (slot j -> piece (j + rot) & 3,
// conflict-free), lane 0 writes the chunk out with one bulk copy.
struct Emitter {
  uint8_t* stage;   // this warp's two buffers
  uint32_t n_store; // stores issued so far
};

// bf16 of the prefix sums of this lane's 32 weights to out[c0 ..] (warp-wide:
// every lane calls it, also lanes past the end of the matrix).
__device__ __forceinline__ void emit_prefix(Emitter& em, uint16_t* out, int64_t c0, int64_t n,
                                            const f32x2 (&w)[16], int lane, int rot) {
  uint32_t h[16];
#pragma unroll
  for (int m = 0; m < 16; ++m) {
    float a, b;
    unpack2(w[m], a, b);
    const __nv_bfloat162 x = __floats2bfloat162_rn(a, b);
    h[m] = *reinterpret_cast<const uint32_t*>(&x);
  }
  uint8_t* buf = em.stage + (em.n_store & 1) * kChunkBytes;
  ++em.n_store;
  if (lane == 0) bulk_wait_read<1>();  // the copy that last used this buffer has read it
  __syncwarp();
  uint4* dst = reinterpret_cast<uint4*>(buf + lane * 64);
#pragma unroll
  for (int j = 0; j < 4; ++j) dst[(j + rot) & 3] = make_uint4(h[4 * j], h[4 * j + 1], h[4 * j + 2], h[4 * j + 3]);
  fence_proxy_async_smem();
  __syncwarp();
  if (lane == 0) {
    const int64_t left = n - c0;
    bulk_store(out + c0, smem_u32(buf), static_cast<uint32_t>((left < kChunkElems ? left : kChunkElems) * 2));
    bulk_commit();
  }
}

template <int G, int M>
__device__ __forceinline__ void quantize_chunk_asym(const QuantizeBatch& p, const QuantizeItem& it,
                                                    int64_t e0, int lane, uint4 (&raw)[4],
                                                    uint32_t sel_lo, uint32_t sel_hi, const BaseWords& bw,
                                                    uint32_t ld_lo, uint32_t ld_hi, int rot, Emitter& em) {
  constexpr bool kBase = M == kModeBase;
  constexpr bool kEmit = M == kModeEmit;
  constexpr int L = G / 32;  // lanes per group
  const bool valid = e0 < it.n;
  // prefix sums (kModeEmit), starting at -0: fl(-0 + x) = x for every x,
  // including both zeros, so the first stage needs no special case
  f32x2 wsum[kEmit ? 16 : 1];
#pragma unroll
  for (int i = 0; i < (kEmit ? 16 : 1); ++i) wsum[i] = pack2(-0.0f, -0.0f);
  if (!valid) {
#pragma unroll
    for (int j = 0; j < 4; ++j) raw[j] = make_uint4(0u, 0u, 0u, 0u);
  }

  // bf16 -> binary32 (exact), pairs of consecutive weights, slot order
  f32x2 v[16];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const uint32_t w4[4] = {raw[j].x, raw[j].y, raw[j].z, raw[j].w};
#pragma unroll
    for (int m = 0; m < 4; ++m) v[4 * j + m] = pack2u(w4[m] << 16, w4[m] & 0xffff0000u);
  }
  if constexpr (kBase) subtract_base<kAsymF32>(v, bw, ld_lo, ld_hi);  // R_0 = W - W_0

  float lo, hi;
  lane_minmax(v, lo, hi);
  group_minmax<L>(lo, hi);

  // A stage's codes, scale, offset and prefix are written in the next stage's
  // prologue (the last stage's after the loop): independent stores that fill
  // the latency of the next range, scale and reciprocal.
  uint32_t acc[4] = {0u, 0u, 0u, 0u};
  float s_out = 0.0f, lo_out = 0.0f;
  auto write_stage = [&](int k) {
    if (valid) {
      store_codes(it.codes[k], e0, acc, sel_lo, sel_hi);
      if ((lane & (L - 1)) == 0) {
        __stcs(static_cast<float*>(it.scales[k]) + e0 / G, s_out);
        __stcs(it.zeros[k] + e0 / G, lo_out);
      }
    }
    if constexpr (kEmit) emit_prefix(em, it.out[k], e0 - lane * kLaneElems, it.n, wsum, lane, rot);
  };
  const int k0 = kBase ? 1 : 0;
#pragma unroll 1
  for (int k = k0; k < p.n_stages; ++k) {
    // A zero minimum: the stored offset is -0 if the group holds a -0.
    if (__any_sync(kFullMask, lo == 0.0f)) {
      uint32_t neg = 0;
      if (lo == 0.0f) {
#pragma unroll
        for (int i = 0; i < 16; ++i)
          neg |= (static_cast<uint32_t>(v[i]) == 0x80000000u) |
                 (static_cast<uint32_t>(v[i] >> 32) == 0x80000000u);
      }
      neg = group_or<L>(neg);
      if (lo == 0.0f) lo = neg ? -0.0f : 0.0f;
    }

    const float s = div3(__fsub_rn(hi, lo));
    const bool fast = !(p.flags & kDebugForceExact) && (s == 0.0f || corrected_quotient_safe(s));
    float r_hi, r_lo;
    recip2(s, r_hi, r_lo);
    if (!(s > 0.0f)) r_hi = r_lo = 0.0f;  // s = 0: every quotient 0
    if (k > k0) write_stage(k - 1);
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[j] = 0u;
    // min/max of the new residual (next stage's range), gathered in the loop
    float mn0 = __int_as_float(0x7f800000), mn1 = mn0, mx0 = -mn0, mx1 = mx0;
    if (fast) {
      const float c = __fmul_rn(-kTwo23, s);  // exact: power-of-two scaling
      const f32x2 LO = pack2(lo, lo), RH = pack2(r_hi, r_hi), RL = pack2(r_lo, r_lo), S = pack2(s, s);
      const f32x2 T23 = pack2(kTwo23, kTwo23), C = pack2(c, c);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const f32x2 d = sub2(v[i], LO);
        const f32x2 q = fma2(d, RH, mul2(d, RL));  // d/s to 2^-45.3
        const f32x2 t = add2(q, T23);              // 2^23 + rhe(q)
        const f32x2 step = fma2(t, S, C);    // fl(Q*s)
        const f32x2 lv = add2(LO, step);     // fl(lo + fl(Q*s))
        v[i] = sub2(v[i], lv);               // v - fl(lo + fl(Q*s))
        if constexpr (kEmit) wsum[i] = add2(wsum[i], lv);
        acc[i >> 2] = push_code(push_code(acc[i >> 2], static_cast<uint32_t>(t)),
                                static_cast<uint32_t>(t >> 32));
        float a, b;
        unpack2(v[i], a, b);
        if (i & 1) {
          mn1 = min3(mn1, a, b);
          mx1 = max3(mx1, a, b);
        } else {
          mn0 = min3(mn0, a, b);
          mx0 = max3(mx0, a, b);
        }
      }
    } else {  // this group: IEEE division element by element
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const ExactPair x = exact_pair(v[i], lo, s);
        v[i] = x.w;
        if constexpr (kEmit) wsum[i] = add2(wsum[i], x.l);
        acc[i >> 2] = push_code(push_code(acc[i >> 2], x.q0), x.q1);
      }
      lane_minmax(v, mn0, mx0);
    }
    s_out = s;
    lo_out = lo;
    if (k + 1 < p.n_stages) {  // range of the residual = next stage's lo, hi
      lo = fminf(mn0, mn1);
      hi = fmaxf(mx0, mx1);
      group_minmax<L>(lo, hi);
    }
  }
  if (p.n_stages > k0) write_stage(p.n_stages - 1);
}

// Symmetric grid; kF16: the scale is rounded to binary16, stored as such, and
// the stage quantizes against the rounded value.
template <int G, bool kF16, int M>
__device__ __forceinline__ void quantize_chunk_sym(const QuantizeBatch& p, const QuantizeItem& it,
                                                   int64_t e0, int lane, uint4 (&raw)[4],
                                                   uint32_t sel_lo, uint32_t sel_hi, const BaseWords& bw,
                                                   uint32_t ld_lo, uint32_t ld_hi, int rot, Emitter& em) {
  constexpr bool kBase = M == kModeBase;
  constexpr bool kEmit = M == kModeEmit;
  constexpr int L = G / 32;  // lanes per group
  const bool valid = e0 < it.n;
  // prefix sums (kModeEmit), starting at -0: fl(-0 + x) = x for every x,
  // including both zeros, so the first stage needs no special case
  f32x2 wsum[kEmit ? 16 : 1];
#pragma unroll
  for (int i = 0; i < (kEmit ? 16 : 1); ++i) wsum[i] = pack2(-0.0f, -0.0f);
  if (!valid) {
#pragma unroll
    for (int j = 0; j < 4; ++j) raw[j] = make_uint4(0u, 0u, 0u, 0u);
  }
  f32x2 v[16];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const uint32_t w4[4] = {raw[j].x, raw[j].y, raw[j].z, raw[j].w};
#pragma unroll
    for (int m = 0; m < 4; ++m) v[4 * j + m] = pack2u(w4[m] << 16, w4[m] & 0xffff0000u);
  }
  if constexpr (kBase) subtract_base<kSymF32>(v, bw, ld_lo, ld_hi);  // R_0 = W - W_0
  float amax = group_max<L>(lane_amax(v));

  // A stage's codes, scale and prefix are written in the next stage's
  // prologue (the last stage's after the loop), filling its latency.
  uint32_t acc[4] = {0u, 0u, 0u, 0u};
  float s_out = 0.0f;
  uint16_t s16_out = 0;
  auto write_stage = [&](int k) {
    if (valid) {
      store_codes(it.codes[k], e0, acc, sel_lo, sel_hi);
      if ((lane & (L - 1)) == 0) {
        if (kF16) stcs_u16(static_cast<uint16_t*>(it.scales[k]) + e0 / G, s16_out);
        else __stcs(static_cast<float*>(it.scales[k]) + e0 / G, s_out);
      }
    }
    if constexpr (kEmit) emit_prefix(em, it.out[k], e0 - lane * kLaneElems, it.n, wsum, lane, rot);
  };
  const int k0 = kBase ? 1 : 0;
#pragma unroll 1
  for (int k = k0; k < p.n_stages; ++k) {
    float s = div3(__fmul_rn(amax, 2.0f));  // 2 * amax is exact
    uint16_t s16 = 0;
    if (kF16) {
      s16 = __half_as_ushort(__float2half_rn(s));
      s = __half2float(__ushort_as_half(s16));
    }
    const bool fast = !(p.flags & kDebugForceExact) && (kF16 || s == 0.0f || corrected_quotient_safe(s));
    float r_hi, r_lo;
    recip2(s, r_hi, r_lo);
    if (!(s > 0.0f)) r_hi = r_lo = 0.0f;  // s = 0: every quotient 0
    if (k > k0) write_stage(k - 1);
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[j] = 0u;
    float mx0 = 0.0f, mx1 = 0.0f;  // max |new residual|, gathered in the loop
    if (fast) {
      const f32x2 RH = pack2(r_hi, r_hi), RL = pack2(r_lo, r_lo), NS = pack2(-s, -s), S = pack2(s, s);
      const f32x2 C = pack2(kSymRound, kSymRound);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const f32x2 q = fma2(v[i], RH, mul2(v[i], RL));  // v/s to 2^-45.3
        float qa, qb;
        unpack2(q, qa, qb);
        const f32x2 t = add2(pack2(fminf(qa, 1.0f), fminf(qb, 1.0f)), C);  // C + rhe, clamped
        const f32x2 u = sub2(t, C);                                       // Q - 2, exact
        v[i] = fma2(u, NS, v[i]);                                         // v - (Q-2) s
        if constexpr (kEmit) wsum[i] = fma2(u, S, wsum[i]);  // + (Q-2) s, exact product
        acc[i >> 2] = push_code(push_code(acc[i >> 2], static_cast<uint32_t>(t)),
                                static_cast<uint32_t>(t >> 32));
        float a, b;
        unpack2(v[i], a, b);
        if (i & 1) mx1 = max3(mx1, fabsf(a), fabsf(b));
        else mx0 = max3(mx0, fabsf(a), fabsf(b));
      }
    } else {  // this group: IEEE division element by element
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const ExactPair x = exact_pair_sym(v[i], s);
        v[i] = x.w;
        if constexpr (kEmit) wsum[i] = add2(wsum[i], x.l);
        acc[i >> 2] = push_code(push_code(acc[i >> 2], x.q0), x.q1);
      }
      mx0 = lane_amax(v);
    }
    s_out = s;
    s16_out = s16;
    if (k + 1 < p.n_stages) amax = group_max<L>(fmaxf(mx0, mx1));
  }
  if (p.n_stages > k0) write_stage(p.n_stages - 1);
}

template <int G, int F, int M>
__device__ __forceinline__ void quantize_chunk(const QuantizeBatch& p, const QuantizeItem& it,
                                               int64_t e0, int lane, uint4 (&raw)[4],
                                               uint32_t sel_lo, uint32_t sel_hi, const BaseWords& bw,
                                               uint32_t ld_lo, uint32_t ld_hi, int rot, Emitter& em) {
  if constexpr (F == kAsymF32)
    quantize_chunk_asym<G, M>(p, it, e0, lane, raw, sel_lo, sel_hi, bw, ld_lo, ld_hi, rot, em);
  else if constexpr (F == kAsymBits)
    quantize_chunk_bits<G, M == kModeBase>(p, it, e0, lane, raw);
  else
    quantize_chunk_sym<G, F == kSymF16, M>(p, it, e0, lane, raw, sel_lo, sel_hi, bw, ld_lo, ld_hi, rot, em);
}

// (the width-generic stages and the prefix sums need more registers: two
// CTAs per SM)
template <int G, int F, int M>
__global__ void __launch_bounds__(kThreads, (F == kAsymBits || M == kModeEmit) ? 2 : RRQ_QUANTIZE_CTAS_PER_SM)
quantize_kernel(const __grid_constant__ QuantizeBatch p) {
  constexpr bool kBase = M == kModeBase;
  extern __shared__ __align__(128) uint8_t smem[];
  const int lane = threadIdx.x & 31;
  // the warp index by broadcast: the compiler then knows it (and every copy
  // and store operand derived from it) to be warp-uniform
  const int warp = __shfl_sync(kFullMask, static_cast<int>(threadIdx.x >> 5), 0);
  uint8_t* ring = smem + warp * (kRing * kChunkBytes);
  const uint32_t ring_s = smem_u32(ring);
  const uint32_t bar0 = smem_u32(smem + kWarps * kRing * kChunkBytes) + warp * kRing * 8;
  Emitter em{smem + kSmemBytes + warp * 2 * kChunkBytes, 0u};  // used by the build with prefixes

  const int64_t first = static_cast<int64_t>(blockIdx.x) * kWarps + warp;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kWarps;
  if (first >= p.total_chunks) return;  // warp-uniform: nothing issued, nothing to wait for

  if (lane == 0) {
#pragma unroll
    for (int b = 0; b < kRing; ++b) mbar_init(bar0 + 8 * b, 1);
    fence_mbarrier_init();
  }
  __syncwarp();

  // matrix of a chunk: chunks only move forward, so a running index suffices
  int m_issue = 0, m_work = 0;
  auto item_of = [&](int64_t chunk, int& m) -> const QuantizeItem& {
    while (m + 1 < p.count && chunk >= p.item[m + 1].chunk_begin) ++m;
    return p.item[m];
  };
  auto issue = [&](int64_t chunk, int b) {  // lane 0 only
    const QuantizeItem& it = item_of(chunk, m_issue);
    const int64_t e = (chunk - it.chunk_begin) * kChunkElems;
    const int64_t left = it.n - e;
    const uint32_t bytes = static_cast<uint32_t>((left < kChunkElems ? left : kChunkElems) * 2);
    mbar_arrive_expect_tx(bar0 + 8 * b, bytes);
    bulk_load(ring_s + b * kChunkBytes, it.W + e, bytes, bar0 + 8 * b);
  };
  if (lane == 0) {
#pragma unroll
    for (int b = 0; b < kRing; ++b) {
      const int64_t c = first + b * stride;
      if (c < p.total_chunks) issue(c, b);
    }
  }

  // Lane l reads its four 16-byte pieces in rotated order so that a quarter
  // warp touches eight distinct bank groups; slot j holds piece (j+rot)&3.
  // (The heterogeneous-width format packs its codes in natural order.)
  const int rot = F == kAsymBits ? 0 : (lane >> 1) & 3;
  const uint32_t sel_lo = rot == 0 ? 0x3210u : rot == 1 ? 0x1076u : rot == 2 ? 0x7654u : 0x5432u;
  const uint32_t sel_hi = rot == 0 ? 0x7654u : rot == 1 ? 0x5432u : rot == 2 ? 0x3210u : 0x1076u;
  // the inverse rotation, for a base code word read in memory order
  const uint32_t ld_lo = rot == 0 ? 0x3210u : rot == 1 ? 0x5432u : rot == 2 ? 0x7654u : 0x1076u;
  const uint32_t ld_hi = rot == 0 ? 0x7654u : rot == 1 ? 0x1076u : rot == 2 ? 0x3210u : 0x5432u;

  // base words of this warp's chunks, loaded one chunk ahead
  int m_base = 0;
  auto base_of = [&](int64_t chunk) -> BaseWords {
    // (per-stage widths read their base inside the chunk routine)
    if (!kBase || F == kAsymBits || chunk >= p.total_chunks) return BaseWords{make_uint2(0u, 0u), 0.0f, 0.0f};
    const QuantizeItem& it = item_of(chunk, m_base);
    return load_base<G, F>(it, (chunk - it.chunk_begin) * kChunkElems + static_cast<int64_t>(lane) * kLaneElems);
  };
  BaseWords bw_next = base_of(first);

  uint32_t iter = 0;
  for (int64_t chunk = first; chunk < p.total_chunks; chunk += stride, ++iter) {
    const int b = iter % kRing;
    const bool ready = mbar_wait(bar0 + 8 * b, (iter / kRing) & 1, p.wait_limit_us);
    if (!__all_sync(kFullMask, ready)) {
      // Give up: record it, wait (bounded) for this warp's copies in flight
      // so that none lands in freed shared memory, and leave.
      if (lane == 0) {
        atomicOr(p.status, kStatusTimeout);
        for (int j = 0; j < kRing; ++j) {
          if (chunk + j * stride >= p.total_chunks) break;
          const uint32_t jt = iter + j;
          mbar_wait(bar0 + 8 * (jt % kRing), (jt / kRing) & 1, kDrainLimitUs);
        }
        if (M == kModeEmit) bulk_wait<0>();  // this warp's output copies
      }
      __syncwarp();
      return;
    }
    const uint4* src = reinterpret_cast<const uint4*>(ring + b * kChunkBytes + lane * 64);
    uint4 raw[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) raw[j] = src[(j + rot) & 3];
    __syncwarp();
    if (lane == 0) {
      const int64_t next = chunk + kRing * stride;
      if (next < p.total_chunks) {
        fence_proxy_async_smem();
        issue(next, b);
      }
    }
    const QuantizeItem& it = item_of(chunk, m_work);
    const int64_t e0 = (chunk - it.chunk_begin) * kChunkElems + static_cast<int64_t>(lane) * kLaneElems;
    const BaseWords bw = bw_next;
    if (kBase) bw_next = base_of(chunk + stride);  // in flight while this chunk computes
    quantize_chunk<G, F, M>(p, it, e0, lane, raw, sel_lo, sel_hi, bw, ld_lo, ld_hi, rot, em);
  }
  if (M == kModeEmit && lane == 0) bulk_wait<0>();  // output copies done before the CTA exits
}

template <int M>
__host__ __device__ constexpr int smem_bytes() {
  return kSmemBytes + (M == kModeEmit ? kWarps * 2 * kChunkBytes : 0);
}

template <int G, int F, int M>
cudaError_t launch_gf(const QuantizeBatch& p, cudaStream_t stream, int sms) {
  // resident CTAs per multiprocessor: the same for every device of this
  // build, asked once (an atomic: any thread may launch)
  static std::atomic<int> cached{0};
  int blocks_per_sm = cached.load(std::memory_order_relaxed);
  if (blocks_per_sm == 0) {
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
        &blocks_per_sm, quantize_kernel<G, F, M>, kThreads, smem_bytes<M>());
    if (e != cudaSuccess) return e;
    if (blocks_per_sm < 1) blocks_per_sm = 1;
    cached.store(blocks_per_sm, std::memory_order_relaxed);
  }
  const int64_t want = (p.total_chunks + kWarps - 1) / kWarps;
  const int64_t cap = static_cast<int64_t>(sms) * blocks_per_sm;
  const int grid = static_cast<int>(want < cap ? want : cap);
  quantize_kernel<G, F, M><<<grid, kThreads, smem_bytes<M>(), stream>>>(p);
  return cudaGetLastError();
}

template <int F, int M>
cudaError_t launch_f(int group, const QuantizeBatch& p, cudaStream_t stream, int sms) {
  switch (group) {
    case 32: return launch_gf<32, F, M>(p, stream, sms);
    case 64: return launch_gf<64, F, M>(p, stream, sms);
    case 128: return launch_gf<128, F, M>(p, stream, sms);
    case 256: return launch_gf<256, F, M>(p, stream, sms);
    default: return cudaErrorInvalidValue;
  }
}

template <int F, int M>
cudaError_t prepare_f() {
  cudaError_t e;
  const cudaFuncAttribute a = cudaFuncAttributeMaxDynamicSharedMemorySize;
  if ((e = cudaFuncSetAttribute(quantize_kernel<32, F, M>, a, smem_bytes<M>()))) return e;
  if ((e = cudaFuncSetAttribute(quantize_kernel<64, F, M>, a, smem_bytes<M>()))) return e;
  if ((e = cudaFuncSetAttribute(quantize_kernel<128, F, M>, a, smem_bytes<M>()))) return e;
  return cudaFuncSetAttribute(quantize_kernel<256, F, M>, a, smem_bytes<M>());
}

// Set-up and launch of every format in one mode (instantiated by quantize.cu,
// quantize_base.cu and quantize_emit.cu).
template <int M>
cudaError_t prepare_all() {
  cudaError_t e;
  if ((e = prepare_f<kAsymF32, M>())) return e;
  if ((e = prepare_f<kSymF32, M>())) return e;
  if ((e = prepare_f<kSymF16, M>())) return e;
  if constexpr (M != kModeEmit) return prepare_f<kAsymBits, M>();
  return cudaSuccess;
}

template <int M>
cudaError_t launch_all(int group, Format fmt, const QuantizeBatch& p, cudaStream_t stream, int sms) {
  switch (fmt) {
    case kAsymF32: return launch_f<kAsymF32, M>(group, p, stream, sms);
    case kSymF32: return launch_f<kSymF32, M>(group, p, stream, sms);
    case kSymF16: return launch_f<kSymF16, M>(group, p, stream, sms);
    case kAsymBits:
      if constexpr (M != kModeEmit) return launch_f<kAsymBits, M>(group, p, stream, sms);
      break;
  }
  return cudaErrorInvalidValue;
}

}  // namespace
}  // namespace rrq
