// Device-side building blocks shared by the RRQ kernels (sm_103a):
// bulk-copy (TMA) and mbarrier wrappers with bounded waits, packed fp32x2
// arithmetic, and warp reductions.  Inline PTX only; no library kernels.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "rrq_internal.h"

namespace rrq {

constexpr unsigned kFullMask = 0xffffffffu;

// ---------------------------------------------------------------------------
// shared-memory addresses, mbarriers and 1-D bulk copies
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

// Makes the initialised barriers visible to the bulk-copy (async) proxy.
__device__ __forceinline__ void fence_mbarrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
      : "=r"(done)
      : "r"(bar), "r"(parity)
      : "memory");
  return done != 0;
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Waits for phase `parity` of a barrier for at most limit_us microseconds of
// wall time.  limit_us == 0 gives up at once (used to exercise error paths).
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, uint32_t limit_us) {
  if (limit_us == 0) return false;
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  const uint64_t limit_ns = static_cast<uint64_t>(limit_us) * 1000u;
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (globaltimer_ns() - t0 > limit_ns) return false;
  }
}

// Bounded wait that sleeps in the barrier instead of spinning: each try
// suspends the thread until the phase completes or about a millisecond
// passes, so waiting warps take no issue slots from the working ones.
__device__ __forceinline__ bool mbar_wait_sleep(uint32_t bar, uint32_t parity, uint32_t limit_us) {
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
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

// Orders this thread's generic-proxy shared-memory accesses before later
// bulk-copy (async-proxy) accesses of the same memory.
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// global -> shared bulk copy completing on `bar` (bytes % 16 == 0, both
// addresses 16-byte aligned).
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes,
                                          uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}

// shared -> global bulk copy tracked by the issuing thread's bulk groups.
__device__ __forceinline__ void bulk_store(void* dst, uint32_t src, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(src),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() {
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
// Waits until at most N committed bulk groups still read shared memory.
template <int N>
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
// Waits until at most N committed bulk groups are incomplete.
template <int N>
__device__ __forceinline__ void bulk_wait() {
  asm volatile("cp.async.bulk.wait_group %0;" ::"n"(N) : "memory");
}

// Per-thread asynchronous global -> shared copies (cp.async), tracked by the
// issuing thread's commit groups.  src_bytes = 0 fills the destination with
// zeros without reading global memory.
__device__ __forceinline__ void cp_async_8(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;" ::"r"(dst), "l"(src), "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_4(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(dst), "l"(src), "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_16(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes)
               : "memory");
}
// streaming (evict-first) 16-bit global store
__device__ __forceinline__ void stcs_u16(uint16_t* p, uint16_t v) {
  asm volatile("st.global.cs.u16 [%0], %1;" ::"l"(p), "h"(v) : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
// Waits until at most N of this thread's committed groups are pending.
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
// Arrives on `bar` once every earlier cp.async of this thread has landed,
// without raising the barrier's expected count (the count given at init
// includes this arrival).
__device__ __forceinline__ void cp_async_mbar_arrive_noinc(uint32_t bar) {
  asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(bar) : "memory");
}

// ---------------------------------------------------------------------------
// packed fp32x2 arithmetic (one instruction, two independent IEEE binary32
// operations rounded to nearest-even; subnormals kept)
// ---------------------------------------------------------------------------
typedef unsigned long long f32x2;

__device__ __forceinline__ f32x2 pack2(float lo, float hi) {
  f32x2 r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ f32x2 pack2u(uint32_t lo, uint32_t hi) {
  f32x2 r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "r"(lo), "r"(hi));
  return r;
}
// (x & M) | e in one three-input logic instruction, with e in a register: a
// code field masked in place under a float exponent (the code-to-float step
// of every dequantisation).  Written out because the two constants of the
// plain C form otherwise become an AND and an OR.
template <uint32_t M>
__device__ __forceinline__ uint32_t field_or(uint32_t x, uint32_t e) {
  uint32_t r;
  asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(r) : "r"(x), "n"(M), "r"(e));
  return r;
}
// the float (2^23 + Q 2^k) for the field of x at bits k, k+1 (mask M = 3 << k)
template <uint32_t M>
__device__ __forceinline__ uint32_t magic23(uint32_t x) {
  return field_or<M>(x, 0x4B000000u);
}

__device__ __forceinline__ void unpack2(f32x2 v, float& a, float& b) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(v));
}
__device__ __forceinline__ f32x2 add2(f32x2 a, f32x2 b) {
  f32x2 d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ f32x2 sub2(f32x2 a, f32x2 b) {
  f32x2 d;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ f32x2 mul2(f32x2 a, f32x2 b) {
  f32x2 d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ f32x2 fma2(f32x2 a, f32x2 b, f32x2 c) {
  f32x2 d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}

// three-input minimum / maximum (sm_100+)
__device__ __forceinline__ float min3(float a, float b, float c) {
  float d;
  asm("min.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
__device__ __forceinline__ float max3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// Stage values of 32 codes of width B (element j at bits B*j of w), natural
// order: acc = level (first stage) or fl(acc + level).
template <int B>
__device__ __forceinline__ void dequant_bits(const uint4& w4, float s, float z, bool first, f32x2 (&acc)[16]) {
  const uint32_t w[4] = {w4.x, w4.y, w4.z, w4.w};
  auto code = [&](int j) -> uint32_t {  // bits B*j.. of the code, unmasked above
    const int bit = B * j, i = bit >> 5, sh = bit & 31;
    uint32_t c = w[i] >> sh;
    if (sh + B > 32) c |= w[i + 1] << (32 - sh);
    return c;
  };
  const f32x2 S = pack2(s, s), Z = pack2(z, z), T23 = pack2(8388608.0f, 8388608.0f), Z0 = pack2(0.0f, 0.0f);
#pragma unroll
  for (int m = 0; m < 16; ++m) {
    const f32x2 t = pack2u(magic23<(1u << B) - 1u>(code(2 * m)), magic23<(1u << B) - 1u>(code(2 * m + 1)));
    const f32x2 level = add2(Z, fma2(sub2(t, T23), S, Z0));  // fl(zero + fl(Q s))
    acc[m] = first ? level : add2(acc[m], level);
  }
}

// A scale for which 2^17 s .. 2^23 s (and s / 64) are exact binary32
// values, so that a code left in its bit field gives Q s with a single
// rounding inside one fma (see asym_levels; a conservative range).
__device__ __forceinline__ bool prescale_ok(float s) {
  return s == 0.0f || (s >= 0x1p-100f && s <= 0x1p+100f);
}

// ---------------------------------------------------------------------------
// stage levels of 2-bit codes, four to a byte (code j at bits 2j, 2j+1)
// ---------------------------------------------------------------------------
// Code j stays in place under the float exponent of 2^(23-2j), so that
// t_j = 2^(23-2j) + Q exactly (one logic op).  Asymmetric level
// fl(zero + fl(Q s)): fma(t_j, s, -2^(23-2j) s) rounds Q s once when
// 2^(23-2j) s is exact (prescale_ok(s)), then one add.  Symmetric level
// (Q - 2) s: t_j - (2^(23-2j) + 2) = Q - 2 exactly, and its product with s is
// exact (or overflows exactly as the definition's does) for every s.
struct StageConsts {
  f32x2 S;    // (s, s)
  f32x2 C01;  // (-2^23 s, -2^21 s)
  f32x2 C23;  // (-2^19 s, -2^17 s)
  f32x2 Z;    // (zero, zero)
};

__device__ __forceinline__ StageConsts stage_consts(float s, float zero) {
  const f32x2 S = pack2(s, s);
  return {S, mul2(S, pack2(-0x1p23f, -0x1p21f)), mul2(S, pack2(-0x1p19f, -0x1p17f)), pack2(zero, zero)};
}
// (t_0, t_1) and (t_2, t_3) of byte b
__device__ __forceinline__ f32x2 code_t01(uint32_t b) {
  return pack2u(field_or<0x03u>(b, 0x4B000000u), field_or<0x0Cu>(b, 0x4A000000u));
}
__device__ __forceinline__ f32x2 code_t23(uint32_t b) {
  return pack2u(field_or<0x30u>(b, 0x49000000u), field_or<0xC0u>(b, 0x48000000u));
}
// asymmetric levels fl(zero + fl(Q s)) of codes 0,1 and 2,3 of byte b
// (prescale_ok(s) required)
__device__ __forceinline__ void asym_levels(uint32_t b, const StageConsts& c, f32x2& l01, f32x2& l23) {
  l01 = add2(c.Z, fma2(code_t01(b), c.S, c.C01));
  l23 = add2(c.Z, fma2(code_t23(b), c.S, c.C23));
}
// Q - 2 of codes 0,1 and 2,3 of byte b (exact)
__device__ __forceinline__ void sym_offsets(uint32_t b, f32x2& u01, f32x2& u23) {
  u01 = sub2(code_t01(b), pack2(0x1p23f + 2.0f, 0x1p21f + 2.0f));
  u23 = sub2(code_t23(b), pack2(0x1p19f + 2.0f, 0x1p17f + 2.0f));
}

// min and max over 16 packed pairs (32 values) held by one lane
__device__ __forceinline__ void lane_minmax(const f32x2 (&v)[16], float& lo, float& hi) {
  float a, b, c, d;
  unpack2(v[0], a, b);
  unpack2(v[1], c, d);
  float lo0 = fminf(a, b), hi0 = fmaxf(a, b);
  float lo1 = fminf(c, d), hi1 = fmaxf(c, d);
#pragma unroll
  for (int i = 2; i < 16; i += 2) {
    unpack2(v[i], a, b);
    unpack2(v[i + 1], c, d);
    lo0 = min3(lo0, a, b);
    hi0 = max3(hi0, a, b);
    lo1 = min3(lo1, c, d);
    hi1 = max3(hi1, c, d);
  }
  lo = fminf(lo0, lo1);
  hi = fmaxf(hi0, hi1);
}

// max |v| over 16 packed pairs held by one lane
__device__ __forceinline__ float lane_amax(const f32x2 (&v)[16]) {
  float m0 = 0.0f, m1 = 0.0f;
#pragma unroll
  for (int i = 0; i < 16; i += 2) {
    float a, b, c, d;
    unpack2(v[i], a, b);
    unpack2(v[i + 1], c, d);
    m0 = max3(m0, fabsf(a), fabsf(b));
    m1 = max3(m1, fabsf(c), fabsf(d));
  }
  return fmaxf(m0, m1);
}

// reductions over the L consecutive lanes that share one group (L | 32)
template <int L>
__device__ __forceinline__ float group_max(float x) {
#pragma unroll
  for (int off = 1; off < L; off <<= 1) x = fmaxf(x, __shfl_xor_sync(kFullMask, x, off));
  return x;
}
template <int L>
__device__ __forceinline__ void group_minmax(float& lo, float& hi) {
#pragma unroll
  for (int off = 1; off < L; off <<= 1) {
    lo = fminf(lo, __shfl_xor_sync(kFullMask, lo, off));
    hi = fmaxf(hi, __shfl_xor_sync(kFullMask, hi, off));
  }
}
template <int L>
__device__ __forceinline__ uint32_t group_or(uint32_t x) {
#pragma unroll
  for (int off = 1; off < L; off <<= 1) x |= __shfl_xor_sync(kFullMask, x, off);
  return x;
}

}  // namespace rrq
