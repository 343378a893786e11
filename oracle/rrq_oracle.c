/*
 * RRQ CPU oracle -- TEST INFRASTRUCTURE ONLY (see rrq_oracle.h).
 *
 * Plain, slow, single-threaded.  Every floating-point step is one IEEE-754
 * binary32 operation rounded to nearest-even; the build uses
 * -ffp-contract=off so that no multiply and add are fused, and no fast-math
 * flag, so subnormals are kept.
 *
 * What the paper fixes:
 *   Eq. 1   q = x / s + z            affine map of a group with shared s, z
 *   Eq. 2   Q = R(q)                 rounding to an integer code
 *   Eq. 3   r = x - (Q - z) s        residual after one stage
 *   Eq. 4-7 the base stage quantizes x, each residual stage k quantizes the
 *           running residual r_{k-1} and subtracts its dequantized value
 *   Eq. 8   prefix reconstruction = base + sum of the first t residual stages
 *   Algorithm 1 (no base checkpoint): quantize, store codes/scale/zero,
 *           dequantize, subtract, repeat for the residual stages
 *   Section 3.2: a 2-bit base plus three 2-bit residual stages gives the
 *           2/4/6/8-bit operating points; Section 5.1: group size 128.
 *
 * Readings taken where the paper leaves a detail open:
 *   - 2-bit asymmetric min/max grid: 4 levels, 2^2 - 1 = 3 steps over the
 *     group range (the range/(2^B - 1) step of Eq. 9).
 *   - The stored zero is the real offset m = lo = -z*s (the group minimum),
 *     so the dequantized value of code Q is m + Q*s, evaluated as
 *     fl(m + fl(Q*s)).  The range is not widened to include 0.
 *   - s = fl(fl(hi - lo) / 3);  Q = clamp(rhe(fl(fl(x - lo) / s)), 0, 3);
 *     if s == 0 every code is 0.
 *   - R is round-half-to-even (rhe).
 *   - Scale, zero and the running residual are binary32; the residual
 *     r = fl(x - fl(m + fl(Q*s))) never leaves binary32.
 *   - Every stage uses the same group partition.
 *   - min/max order -0 before +0, so the stored zero's sign is unique.
 *   - Reconstruction sums stage values in stage order in binary32:
 *     acc = L_0; acc = fl(acc + L_i) for i = 1..k-1; then bf16 round to
 *     nearest-even.
 */
#include "rrq_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

float rrq_oracle_bf16_to_f32(uint16_t h) {
  uint32_t u = (uint32_t)h << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return f;
}

uint16_t rrq_oracle_f32_to_bf16(float f) {
  uint32_t u;
  memcpy(&u, &f, sizeof u);
  if ((u & 0x7fffffffu) > 0x7f800000u) /* NaN: keep it a quiet NaN */
    return (uint16_t)((u >> 16) | 0x0040u);
  /* round to nearest, ties to even, on the upper 16 bits */
  u += 0x7fffu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

/* a comes strictly before b in the order  ... < -0 < +0 < ...  */
static int before(float a, float b) {
  if (a < b) return 1;
  if (a == b && signbit(a) && !signbit(b)) return 1;
  return 0;
}

/* round half to even, for 0 <= u < 2^22 (u - floor(u) is then exact) */
static float round_half_even(float u) {
  float f = floorf(u);
  float frac = u - f;
  if (frac > 0.5f) return f + 1.0f;
  if (frac < 0.5f) return f;
  /* exact tie: go to the even neighbour */
  return (fmodf(f, 2.0f) == 0.0f) ? f : f + 1.0f;
}

int rrq_oracle_quantize_group(const float* x, int g, int n_stages, uint8_t* Q,
                              float* scale, float* zero, float* resid) {
  if (g < 1 || n_stages < 1 || !x || !Q || !scale || !zero) return -1;
  float* v = (float*)malloc(sizeof(float) * (size_t)g);
  if (!v) return -1;
  for (int j = 0; j < g; ++j) v[j] = x[j];

  for (int k = 0; k < n_stages; ++k) {
    /* group range of the values this stage quantizes (x, then r_{k-1}) */
    float lo = v[0], hi = v[0];
    for (int j = 1; j < g; ++j) {
      if (before(v[j], lo)) lo = v[j];
      if (before(hi, v[j])) hi = v[j];
    }
    float range = hi - lo;
    float s = range / 3.0f; /* 2-bit grid: 2^2 - 1 steps */

    /* dequantized value of each code: m + Q*s with m = lo */
    float level[4];
    for (int q = 0; q < 4; ++q) {
      float qs = (float)q * s;
      level[q] = lo + qs;
    }

    for (int j = 0; j < g; ++j) {
      int code = 0;
      if (s != 0.0f) {
        float d = v[j] - lo;    /* x/s + z with z = -lo/s, evaluated as (x - lo)/s */
        float u = d / s;
        float r = round_half_even(u);
        code = (int)r;
        if (code < 0) code = 0;
        if (code > 3) code = 3;
      }
      Q[(size_t)k * g + j] = (uint8_t)code;
      v[j] = v[j] - level[code]; /* residual, Eq. 3 / Eq. 5 / Eq. 7 */
    }
    scale[k] = s;
    zero[k] = lo;
    if (resid)
      for (int j = 0; j < g; ++j) resid[(size_t)k * g + j] = v[j];
  }
  free(v);
  return 0;
}

int rrq_oracle_quantize(const uint16_t* W, int64_t rows, int64_t cols, int group,
                        int n_stages, uint8_t* const* codes, float* const* scales,
                        float* const* zeros) {
  if (!W || !codes || !scales || !zeros) return -1;
  if (rows < 1 || cols < 1 || group < 1 || n_stages < 1) return -1;
  if (cols % group != 0) return -1;
  const int64_t n = rows * cols;
  const int64_t n_groups = n / group;

  float* x = (float*)malloc(sizeof(float) * (size_t)group);
  uint8_t* Q = (uint8_t*)malloc((size_t)n_stages * (size_t)group);
  float* s = (float*)malloc(sizeof(float) * (size_t)n_stages);
  float* z = (float*)malloc(sizeof(float) * (size_t)n_stages);
  if (!x || !Q || !s || !z) {
    free(x); free(Q); free(s); free(z);
    return -1;
  }
  for (int k = 0; k < n_stages; ++k) memset(codes[k], 0, (size_t)((n + 3) / 4));

  for (int64_t gi = 0; gi < n_groups; ++gi) {
    const int64_t base = gi * group; /* groups are consecutive along a row */
    for (int j = 0; j < group; ++j) x[j] = rrq_oracle_bf16_to_f32(W[base + j]);
    rrq_oracle_quantize_group(x, group, n_stages, Q, s, z, NULL);
    for (int k = 0; k < n_stages; ++k) {
      for (int j = 0; j < group; ++j) {
        const int64_t c = base + j;
        codes[k][c / 4] |= (uint8_t)(Q[(size_t)k * group + j] << (2 * (c % 4)));
      }
      scales[k][gi] = s[k];
      zeros[k][gi] = z[k];
    }
  }
  free(x); free(Q); free(s); free(z);
  return 0;
}

int rrq_oracle_reconstruct(const uint8_t* const* codes, const float* const* scales,
                           const float* const* zeros, int64_t rows, int64_t cols,
                           int group, int k, uint16_t* out) {
  if (!codes || !scales || !zeros || !out) return -1;
  if (rows < 1 || cols < 1 || group < 1 || k < 1) return -1;
  if (cols % group != 0) return -1;
  const int64_t n = rows * cols;
  for (int64_t c = 0; c < n; ++c) {
    const int64_t gi = c / group;
    float acc = 0.0f;
    for (int i = 0; i < k; ++i) {
      const int q = (codes[i][c / 4] >> (2 * (c % 4))) & 3;
      float qs = (float)q * scales[i][gi];
      float value = zeros[i][gi] + qs; /* stage i's dequantized value */
      acc = (i == 0) ? value : acc + value;
    }
    out[c] = rrq_oracle_f32_to_bf16(acc);
  }
  return 0;
}
