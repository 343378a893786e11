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
 *
 * Symmetric grid (the paper's timed and packaged configuration: "symmetric"
 * quantization type in Table 4, no stored zero-points and a 16-bit scale per
 * group of 128 in Appendix G), readings where the paper gives no formula:
 *   - the zero-point of Eq. 1-3 is the implicit constant z = 2 (half of the
 *     4 levels), so the dequantized value of code Q is (Q - 2) * s and the
 *     levels are {-2s, -s, 0, s};
 *   - s = fl(fl(2 * amax) / 3) with amax = max |x| over the group, so that
 *     the extreme magnitude sits 1.5 steps from 0;
 *   - Q = clamp(rhe(fl(x / s)) + 2, 0, 3) (the clamp is active at the
 *     positive end: fl(amax / s) rounds to 2); if s == 0 every code is 2;
 *   - with 16-bit scales, s is rounded to IEEE binary16 (nearest-even) first
 *     and the stage quantizes against the stored value, so that construction
 *     and reconstruction use the same scale;
 *   - (Q - 2) * s is exact in binary32, so the residual is fl(x - (Q-2)*s).
 *
 * Stage-wise product (Appendix C: A W~_(t) = A W^_0 + sum_k A R^_k): with
 * the prefix-k weight W~[r][c] = the binary32 stage sum of the reconstruction
 * (before its bf16 rounding), Y[b][r] = sum_c W~[r][c] * A[b][c], the
 * products and the sum taken in binary64 (each product of a binary32 and a
 * bf16 value is exact there).
 *
 * Prefill form of the same product (many activation rows, bf16 operands as
 * a tensor-core GEMM takes them): the weight is the bf16 prefix
 * reconstruction itself, Y[t][r] = sum_c bf16(W~[r][c]) * A[t][c] in
 * binary64 (products of two bf16 values are exact there).
 *
 * Heterogeneous stage widths (Section 3.2: stage k may use b_k bits, B_t is
 * the sum of the widths; the split analysis of Section 3.3 / Table 3 uses
 * zero-point grids): stage k of the asymmetric grid with b bits has
 * m = 2^b - 1 steps, s = fl(fl(hi - lo) / m), Q = clamp(rhe(fl(fl(v - lo)/s)),
 * 0, m), level fl(lo + fl(Q s)); codes are packed LSB-first, element c of the
 * stage at bits b*c .. b*c + b - 1 of the stage's byte array.
 *
 * Group peak-to-mean ratio (Section 3.1 and Table 9's K/MAE): for a group,
 * max |x| / (sum |x| / g), taken in binary64; 0 for an all-zero group.
 *
 * Algorithm 1 with a base checkpoint: stage 0 of the package is given (codes,
 * scales and, for the asymmetric grid, zeros, in the package's own format);
 * it is dequantized with the same level formula as a computed stage 0, the
 * running residual starts as fl(x - L_0), and stages 1.. are quantized from it
 * exactly as in the build without a checkpoint.
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

/* Round half to even of a double holding an integer plus a fraction that is
 * exact (at most 53 significant bits, 0 <= u). */
static double rhe_double(double u) {
  double f = floor(u);
  double frac = u - f;
  if (frac > 0.5) return f + 1.0;
  if (frac < 0.5) return f;
  return (fmod(f, 2.0) == 0.0) ? f : f + 1.0;
}

/* IEEE 754 binary16 (1 sign, 5 exponent, 10 fraction bits, bias 15) nearest
 * to f, ties to even; subnormals kept; magnitudes from 65520 (the midpoint
 * between the largest finite 65504 and 2^16) up round to infinity. */
uint16_t rrq_oracle_f32_to_f16(float f) {
  const uint16_t sign = signbit(f) ? 0x8000u : 0u;
  if (isnan(f)) return (uint16_t)(sign | 0x7e00u);
  const double a = fabs((double)f);
  if (a >= 65520.0) return (uint16_t)(sign | 0x7c00u);
  if (a < ldexp(1.0, -14)) {
    /* subnormal range: multiples of 2^-24; 1024 * 2^-24 is the smallest
     * normal, whose encoding is 1024 as well */
    const double n = rhe_double(a * ldexp(1.0, 24)); /* exact scaling */
    return (uint16_t)(sign | (uint16_t)n);
  }
  int e;
  const double m = frexp(a, &e); /* a = m * 2^e, 0.5 <= m < 1 */
  int exp = e - 1;               /* a = (2m) * 2^exp, 1 <= 2m < 2 */
  double frac = rhe_double((2.0 * m - 1.0) * 1024.0); /* 10 fraction bits */
  if (frac == 1024.0) { frac = 0.0; exp += 1; }         /* rounded up to 2^(exp+1) */
  if (exp + 15 >= 31) return (uint16_t)(sign | 0x7c00u);
  return (uint16_t)(sign | (uint16_t)((exp + 15) << 10) | (uint16_t)frac);
}

float rrq_oracle_f16_to_f32(uint16_t h) {
  const int e = (h >> 10) & 0x1f;
  const int frac = h & 0x3ff;
  double v;
  if (e == 0) v = ldexp((double)frac, -24);
  else if (e == 31) v = frac ? NAN : INFINITY;
  else v = ldexp((double)(1024 + frac), e - 25);
  return (float)((h & 0x8000u) ? -v : v);
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

/* element c's 2-bit code goes to byte c/4, bits 2*(c%4) and up */
static void put_code(uint8_t* codes, int64_t c, int q) {
  codes[c / 4] |= (uint8_t)(q << (2 * (c % 4)));
}

/* rhe for either sign: rounding half to even is odd-symmetric */
static float round_half_even_signed(float u) {
  return u < 0.0f ? -round_half_even(-u) : round_half_even(u);
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
      for (int j = 0; j < group; ++j) put_code(codes[k], base + j, Q[(size_t)k * group + j]);
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

int rrq_oracle_quantize_group_sym(const float* x, int g, int n_stages, int scale_f16,
                                  uint8_t* Q, float* scale, float* resid) {
  if (g < 1 || n_stages < 1 || !x || !Q || !scale) return -1;
  float* v = (float*)malloc(sizeof(float) * (size_t)g);
  if (!v) return -1;
  for (int j = 0; j < g; ++j) v[j] = x[j];

  for (int k = 0; k < n_stages; ++k) {
    /* largest magnitude of the values this stage quantizes */
    float amax = 0.0f;
    for (int j = 0; j < g; ++j)
      if (fabsf(v[j]) > amax) amax = fabsf(v[j]);
    float span = 2.0f * amax; /* exact: power-of-two scaling */
    float s = span / 3.0f;    /* levels -2s..s: amax is 1.5 steps from 0 */
    if (scale_f16) s = rrq_oracle_f16_to_f32(rrq_oracle_f32_to_f16(s));

    for (int j = 0; j < g; ++j) {
      int code = 2; /* implicit zero-point */
      if (s != 0.0f) {
        float u = v[j] / s; /* Eq. 1 with z = 2 applied after rounding */
        code = (int)round_half_even_signed(u) + 2;
        code = code < 0 ? 0 : code;
        code = code > 3 ? 3 : code;
      }
      Q[(size_t)k * g + j] = (uint8_t)code;
      float level = (float)(code - 2) * s; /* (Q - z) s, Eq. 3; exact */
      v[j] = v[j] - level;
    }
    scale[k] = s;
    if (resid)
      for (int j = 0; j < g; ++j) resid[(size_t)k * g + j] = v[j];
  }
  free(v);
  return 0;
}

int rrq_oracle_quantize_sym(const uint16_t* W, int64_t rows, int64_t cols, int group,
                            int n_stages, int scale_f16, uint8_t* const* codes,
                            void* const* scales) {
  if (!W || !codes || !scales) return -1;
  if (rows < 1 || cols < 1 || group < 1 || n_stages < 1) return -1;
  if (cols % group != 0) return -1;
  const int64_t n = rows * cols;
  const int64_t n_groups = n / group;

  float* x = (float*)malloc(sizeof(float) * (size_t)group);
  uint8_t* Q = (uint8_t*)malloc((size_t)n_stages * (size_t)group);
  float* s = (float*)malloc(sizeof(float) * (size_t)n_stages);
  if (!x || !Q || !s) {
    free(x); free(Q); free(s);
    return -1;
  }
  for (int k = 0; k < n_stages; ++k) memset(codes[k], 0, (size_t)((n + 3) / 4));

  for (int64_t gi = 0; gi < n_groups; ++gi) {
    const int64_t base = gi * group;
    for (int j = 0; j < group; ++j) x[j] = rrq_oracle_bf16_to_f32(W[base + j]);
    rrq_oracle_quantize_group_sym(x, group, n_stages, scale_f16, Q, s, NULL);
    for (int k = 0; k < n_stages; ++k) {
      for (int j = 0; j < group; ++j) put_code(codes[k], base + j, Q[(size_t)k * group + j]);
      if (scale_f16) ((uint16_t*)scales[k])[gi] = rrq_oracle_f32_to_f16(s[k]);
      else ((float*)scales[k])[gi] = s[k];
    }
  }
  free(x); free(Q); free(s);
  return 0;
}

int rrq_oracle_reconstruct_sym(const uint8_t* const* codes, const void* const* scales,
                               int64_t rows, int64_t cols, int group, int k, int scale_f16,
                               uint16_t* out) {
  if (!codes || !scales || !out) return -1;
  if (rows < 1 || cols < 1 || group < 1 || k < 1) return -1;
  if (cols % group != 0) return -1;
  const int64_t n = rows * cols;
  for (int64_t c = 0; c < n; ++c) {
    const int64_t gi = c / group;
    float acc = 0.0f;
    for (int i = 0; i < k; ++i) {
      const int q = (codes[i][c / 4] >> (2 * (c % 4))) & 3;
      const float s = scale_f16 ? rrq_oracle_f16_to_f32(((const uint16_t*)scales[i])[gi])
                                : ((const float*)scales[i])[gi];
      float level = (float)(q - 2) * s; /* stage i's dequantized value */
      acc = (i == 0) ? level : acc + level;
    }
    out[c] = rrq_oracle_f32_to_bf16(acc);
  }
  return 0;
}

/* dequantized value of one given base code (the level formula of the grid) */
static float base_level(int grid_sym, int q, float s, float z) {
  if (grid_sym) return (float)(q - 2) * s;
  float qs = (float)q * s;
  return z + qs;
}

int rrq_oracle_quantize_from_base(const uint16_t* W, int64_t rows, int64_t cols, int group,
                                  int n_stages, int grid_sym, int scale_f16,
                                  uint8_t* const* codes, void* const* scales,
                                  float* const* zeros) {
  if (!W || !codes || !scales || (!grid_sym && !zeros)) return -1;
  if (rows < 1 || cols < 1 || group < 1 || n_stages < 2) return -1;
  if (cols % group != 0 || (scale_f16 && !grid_sym)) return -1;
  const int64_t n = rows * cols;
  const int64_t n_groups = n / group;
  const int rs = n_stages - 1; /* residual stages computed here */

  float* r = (float*)malloc(sizeof(float) * (size_t)group);
  uint8_t* Q = (uint8_t*)malloc((size_t)rs * (size_t)group);
  float* s = (float*)malloc(sizeof(float) * (size_t)rs);
  float* z = (float*)malloc(sizeof(float) * (size_t)rs);
  if (!r || !Q || !s || !z) {
    free(r); free(Q); free(s); free(z);
    return -1;
  }
  for (int k = 1; k < n_stages; ++k) memset(codes[k], 0, (size_t)((n + 3) / 4));

  for (int64_t gi = 0; gi < n_groups; ++gi) {
    const int64_t base = gi * group;
    const float s0 = scale_f16 ? rrq_oracle_f16_to_f32(((const uint16_t*)scales[0])[gi])
                               : ((const float*)scales[0])[gi];
    const float z0 = grid_sym ? 0.0f : zeros[0][gi];
    for (int j = 0; j < group; ++j) {
      const int64_t c = base + j;
      const int q0 = (codes[0][c / 4] >> (2 * (c % 4))) & 3;
      const float x = rrq_oracle_bf16_to_f32(W[c]);
      r[j] = x - base_level(grid_sym, q0, s0, z0); /* R_0 = W - W_0 */
    }
    if (grid_sym) rrq_oracle_quantize_group_sym(r, group, rs, scale_f16, Q, s, NULL);
    else rrq_oracle_quantize_group(r, group, rs, Q, s, z, NULL);
    for (int k = 1; k < n_stages; ++k) {
      for (int j = 0; j < group; ++j) put_code(codes[k], base + j, Q[(size_t)(k - 1) * group + j]);
      if (scale_f16) ((uint16_t*)scales[k])[gi] = rrq_oracle_f32_to_f16(s[k - 1]);
      else ((float*)scales[k])[gi] = s[k - 1];
      if (!grid_sym) zeros[k][gi] = z[k - 1];
    }
  }
  free(r); free(Q); free(s); free(z);
  return 0;
}

int rrq_oracle_gemv(const uint8_t* const* codes, const void* const* scales,
                    const float* const* zeros, int64_t rows, int64_t cols, int group, int k,
                    int grid_sym, int scale_f16, const uint16_t* A, int batch, double* Y) {
  if (!codes || !scales || (!grid_sym && !zeros) || !A || !Y) return -1;
  if (rows < 1 || cols < 1 || group < 1 || k < 1 || batch < 1) return -1;
  if (cols % group != 0 || (scale_f16 && !grid_sym)) return -1;
  for (int b = 0; b < batch; ++b)
    for (int64_t r = 0; r < rows; ++r) Y[(size_t)b * rows + r] = 0.0;
  for (int64_t r = 0; r < rows; ++r) {
    for (int64_t j = 0; j < cols; ++j) {
      const int64_t c = r * cols + j;
      const int64_t gi = c / group;
      float w = 0.0f; /* prefix weight W~[r][j] */
      for (int i = 0; i < k; ++i) {
        const int q = (codes[i][c / 4] >> (2 * (c % 4))) & 3;
        const float s = scale_f16 ? rrq_oracle_f16_to_f32(((const uint16_t*)scales[i])[gi])
                                  : ((const float*)scales[i])[gi];
        const float lv = base_level(grid_sym, q, s, grid_sym ? 0.0f : zeros[i][gi]);
        w = (i == 0) ? lv : w + lv;
      }
      for (int b = 0; b < batch; ++b)
        Y[(size_t)b * rows + r] += (double)w * (double)rrq_oracle_bf16_to_f32(A[(size_t)b * cols + j]);
    }
  }
  return 0;
}

/* Asymmetric 2^b-level stages with per-stage widths; see the file comment. */
int rrq_oracle_quantize_group_bits(const float* x, int g, int n_stages, const int* bits,
                                   uint8_t* Q, float* scale, float* zero, float* resid) {
  if (g < 1 || n_stages < 1 || !x || !bits || !Q || !scale || !zero) return -1;
  for (int k = 0; k < n_stages; ++k)
    if (bits[k] < 1 || bits[k] > 4) return -1;
  float* v = (float*)malloc(sizeof(float) * (size_t)g);
  if (!v) return -1;
  for (int j = 0; j < g; ++j) v[j] = x[j];

  for (int k = 0; k < n_stages; ++k) {
    const int m = (1 << bits[k]) - 1; /* steps of a b-bit grid */
    float lo = v[0], hi = v[0]; /* range of this stage's values, -0 before +0 */
    for (int j = 1; j < g; ++j) {
      lo = before(v[j], lo) ? v[j] : lo;
      hi = before(hi, v[j]) ? v[j] : hi;
    }
    const float span = hi - lo;
    float s = span / (float)m;
    for (int j = 0; j < g; ++j) {
      int code = 0;
      if (s != 0.0f) {
        const float dist = v[j] - lo;
        const float u = dist / s;
        code = (int)round_half_even(u);
        code = code < 0 ? 0 : (code > m ? m : code);
      }
      Q[(size_t)k * g + j] = (uint8_t)code;
      float qs = (float)code * s;
      float lv = lo + qs;
      v[j] = v[j] - lv;
    }
    scale[k] = s;
    zero[k] = lo;
    if (resid)
      for (int j = 0; j < g; ++j) resid[(size_t)k * g + j] = v[j];
  }
  free(v);
  return 0;
}

/* element c's b-bit code at bits b*c.. of the stage's byte array (LSB first) */
static void put_bits(uint8_t* codes, int64_t c, int b, int q) {
  for (int t = 0; t < b; ++t) {
    const int64_t bit = c * b + t;
    if ((q >> t) & 1) codes[bit / 8] |= (uint8_t)(1u << (bit % 8));
  }
}
static int get_bits(const uint8_t* codes, int64_t c, int b) {
  int q = 0;
  for (int t = 0; t < b; ++t) {
    const int64_t bit = c * b + t;
    q |= ((codes[bit / 8] >> (bit % 8)) & 1) << t;
  }
  return q;
}

int rrq_oracle_quantize_bits(const uint16_t* W, int64_t rows, int64_t cols, int group,
                             int n_stages, const int* bits, uint8_t* const* codes,
                             float* const* scales, float* const* zeros) {
  if (!W || !bits || !codes || !scales || !zeros) return -1;
  if (rows < 1 || cols < 1 || group < 1 || n_stages < 1 || cols % group != 0) return -1;
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
  for (int k = 0; k < n_stages; ++k) memset(codes[k], 0, (size_t)((n * bits[k] + 7) / 8));
  for (int64_t gi = 0; gi < n_groups; ++gi) {
    const int64_t base = gi * group;
    for (int j = 0; j < group; ++j) x[j] = rrq_oracle_bf16_to_f32(W[base + j]);
    if (rrq_oracle_quantize_group_bits(x, group, n_stages, bits, Q, s, z, NULL) != 0) {
      free(x); free(Q); free(s); free(z);
      return -1;
    }
    for (int k = 0; k < n_stages; ++k) {
      for (int j = 0; j < group; ++j) put_bits(codes[k], base + j, bits[k], Q[(size_t)k * group + j]);
      scales[k][gi] = s[k];
      zeros[k][gi] = z[k];
    }
  }
  free(x); free(Q); free(s); free(z);
  return 0;
}

int rrq_oracle_reconstruct_bits(const uint8_t* const* codes, const float* const* scales,
                                const float* const* zeros, int64_t rows, int64_t cols, int group,
                                int k, const int* bits, uint16_t* out) {
  if (!codes || !scales || !zeros || !bits || !out) return -1;
  if (rows < 1 || cols < 1 || group < 1 || k < 1 || cols % group != 0) return -1;
  const int64_t n = rows * cols;
  for (int64_t c = 0; c < n; ++c) {
    const int64_t gi = c / group;
    float acc = 0.0f;
    for (int i = 0; i < k; ++i) {
      const int q = get_bits(codes[i], c, bits[i]);
      float qs = (float)q * scales[i][gi];
      float lv = zeros[i][gi] + qs;
      if (i == 0) acc = lv;
      else acc = acc + lv;
    }
    out[c] = rrq_oracle_f32_to_bf16(acc);
  }
  return 0;
}

int rrq_oracle_group_pmr(const uint16_t* W, int64_t rows, int64_t cols, int group, double* pmr) {
  if (!W || !pmr || rows < 1 || cols < 1 || group < 1 || cols % group != 0) return -1;
  const int64_t n_groups = rows * cols / group;
  for (int64_t gi = 0; gi < n_groups; ++gi) {
    double peak = 0.0, sum = 0.0;
    for (int j = 0; j < group; ++j) {
      const double a = fabs((double)rrq_oracle_bf16_to_f32(W[gi * group + j]));
      if (a > peak) peak = a;
      sum += a;
    }
    pmr[gi] = sum > 0.0 ? peak / (sum / (double)group) : 0.0;
  }
  return 0;
}

/* bf16 prefix-k weight of flat element c: the binary32 stage sum of the
 * first k stages (stage order), rounded to nearest-even bf16 -- the value the
 * prefix reconstruction returns for that element. */
static uint16_t prefill_weight(const uint8_t* const* codes, const void* const* scales,
                               const float* const* zeros, int64_t c, int group, int k,
                               int grid_sym, int scale_f16) {
  const int64_t g = c / group;
  float sum = 0.0f;
  for (int st = 0; st < k; ++st) {
    const int code = (codes[st][c / 4] >> (2 * (c % 4))) & 3;
    const float sc = scale_f16 ? rrq_oracle_f16_to_f32(((const uint16_t*)scales[st])[g])
                               : ((const float*)scales[st])[g];
    const float level = base_level(grid_sym, code, sc, grid_sym ? 0.0f : zeros[st][g]);
    sum = st == 0 ? level : sum + level;
  }
  return rrq_oracle_f32_to_bf16(sum);
}

int rrq_oracle_prefill(const uint8_t* const* codes, const void* const* scales,
                       const float* const* zeros, int64_t rows, int64_t cols, int group, int k,
                       int grid_sym, int scale_f16, const uint16_t* A, int64_t tokens, double* Y) {
  if (!codes || !scales || (!grid_sym && !zeros) || !A || !Y) return -1;
  if (rows < 1 || cols < 1 || group < 1 || k < 1 || tokens < 1) return -1;
  if (cols % group != 0 || (scale_f16 && !grid_sym)) return -1;
  double* wrow = (double*)malloc(sizeof(double) * (size_t)cols);
  if (!wrow) return -1;
  for (int64_t r = 0; r < rows; ++r) {
    for (int64_t j = 0; j < cols; ++j)
      wrow[j] = (double)rrq_oracle_bf16_to_f32(
          prefill_weight(codes, scales, zeros, r * cols + j, group, k, grid_sym, scale_f16));
    for (int64_t t = 0; t < tokens; ++t) {
      double dot = 0.0;
      for (int64_t j = 0; j < cols; ++j)
        dot += wrow[j] * (double)rrq_oracle_bf16_to_f32(A[(size_t)t * cols + j]);
      Y[(size_t)t * rows + r] = dot;
    }
  }
  free(wrow);
  return 0;
}

/* Products with the prefix weights of a package with per-stage widths
 * (asymmetric grid, codes LSB-first at bits[i] per weight): the prefix-k
 * weight is the binary32 stage sum of zero + fl(Q s), as in
 * rrq_oracle_reconstruct_bits; taken as it is (the decode form) or rounded
 * to nearest-even bf16 (the prefill form, bf16_weights != 0), and
 * Y[t][r] = sum_c w(r, c) A[t][c] in binary64. */
int rrq_oracle_product_bits(const uint8_t* const* codes, const float* const* scales,
                            const float* const* zeros, int64_t rows, int64_t cols, int group, int k,
                            const int* bits, const uint16_t* A, int64_t tokens, int bf16_weights,
                            double* Y) {
  if (!codes || !scales || !zeros || !bits || !A || !Y) return -1;
  if (rows < 1 || cols < 1 || group < 1 || k < 1 || tokens < 1 || cols % group != 0) return -1;
  for (int i = 0; i < k; ++i)
    if (bits[i] < 1 || bits[i] > 4) return -1;
  double* wts = (double*)malloc(sizeof(double) * (size_t)cols);
  if (!wts) return -1;
  for (int64_t r = 0; r < rows; ++r) {
    for (int64_t j = 0; j < cols; ++j) {
      const int64_t c = r * cols + j;
      const int64_t g = c / group;
      float running = 0.0f;
      for (int st = 0; st != k; ++st) {
        const int code = get_bits(codes[st], c, bits[st]);
        const float scaled = (float)code * scales[st][g];
        const float lvl = zeros[st][g] + scaled;
        running = st == 0 ? lvl : running + lvl;
      }
      wts[j] = bf16_weights ? (double)rrq_oracle_bf16_to_f32(rrq_oracle_f32_to_bf16(running)) : (double)running;
    }
    for (int64_t t = 0; t < tokens; ++t) {
      double sum = 0.0;
      for (int64_t j = 0; j < cols; ++j) sum += wts[j] * (double)rrq_oracle_bf16_to_f32(A[(size_t)t * cols + j]);
      Y[(size_t)t * rows + r] = sum;
    }
  }
  free(wts);
  return 0;
}

/* Algorithm 1 with a base checkpoint, per-stage widths (asymmetric grid):
 * stage 0 is given (bits[0]-bit codes, scale and zero in codes[0],
 * scales[0], zeros[0]); R_0 = x - fl(zero + fl(Q s)); stages 1..n_stages-1
 * quantize the running residual at widths bits[1..] exactly as
 * rrq_oracle_quantize_group_bits does. */
int rrq_oracle_quantize_from_base_bits(const uint16_t* W, int64_t rows, int64_t cols, int group,
                                       int n_stages, const int* bits, uint8_t* const* codes,
                                       float* const* scales, float* const* zeros) {
  if (!W || !bits || !codes || !scales || !zeros) return -1;
  if (rows < 1 || cols < 1 || group < 1 || n_stages < 2 || cols % group != 0) return -1;
  for (int k = 0; k < n_stages; ++k)
    if (bits[k] < 1 || bits[k] > 4) return -1;
  const int64_t n = rows * cols;
  const int64_t n_groups = n / group;
  const int rest = n_stages - 1;
  float* r0 = (float*)malloc(sizeof(float) * (size_t)group);
  uint8_t* Qr = (uint8_t*)malloc((size_t)rest * (size_t)group);
  float* sr = (float*)malloc(sizeof(float) * (size_t)rest);
  float* zr = (float*)malloc(sizeof(float) * (size_t)rest);
  if (!r0 || !Qr || !sr || !zr) {
    free(r0); free(Qr); free(sr); free(zr);
    return -1;
  }
  for (int k = 1; k < n_stages; ++k) memset(codes[k], 0, (size_t)((n * bits[k] + 7) / 8));
  for (int64_t gi = 0; gi < n_groups; ++gi) {
    const int64_t first = gi * group;
    for (int j = 0; j < group; ++j) {
      const int q0 = get_bits(codes[0], first + j, bits[0]);
      const float based = (float)q0 * scales[0][gi];
      const float base_level_w = zeros[0][gi] + based;
      r0[j] = rrq_oracle_bf16_to_f32(W[first + j]) - base_level_w; /* R_0 = W - W_0 */
    }
    if (rrq_oracle_quantize_group_bits(r0, group, rest, bits + 1, Qr, sr, zr, NULL) != 0) {
      free(r0); free(Qr); free(sr); free(zr);
      return -1;
    }
    for (int k = 1; k < n_stages; ++k) {
      for (int j = 0; j < group; ++j) put_bits(codes[k], first + j, bits[k], Qr[(size_t)(k - 1) * group + j]);
      scales[k][gi] = sr[k - 1];
      zeros[k][gi] = zr[k - 1];
    }
  }
  free(r0); free(Qr); free(sr); free(zr);
  return 0;
}
