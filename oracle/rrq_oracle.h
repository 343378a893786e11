/*
 * Plain CPU oracle for Recurrent Residual Quantization (RRQ) with 2-bit
 * round-to-nearest stages: TEST INFRASTRUCTURE ONLY.
 *
 * Only the test suite, the smoke check and the benchmark's CPU-baseline leg
 * may load this library.  The product path (the CUDA library) never calls it
 * and shares no code, header, table or helper with it.
 *
 * The arithmetic follows the paper's representation statement (Section 3.1,
 * Eq. 1-3), the recursion (Section 3.2, Eq. 4-7), Algorithm 1 (build without
 * a base checkpoint) and the prefix reconstruction (Eq. 8), in IEEE-754
 * binary32, one operation at a time, with no fused multiply-add and
 * round-half-to-even for the code rounding.  See rrq_oracle.c for the
 * readings taken where the paper leaves a detail open.
 */
#ifndef RRQ_ORACLE_H
#define RRQ_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* One group of g float values through n_stages 2-bit stages.
 *   x      [g]               input values (any finite binary32)
 *   Q      [n_stages][g]     unpacked codes 0..3 (output)
 *   scale  [n_stages]        per-stage scale s_k (output)
 *   zero   [n_stages]        per-stage offset m_k = group minimum (output)
 *   resid  [n_stages][g]     residual after each stage (output, may be NULL)
 * Returns 0, or -1 on a bad argument (g < 1, n_stages < 1). */
int rrq_oracle_quantize_group(const float* x, int g, int n_stages, uint8_t* Q,
                              float* scale, float* zero, float* resid);

/* A row-major bf16 matrix [rows, cols] (raw bf16 bit patterns), groups of
 * `group` consecutive columns.  Outputs, for each stage k < n_stages:
 *   codes[k]  uint8 [rows*cols/4]: element c at byte c/4, bits 2*(c%4)..+1
 *   scales[k] float [rows*cols/group]
 *   zeros[k]  float [rows*cols/group]
 * Returns 0, or -1 on a bad argument (cols % group != 0, group < 1, ...). */
int rrq_oracle_quantize(const uint16_t* W, int64_t rows, int64_t cols, int group,
                        int n_stages, uint8_t* const* codes, float* const* scales,
                        float* const* zeros);

/* Prefix reconstruction with the first k stages (k = 1 is the 2-bit base),
 * written as bf16 bit patterns [rows*cols].  Returns 0 or -1. */
int rrq_oracle_reconstruct(const uint8_t* const* codes, const float* const* scales,
                           const float* const* zeros, int64_t rows, int64_t cols,
                           int group, int k, uint16_t* out);

/* Symmetric grid (levels (Q-2)*s, s = 2*max|x|/3, no zero stored; see
 * rrq_oracle.c).  scale_f16 != 0 rounds each scale to binary16 and
 * quantizes against the rounded value.
 *   scale  [n_stages]  the scale each stage used (a binary16 value when
 *                      scale_f16), as binary32 */
int rrq_oracle_quantize_group_sym(const float* x, int g, int n_stages, int scale_f16,
                                  uint8_t* Q, float* scale, float* resid);

/* Matrix form of the symmetric grid: codes[k] as for rrq_oracle_quantize;
 * scales[k] is float[rows*cols/group], or uint16_t binary16 bit patterns
 * when scale_f16. */
int rrq_oracle_quantize_sym(const uint16_t* W, int64_t rows, int64_t cols, int group,
                            int n_stages, int scale_f16, uint8_t* const* codes,
                            void* const* scales);

/* Prefix-k reconstruction of a symmetric package:
 * acc = (Q_0 - 2) s_0; acc = fl(acc + (Q_i - 2) s_i); bf16. */
int rrq_oracle_reconstruct_sym(const uint8_t* const* codes, const void* const* scales,
                               int64_t rows, int64_t cols, int group, int k, int scale_f16,
                               uint16_t* out);

/* Algorithm 1 with a base checkpoint: codes[0], scales[0] (and zeros[0] for
 * the asymmetric grid) are inputs holding stage 0 in the package's format;
 * stages 1..n_stages-1 are written (n_stages >= 2).  grid_sym selects the
 * symmetric grid (zeros unused, may be NULL); scale_f16 requires grid_sym. */
int rrq_oracle_quantize_from_base(const uint16_t* W, int64_t rows, int64_t cols, int group,
                                  int n_stages, int grid_sym, int scale_f16,
                                  uint8_t* const* codes, void* const* scales,
                                  float* const* zeros);

/* Product of activations with the prefix-k weights (Appendix C):
 * Y[b][r] = sum_c W~[r][c] * A[b][c] in binary64, W~ = the binary32 stage sum
 * of the first k stages (the reconstruction before bf16 rounding).
 *   A  bf16 bit patterns [batch][cols];  Y  double [batch][rows]. */
int rrq_oracle_gemv(const uint8_t* const* codes, const void* const* scales,
                    const float* const* zeros, int64_t rows, int64_t cols, int group, int k,
                    int grid_sym, int scale_f16, const uint16_t* A, int batch, double* Y);

/* Product of many activation rows with the prefix-k weights, the prefill
 * form of Appendix C's stage-wise product with bf16 operands (as a tensor-core
 * GEMM takes them): Y[t][r] = sum_c bf16(W~[r][c]) * A[t][c] in binary64,
 * bf16(W~) = the prefix-k reconstruction (the binary32 stage sum rounded to
 * nearest-even bf16), each product of two bf16 values exact in binary64.
 *   A  bf16 bit patterns [tokens][cols];  Y  double [tokens][rows]. */
int rrq_oracle_prefill(const uint8_t* const* codes, const void* const* scales,
                       const float* const* zeros, int64_t rows, int64_t cols, int group, int k,
                       int grid_sym, int scale_f16, const uint16_t* A, int64_t tokens, double* Y);

/* Products (decode form with binary32 weights, prefill form with bf16
 * weights when bf16_weights != 0) with the prefix-k weights of a package with
 * per-stage widths bits[i] in 1..4 (asymmetric grid):
 * Y[t][r] = sum_c w(r, c) A[t][c] in binary64.
 *   A  bf16 bit patterns [tokens][cols];  Y  double [tokens][rows]. */
int rrq_oracle_product_bits(const uint8_t* const* codes, const float* const* scales,
                            const float* const* zeros, int64_t rows, int64_t cols, int group, int k,
                            const int* bits, const uint16_t* A, int64_t tokens, int bf16_weights,
                            double* Y);

/* Algorithm 1 with a base checkpoint for a package with per-stage widths
 * (asymmetric grid): stage 0 given in codes[0] (bits[0] bits per weight,
 * LSB-first), scales[0], zeros[0]; stages 1..n_stages-1 are written. */
int rrq_oracle_quantize_from_base_bits(const uint16_t* W, int64_t rows, int64_t cols, int group,
                                       int n_stages, const int* bits, uint8_t* const* codes,
                                       float* const* scales, float* const* zeros);

/* Asymmetric stages with per-stage widths bits[k] in 1..4 (2^b levels,
 * 2^b - 1 steps).  Group form as rrq_oracle_quantize_group; matrix form packs
 * stage k's codes LSB-first, element c at bits bits[k]*c.., into
 * codes[k] (rows*cols*bits[k]/8 bytes). */
int rrq_oracle_quantize_group_bits(const float* x, int g, int n_stages, const int* bits,
                                   uint8_t* Q, float* scale, float* zero, float* resid);
int rrq_oracle_quantize_bits(const uint16_t* W, int64_t rows, int64_t cols, int group,
                             int n_stages, const int* bits, uint8_t* const* codes,
                             float* const* scales, float* const* zeros);
int rrq_oracle_reconstruct_bits(const uint8_t* const* codes, const float* const* scales,
                                const float* const* zeros, int64_t rows, int64_t cols, int group,
                                int k, const int* bits, uint16_t* out);

/* Per-group peak-to-mean ratio max|x| / (sum|x| / g) of a bf16 matrix, in
 * binary64 (0 for an all-zero group): pmr[rows*cols/group]. */
int rrq_oracle_group_pmr(const uint16_t* W, int64_t rows, int64_t cols, int group, double* pmr);

/* The scalar conversions the oracle uses, exported for tests. */
float rrq_oracle_bf16_to_f32(uint16_t h);
uint16_t rrq_oracle_f32_to_bf16(float f);
uint16_t rrq_oracle_f32_to_f16(float f);
float rrq_oracle_f16_to_f32(uint16_t h);

#ifdef __cplusplus
}
#endif

#endif
