/*
 * rrq.h -- C ABI of the GB300 (sm_103a) Recurrent Residual Quantization
 * library: construction of the 2/4/6/8-bit RRQ package from bf16 weights and
 * prefix reconstruction of bf16 weights from it.
 *
 * The operation (paper: "Recurrent Residual Quantization", Section 3):
 *   - Section 3.1, Eq. 1-3: a group of consecutive weights shares a scale s
 *     and zero-point; each weight gets an integer code Q, and the residual is
 *     the weight minus its dequantized value.
 *   - Section 3.2, Eq. 4-7 and Algorithm 1: the base stage quantizes W; each
 *     of the following stages quantizes the running residual of the previous
 *     one and subtracts its dequantized value.  With four 2-bit stages the
 *     package serves the 2-, 4-, 6- and 8-bit operating points.
 *   - Section 3.2, Eq. 8 (and Appendix C): the weight at prefix t is the
 *     base plus the first t residual stages.
 *   - Section 5.1: 2-bit round-to-nearest stages, group size 128.
 *
 * Arithmetic (identical, bit for bit, to the definition below; every step
 * is one IEEE-754 binary32 operation rounded to nearest-even, no fused
 * multiply-add, subnormals kept):
 *     lo = min(v), hi = max(v) over the group, ordering -0 before +0
 *     s  = fl(fl(hi - lo) / 3)                       3 = 2^2 - 1 steps
 *     Q  = s == 0 ? 0 : clamp(rhe(fl(fl(v - lo) / s)), 0, 3)
 *     L  = fl(lo + fl(Q * s))                        dequantized value
 *     v' = fl(v - L)                                 running residual
 *   v starts as the bf16 weight widened to binary32; rhe = round half to
 *   even.  The stored zero of a stage is lo (the real offset m = -z*s).
 *   Reconstruction with k stages: acc = L_0; acc = fl(acc + L_i) for
 *   i = 1..k-1; output = bf16 round-to-nearest-even of acc.
 *
 * Layout (all buffers are caller-owned device memory of the current device):
 *   W         bf16 [rows, cols] row-major; a group is `group` consecutive
 *             elements of a row, so the flattened group index of element
 *             c = r*cols + j is c / group.
 *   codes[k]  uint8 [rows*cols/4] for stage k: element c is at byte c/4,
 *             bits 2*(c%4) and 2*(c%4)+1 (least significant first).
 *   scales[k] float [rows*cols/group], zeros[k] float [rows*cols/group].
 *
 * Calls are asynchronous on `stream` (a cudaStream_t; NULL = the legacy
 * default stream).  Outputs are valid once the stream reaches the call.  The
 * library never allocates, frees or synchronizes in these calls; only
 * rrq_get_device_status synchronizes.  A bad argument returns an error code
 * synchronously and launches nothing.  A call that makes several launches
 * (batches beyond one launch's matrices, decode products split over
 * activation rows) and meets RRQ_ERR_CUDA after its first launch may leave
 * its outputs partly written.  Functions are thread-safe.
 */
#ifndef RRQ_H
#define RRQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

struct CUstream_st;                        /* cudaStream_t is struct CUstream_st* */
typedef struct CUstream_st* rrq_stream_t;

typedef enum {
  RRQ_OK = 0,
  RRQ_ERR_INVALID_ARG = 1, /* null pointer, non-positive size, cols % group != 0,
                              n_stages or k out of range, pointer not device memory
                              of the current device, aliasing outputs */
  RRQ_ERR_UNSUPPORTED = 2, /* group not in {32, 64, 128, 256}, or a format
                              combination the library does not build */
  RRQ_ERR_MISALIGNED = 3,  /* a pointer breaks the alignment stated below */
  RRQ_ERR_CUDA = 4,        /* a CUDA runtime call or kernel launch failed; see
                              rrq_last_cuda_error() */
  RRQ_ERR_TIMEOUT = 5      /* a kernel gave up waiting for its own data copies
                              (reported by rrq_get_device_status) */
} rrq_status;

#define RRQ_MAX_STAGES 4

/* Build the RRQ package of one bf16 weight matrix (Algorithm 1 without a base
 * checkpoint; Eq. 1-7).
 *   W_bf16      device, bf16 bit patterns [rows, cols], 16-byte aligned; read only.
 *   rows, cols  >= 1; cols % group == 0; rows*cols < 2^40.
 *   group       32, 64, 128 or 256 (the paper uses 128).
 *   n_stages    1..4: stage 0 is the 2-bit base, stages 1..n_stages-1 are
 *               2-bit residual stages.
 *   out_codes   host array of n_stages device pointers, each to
 *               rrq_codes_bytes(rows, cols) bytes, 16-byte aligned.
 *   out_scales, out_zeros
 *               host arrays of n_stages device pointers, each to
 *               rrq_meta_count(rows, cols, group) floats, 16-byte aligned.
 * No output may overlap another output or W.  One fused kernel computes all
 * stages; the running residual never leaves registers. */
rrq_status rrq_quantize(const uint16_t* W_bf16, int64_t rows, int64_t cols, int group,
                        int n_stages, uint8_t* const out_codes[],
                        float* const out_scales[], float* const out_zeros[],
                        rrq_stream_t stream);

/* Prefix reconstruction with the first k stages (Eq. 8; Appendix C):
 * k = 1, 2, 3, 4 give the 2-, 4-, 6-, 8-bit operating points.
 *   codes, scales, zeros  host arrays of >= k device pointers laid out as
 *                         written by rrq_quantize (16-byte aligned; the
 *                         kernel copies whole chunks with bulk copies).
 *   rows, cols, group     as given to rrq_quantize.
 *   k                     1..4.
 *   out_bf16              device, bf16 bit patterns [rows, cols], 16-byte
 *                         aligned, not overlapping any input. */
rrq_status rrq_reconstruct(const uint8_t* const codes[], const float* const scales[],
                           const float* const zeros[], int64_t rows, int64_t cols,
                           int group, int k, uint16_t* out_bf16, rrq_stream_t stream);

/* One matrix of rrq_quantize_batch: the arguments of rrq_quantize for it. */
typedef struct {
  const uint16_t* W_bf16;                /* device, bf16 [rows, cols], 16-byte aligned */
  int64_t rows, cols;                    /* cols % group == 0 */
  uint8_t* codes[RRQ_MAX_STAGES];        /* first n_stages entries used */
  float* scales[RRQ_MAX_STAGES];
  float* zeros[RRQ_MAX_STAGES];
} rrq_quantize_item;

/* rrq_quantize for `count` matrices (count >= 1) that share `group` and
 * `n_stages`: the same result as count separate calls, computed by one kernel
 * launch per 64 matrices whose warps take the chunks of all of them in turn
 * (no launch gaps, balanced across small and large matrices).  `items` is a
 * host array, read during the call only.  Every rule of rrq_quantize holds per
 * matrix; in addition no output may overlap any input or output of another
 * matrix of the batch.  The library allocates nothing: the matrix
 * descriptors travel in the kernel parameters. */
rrq_status rrq_quantize_batch(const rrq_quantize_item* items, int count, int group,
                              int n_stages, rrq_stream_t stream);

/* One matrix of rrq_reconstruct_batch. */
typedef struct {
  const uint8_t* codes[RRQ_MAX_STAGES];  /* first k entries used */
  const float* scales[RRQ_MAX_STAGES];
  const float* zeros[RRQ_MAX_STAGES];
  int64_t rows, cols;
  uint16_t* out_bf16;                    /* device, bf16 [rows, cols], 16-byte aligned */
} rrq_reconstruct_item;

/* rrq_reconstruct at prefix k for `count` matrices sharing `group`, one kernel
 * launch per 64 matrices; outputs may not overlap any input or output of the
 * batch. */
rrq_status rrq_reconstruct_batch(const rrq_reconstruct_item* items, int count, int group, int k,
                                 rrq_stream_t stream);

/* All prefixes at once (Eq. 8 for t = 0..k-1; Appendix C): one pass over the
 * first k stages writes the reconstruction after every stage, out_bf16[j]
 * receiving the prefix with j+1 stages (the 2-, 4-, 6-, 8-bit weights for
 * k = 4).  Bit-identical to k separate rrq_reconstruct calls with k = 1..j+1,
 * reading the package once instead of k times.  out_bf16 is a host array of
 * k device pointers (16-byte aligned, not overlapping each other or any
 * input). */
rrq_status rrq_reconstruct_prefixes(const uint8_t* const codes[], const float* const scales[],
                                    const float* const zeros[], int64_t rows, int64_t cols,
                                    int group, int k, uint16_t* const out_bf16[],
                                    rrq_stream_t stream);

/* One matrix of rrq_reconstruct_prefixes_batch. */
typedef struct {
  const uint8_t* codes[RRQ_MAX_STAGES];  /* first k entries used */
  const float* scales[RRQ_MAX_STAGES];
  const float* zeros[RRQ_MAX_STAGES];
  int64_t rows, cols;
  uint16_t* out_bf16[RRQ_MAX_STAGES];    /* out_bf16[j]: prefix with j+1 stages */
} rrq_prefixes_item;

/* rrq_reconstruct_prefixes for `count` matrices sharing `group` and `k`, one
 * kernel launch per 64 matrices. */
rrq_status rrq_reconstruct_prefixes_batch(const rrq_prefixes_item* items, int count, int group,
                                          int k, rrq_stream_t stream);

/* ------------------------------------------------------------------------
 * Package formats.  The calls above build and read the asymmetric package
 * with binary32 scales and zeros.  The format-generic calls below also build
 * and read the symmetric package, the paper's timed and stored
 * configuration ("symmetric" quantization type, Table 4; no stored
 * zero-points and a 16-bit scale per group of 128, Appendix G).
 *
 * Symmetric grid (RRQ_GRID_SYM), per group and stage (bit for bit; binary32
 * steps rounded to nearest-even):
 *     amax = max |v| over the group
 *     s    = fl(fl(2 * amax) / 3)          amax sits 1.5 steps from 0
 *     s    = binary16_rne(s)               only with RRQ_SCALE_F16: the stage
 *                                          quantizes against the stored scale
 *     Q    = s == 0 ? 2 : clamp(rhe(fl(v / s)) + 2, 0, 3)
 *     L    = (Q - 2) * s                   levels -2s, -s, 0, s (exact)
 *     v'   = fl(v - L)
 *   The zero-point is the implicit constant 2 (Eq. 1-3 with z = 2): nothing
 *   is stored for it.  Reconstruction: acc = L_0; acc = fl(acc + L_i);
 *   bf16 round-to-nearest-even.  Inputs need 2 * max|W| finite; with
 *   RRQ_SCALE_F16 also max|W| < 98,000 (the scale must stay finite in
 *   binary16), otherwise the results are unspecified.
 * ------------------------------------------------------------------------ */
typedef enum {
  RRQ_GRID_ASYM = 0, /* zero = group minimum, levels lo + Q*s (the calls above) */
  RRQ_GRID_SYM = 1   /* implicit zero-point 2, levels (Q - 2)*s, no zeros stored */
} rrq_grid;

typedef enum {
  RRQ_SCALE_F32 = 0, /* IEEE binary32 scale, 4 bytes per group and stage */
  RRQ_SCALE_F16 = 1  /* IEEE binary16 scale, 2 bytes per group and stage
                        (RRQ_GRID_SYM only) */
} rrq_scale_type;

typedef struct {
  int group;      /* 32, 64, 128 or 256 */
  int n_stages;   /* 1..4 stages held by the package */
  int grid;       /* rrq_grid */
  int scale_type; /* rrq_scale_type */
  int bits[RRQ_MAX_STAGES]; /* code width of each stage, 1..4 (0 = 2); see below */
} rrq_format;

/* Heterogeneous stage widths (Section 3.2: stage k may have its own width
 * b_k, the operating point after t stages is b_0 + ... + b_t bits; Table 3
 * compares 1+3, 2+2 and 3+1 splits).  A stage of width b on the asymmetric
 * grid has 2^b levels and m = 2^b - 1 steps:
 *     s = fl(fl(hi - lo) / m),  Q = s == 0 ? 0 : clamp(rhe(fl(fl(v - lo) / s)), 0, m),
 *     L = fl(lo + fl(Q * s)),   v' = fl(v - L)
 * (b = 2 is the grid above).  Stage k's codes are packed least significant
 * bit first, element c at bits b_k*c .. b_k*c + b_k - 1 of a byte array of
 * rows*cols*b_k/8 bytes (rrq_stage_codes_bytes).  Widths other than 2 are
 * supported with RRQ_GRID_ASYM and RRQ_SCALE_F32 by rrq_quantize_ex and
 * rrq_reconstruct_ex; other combinations and calls return
 * RRQ_ERR_UNSUPPORTED. */

/* One matrix of rrq_quantize_ex.  scales[k] points to float (RRQ_SCALE_F32)
 * or uint16_t binary16 bit patterns (RRQ_SCALE_F16), rrq_meta_count entries,
 * 16-byte aligned.  zeros[k] is used by RRQ_GRID_ASYM only (ignored, may be
 * NULL, for RRQ_GRID_SYM). */
typedef struct {
  const uint16_t* W_bf16;                /* device, bf16 [rows, cols], 16-byte aligned */
  int64_t rows, cols;                    /* cols % group == 0 */
  uint8_t* codes[RRQ_MAX_STAGES];        /* first n_stages entries used */
  void* scales[RRQ_MAX_STAGES];
  float* zeros[RRQ_MAX_STAGES];
} rrq_quantize_desc;

/* Build the packages of `count` matrices in format *fmt (Algorithm 1 without
 * a base checkpoint; Eq. 1-7).  Same rules as rrq_quantize_batch (one launch
 * per 64 matrices, no overlap between any output and any input or output of
 * the batch).  RRQ_ERR_UNSUPPORTED for a group outside {32, 64, 128, 256}
 * or RRQ_SCALE_F16 with RRQ_GRID_ASYM; RRQ_ERR_INVALID_ARG for an unknown
 * grid or scale type.  With RRQ_GRID_ASYM and RRQ_SCALE_F32 the result equals
 * rrq_quantize_batch's. */
rrq_status rrq_quantize_ex(const rrq_quantize_desc* items, int count, const rrq_format* fmt,
                           rrq_stream_t stream);

/* One matrix of rrq_quantize_prefixes: rrq_quantize_desc plus the outputs
 * for the reconstruction after every stage. */
typedef struct {
  const uint16_t* W_bf16;                /* device, bf16 [rows, cols], 16-byte aligned */
  int64_t rows, cols;
  uint8_t* codes[RRQ_MAX_STAGES];
  void* scales[RRQ_MAX_STAGES];
  float* zeros[RRQ_MAX_STAGES];          /* RRQ_GRID_ASYM only */
  uint16_t* out_bf16[RRQ_MAX_STAGES];    /* out_bf16[j]: prefix with j+1 stages, bf16 [rows, cols],
                                            16-byte aligned; first n_stages entries used */
} rrq_quantize_prefixes_desc;

/* Build the package and its reconstructions in one pass (Algorithm 1 without
 * a base checkpoint with Eq. 8 at every prefix): the same package as
 * rrq_quantize_ex, and out_bf16[j] the same bits as rrq_reconstruct_ex at
 * prefix j+1 on it -- the stage levels the construction computes are the
 * values the reconstruction sums, so the 2/4/6/8-bit weights come with the
 * package from one read of W (11.25 B per weight moved at group 128 with 4
 * stages, against 12.5 B for the two calls).  Formats: any with 2-bit
 * stages.  No output may overlap any input or output of the batch. */
rrq_status rrq_quantize_prefixes(const rrq_quantize_prefixes_desc* items, int count,
                                 const rrq_format* fmt, rrq_stream_t stream);

/* Algorithm 1 with a base checkpoint (Section 3.2: the construction can start
 * from an existing low-bit checkpoint by skipping the base quantization):
 * stage 0 of every item's package is an INPUT in format *fmt -- codes[0],
 * scales[0] and, for RRQ_GRID_ASYM, zeros[0] (a checkpoint from any
 * quantizer at the width fmt->bits[0], stored in this layout) -- dequantized
 * with the grid's level
 * formula (lo + Q*s, or (Q - 2)*s); the running residual starts at
 * R_0 = fl(W - L_0) and stages 1..n_stages-1 are computed from it exactly as
 * rrq_quantize_ex computes them from its own stage 0 (given the base that
 * rrq_quantize_ex would compute, the results are identical).
 * fmt->n_stages >= 2.  The stage-0 arrays are read only; they may overlap
 * other inputs but no output.  Other rules as for rrq_quantize_ex. */
rrq_status rrq_quantize_from_base(const rrq_quantize_desc* items, int count, const rrq_format* fmt,
                                  rrq_stream_t stream);

/* One matrix of rrq_reconstruct_ex: the package (first k stages) and the
 * outputs, out_bf16[0] only, or out_bf16[0..k-1] when all prefixes are
 * requested (out_bf16[j] = prefix with j+1 stages). */
typedef struct {
  const uint8_t* codes[RRQ_MAX_STAGES];
  const void* scales[RRQ_MAX_STAGES];    /* float or binary16, as in rrq_quantize_desc */
  const float* zeros[RRQ_MAX_STAGES];    /* RRQ_GRID_ASYM only */
  int64_t rows, cols;
  uint16_t* out_bf16[RRQ_MAX_STAGES];    /* device, bf16 [rows, cols], 16-byte aligned */
} rrq_reconstruct_desc;

/* Prefix reconstruction (Eq. 8; Appendix C) of `count` packages in format
 * *fmt: the prefix with k stages (all_prefixes == 0), or every prefix 1..k in
 * one pass over the package (all_prefixes != 0).  1 <= k <= fmt->n_stages.
 * Same rules as rrq_reconstruct_batch / rrq_reconstruct_prefixes_batch. */
rrq_status rrq_reconstruct_ex(const rrq_reconstruct_desc* items, int count, const rrq_format* fmt,
                              int k, int all_prefixes, rrq_stream_t stream);

/* One matrix of rrq_gemv: its package (first k stages, format of the call),
 * the activations and the output. */
typedef struct {
  const uint8_t* codes[RRQ_MAX_STAGES];
  const void* scales[RRQ_MAX_STAGES];    /* float or binary16 */
  const float* zeros[RRQ_MAX_STAGES];    /* RRQ_GRID_ASYM only */
  int64_t rows, cols;                    /* the weight matrix [rows, cols] */
  const uint16_t* A_bf16;                /* device, bf16 [batch, cols] row-major, 16-byte aligned */
  float* Y;                              /* device, float [batch, rows] row-major, 16-byte aligned */
} rrq_gemv_desc;

#define RRQ_MAX_GEMV_BATCH 8
#define RRQ_MAX_GEMV_COLS 57344

/* Product of activations with the prefix-k weights, without materialising
 * them (Appendix C: A W~_(t) = A W^_0 + sum_k A R^_k):
 *     Y[b][r] = sum_c W~[r][c] * A[b][c],   b < batch, r < rows
 * where W~[r][c] is the binary32 prefix sum of the first k stages (acc = L_0;
 * acc = fl(acc + L_i), the value rrq_reconstruct rounds to bf16).  The kernels
 * read only the package (k x (2 + 64/g) bits per weight for RRQ_GRID_ASYM,
 * k x (2 + 16/g) for the binary16 symmetric format) and sum in binary32 in a
 * fixed order (deterministic: two calls give the same bits).  Two forms:
 *   - groups of 64 and more with 2-bit stages: Appendix C's stage-wise form
 *     per group and stage, s D + lo S_g (s (D - 2 S_g) on the symmetric
 *     grid), D = sum Q a over the group's codes on the tensor cores and S_g
 *     = sum a; |Y - sum W~ a| <= d 2^-24 sum_c sum_k (|lo_k| + 3 s_k) |a_c|
 *     (2 s_k symmetric) with d = (k + 1) + g/16 + 8 + 2k (cols/g) + 18.
 *     The activations are held in shared memory as bf16 fragments, 2 bytes
 *     per column and row plus the group sums;
 *   - groups of 32 and per-stage widths (fmt->bits, asymmetric grid, with
 *     the reconstruction's stage sum of that format): the prefix weights
 *     formed per weight, |Y - exact| <= (64 ceil(cols/4096) + 8) 2^-24
 *     sum_c |W~ A|.  The activations are held in shared memory as binary32,
 *     padded to a multiple of 2048 columns (at most 4 rows at k = 4).
 * For decoding: 1 <= batch <= RRQ_MAX_GEMV_BATCH activation rows;
 * 1 <= k <= fmt->n_stages.  Y must not overlap any input or another Y.  A
 * launch takes as many of the batch's rows as fit in 227 KiB of shared
 * memory, so every matrix of a call may have at most RRQ_MAX_GEMV_COLS
 * columns (RRQ_ERR_UNSUPPORTED beyond, before anything is launched).
 * Matrices that take the same number of rows per launch are launched
 * together, up to 64 per launch, once per such share of the batch; other
 * rules as for rrq_reconstruct_ex. */
rrq_status rrq_gemv(const rrq_gemv_desc* items, int count, const rrq_format* fmt, int k, int batch,
                    rrq_stream_t stream);

#define RRQ_MAX_PREFILL_TOKENS (1 << 24)

/* Prefill form of the same product (Appendix C's stage-wise product for many
 * activation rows) on the tensor cores, without materialising the weights:
 *     Y[t][r] = sum_c bf16(W~)[r][c] * A[t][c],   t < tokens, r < rows
 * where bf16(W~) is the prefix-k reconstruction, bit for bit the values
 * rrq_reconstruct_ex returns (the tensor cores take bf16 operands).  The
 * kernel forms those weights from the package tile by tile in shared memory
 * and multiplies with tcgen05 MMAs, accumulating in binary32 (the order of
 * the partial sums is the hardware's; the result is deterministic).  The
 * items are rrq_gemv_desc with A_bf16 = [tokens, cols] and Y = float [tokens,
 * rows], both row-major and 16-byte aligned.  1 <= tokens <=
 * RRQ_MAX_PREFILL_TOKENS; 1 <= k <= fmt->n_stages.  Per-stage widths
 * (fmt->bits, asymmetric grid) are taken with the reconstruction's weights of
 * that format.  Y must not overlap any input or another Y.  One launch per 16
 * matrices; other rules as for rrq_reconstruct_ex. */
rrq_status rrq_prefill(const rrq_gemv_desc* items, int count, const rrq_format* fmt, int k, int64_t tokens,
                       rrq_stream_t stream);

/* One matrix of rrq_group_pmr. */
typedef struct {
  const uint16_t* W_bf16;  /* device, bf16 [rows, cols], 16-byte aligned */
  int64_t rows, cols;      /* cols % group == 0 */
  float* pmr;              /* device, float [rows*cols/group], 16-byte aligned */
  float* stats;            /* device, float [2]: max and mean of pmr over the
                              matrix's groups; NULL to skip */
} rrq_pmr_desc;

/* Group peak-to-mean ratio (Section 3.1; the group-maximum K/MAE of Table 9),
 * the outlier statistic for choosing a stage split (Section 3.3):
 *     pmr[g] = max |x| / (sum |x| / group) over group g (0 if all zero),
 * max |x| exact, the sum in binary32 (|pmr - exact| <= group * 2^-24 * pmr
 * to first order), and per matrix stats = {max_g pmr[g], mean_g pmr[g]}
 * (fixed-order reduction, deterministic).  Same rules as rrq_quantize_batch
 * for shapes, alignment, overlap and the stream. */
rrq_status rrq_group_pmr(const rrq_pmr_desc* items, int count, int group, rrq_stream_t stream);

/* Bytes of one stage's code array at width `bits` (1..4): rows*cols*bits/8.
 * 0 for invalid arguments. */
size_t rrq_stage_codes_bytes(int64_t rows, int64_t cols, int bits);

/* Bytes of one stage's scale array in format *fmt: groups * (4 or 2).
 * 0 for invalid arguments. */
size_t rrq_scales_bytes(int64_t rows, int64_t cols, const rrq_format* fmt);

/* Total package bytes in format *fmt: the sum over its stages of codes (at
 * the stage's width) + scales + zeros, zeros only for RRQ_GRID_ASYM.  0 for
 * invalid arguments. */
size_t rrq_package_bytes_ex(int64_t rows, int64_t cols, const rrq_format* fmt);

/* Bytes of one stage's code array: rows*cols/4 (rows*cols is a multiple of
 * 32 for every valid shape).  0 for invalid sizes. */
size_t rrq_codes_bytes(int64_t rows, int64_t cols);

/* Number of groups = entries of one stage's scale (and zero) array:
 * rows*cols/group.  0 for invalid sizes. */
size_t rrq_meta_count(int64_t rows, int64_t cols, int group);

/* Total package bytes for n_stages stages: n_stages * (codes + 8 * groups). */
size_t rrq_package_bytes(int64_t rows, int64_t cols, int group, int n_stages);

/* Synchronizes `stream`, then reads and clears the current device's status
 * word in one atomic exchange (a one-thread kernel on `stream`).  Returns
 * RRQ_ERR_TIMEOUT if a kernel on this device gave up on a bounded wait since
 * the last call (its outputs are then incomplete), RRQ_ERR_CUDA if the
 * synchronization or the exchange failed, RRQ_OK otherwise.  The word is
 * per device: kernels still running on other streams may set it after the
 * exchange, and the next call reports them. */
rrq_status rrq_get_device_status(rrq_stream_t stream);

/* Whether [p, p + bytes) lies in device memory of the current device (or
 * in managed memory): RRQ_OK if the driver reports every byte of it as part
 * of such allocations, RRQ_ERR_INVALID_ARG otherwise (a null, host, freed or
 * other device's pointer, or a length that runs past the allocation;
 * bytes == 0 checks the first byte).  Every entry point applies this check
 * to each of its buffers before launching anything.  Looks up the driver's
 * pointer attributes on every call (nothing is remembered between calls),
 * launches nothing and does not synchronize.  Paper: no counterpart (it is
 * the library's argument guard). */
rrq_status rrq_check_buffer(const void* p, size_t bytes);

/* Longest time a kernel waits for one of its own bulk copies before it
 * records RRQ_ERR_TIMEOUT and returns (default 1,000,000 us).  0 makes every
 * such wait give up at once; tests use it to exercise the error path.  The
 * setting is process-wide and applies to later launches. */
void rrq_set_wait_limit_us(uint32_t microseconds);

/* Test hook, process-wide: RRQ_DEBUG_FORCE_EXACT makes rrq_quantize take the
 * per-element IEEE-division path for every group instead of only for the
 * groups its check sends there; results are identical either way. */
#define RRQ_DEBUG_FORCE_EXACT 1u
void rrq_set_debug_flags(uint32_t flags);

/* Human-readable name of a status code (static storage). */
const char* rrq_status_string(rrq_status status);

/* The cudaError_t (as int) behind the calling thread's last RRQ_ERR_CUDA. */
int rrq_last_cuda_error(void);

#ifdef __cplusplus
}
#endif

#endif /* RRQ_H */
