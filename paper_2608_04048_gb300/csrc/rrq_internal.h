// Host/device interface between the RRQ C-ABI layer (abi.cu) and the kernel
// translation units (quantize.cu, reconstruct.cu).  Not part of the public
// ABI; the public declarations are in include/rrq.h.
#pragma once

#include <cstdint>
#include <cuda.h>  // CUtensorMap (the type only; no driver call is linked)
#include <cuda_runtime.h>

namespace rrq {

constexpr int kMaxStages = 4;
constexpr int kLaneElems = 32;                    // weights owned by one lane per chunk
constexpr int kChunkElems = 32 * kLaneElems;      // weights per warp chunk (1024)
constexpr int kChunkBytes = kChunkElems * 2;      // bf16 bytes per warp chunk (2 KiB)
constexpr int kMaxBatch = 64;                     // matrices per kernel launch (kernel parameters)

// Package formats built by the kernels (grid x scale type of include/rrq.h).
enum Format : int {
  kAsymF32 = 0,  // zero = group minimum, binary32 scale and zero
  kSymF32 = 1,   // implicit zero-point 2, binary32 scale
  kSymF16 = 2,   // implicit zero-point 2, binary16 scale
  kAsymBits = 3, // zero = group minimum, binary32 scale and zero, per-stage widths 1..4
};

constexpr unsigned kStatusTimeout = 1u;           // bit set in the device status word
constexpr uint32_t kDebugForceExact = 1u;         // same value as RRQ_DEBUG_FORCE_EXACT
constexpr uint32_t kDrainLimitUs = 1000000u;      // wait for own copies before leaving

// One matrix of a quantize launch.  Chunks of all matrices of a launch are
// numbered consecutively; chunk_begin is this matrix's first chunk.
struct QuantizeItem {
  const uint16_t* W;               // bf16 bits, n elements
  int64_t n;                       // rows * cols (multiple of 32)
  int64_t chunk_begin;
  uint8_t* codes[kMaxStages];      // n/4 bytes each
  void* scales[kMaxStages];        // n/group float or binary16 each
  float* zeros[kMaxStages];        // n/group each (asymmetric grid only)
  uint16_t* out[kMaxStages];       // bf16 prefix after each stage (build with prefixes only)
};

struct QuantizeBatch {
  int count;                       // 1..kMaxBatch
  int n_stages;                    // 1..4
  int bits[kMaxStages];            // code width per stage (kAsymBits), else 2
  uint32_t wait_limit_us;
  uint32_t flags;                  // kDebugForceExact
  unsigned* status;                // device status word
  int64_t total_chunks;
  QuantizeItem item[kMaxBatch];
};

// The wide-lane build (quantize_tile_kernel.cuh): the launch's matrices as
// 2-D tensor maps [n / LW, LW] of bf16 (one 32-row box = one warp chunk of
// 32 * LW weights), and the batch with chunk_begin / total_chunks counted in
// those chunks.
struct QuantizeTileBatch {
  CUtensorMap w[kMaxBatch];
  QuantizeBatch b;
};

// Encodes W (n bf16 weights, n % lw == 0, n / lw < 2^31) as the 2-D tensor
// map [n / lw, lw] with 32-row boxes and the 128-byte (lw = 64) or 64-byte
// (lw = 32) swizzle; false if the driver's encoder is unavailable or rejects
// it.
bool encode_lane_tiles(CUtensorMap* map, const uint16_t* W, int64_t n, int lw);

struct ReconstructItem {
  const uint8_t* codes[kMaxStages];
  const void* scales[kMaxStages];  // float or binary16
  const float* zeros[kMaxStages];  // asymmetric grid only
  uint16_t* out[kMaxStages];       // bf16 bits, n elements; out[0] only unless all prefixes
  int64_t n;
  int64_t chunk_begin;
};

struct ReconstructBatch {
  int count;
  int bits[kMaxStages];            // code width per stage (kAsymBits), else 2
  uint32_t wait_limit_us;
  unsigned* status;                // device status word
  int64_t total_chunks;
  ReconstructItem item[kMaxBatch];
};

// One matrix of a stage-wise product launch: Y = A * W~^T with W~ the prefix
// weights of the package's first k stages.  Each matrix's rows are cut into
// blocks of 16; the blocks of all matrices of a launch are numbered
// consecutively and blk_begin is this matrix's first.
// The wide-lane reconstruction at one prefix (reconstruct_tile_kernel.cuh):
// each matrix's bf16 output as the 2-D tensor map [n / 64, 64] (one 32-row
// box = one warp chunk of 2048 weights), and the batch with chunk_begin /
// total_chunks counted in those chunks.
struct ReconstructTileBatch {
  CUtensorMap out[kMaxBatch];
  ReconstructBatch b;
};

struct GemvItem {
  const uint8_t* codes[kMaxStages];
  const void* scales[kMaxStages];  // float or binary16
  const float* zeros[kMaxStages];  // asymmetric grid only
  const uint16_t* A;               // bf16 [activation rows, cols] (this launch's first row)
  float* Y;                        // [activation rows, rows] (this launch's first row)
  int64_t rows, cols;
  int64_t blk_begin;
};

constexpr int kMaxGemvGrid = 512;  // CTAs of one launch

struct GemvBatch {
  int count;
  int log2g;                       // group = 1 << log2g
  int grid;                        // CTAs of the launch
  int bits[kMaxStages];            // per-stage code widths (kAsymBits)
  int64_t total_blocks;
  int64_t cta_begin[kMaxGemvGrid + 1];  // CTA c takes blocks [cta_begin[c], cta_begin[c+1])
  GemvItem item[kMaxBatch];
};

constexpr int kGemvRows = 16;      // rows per block

// Cuts the launch's blocks into `grid` contiguous ranges (one per CTA) with
// equal shares of rows x columns; sets p.grid and p.cta_begin.
inline void gemv_split(GemvBatch& p, int grid) {
  p.grid = grid;
  int64_t total = 0;
  for (int i = 0; i < p.count; ++i) total += p.item[i].rows * p.item[i].cols;
  int c = 0;
  int64_t done = 0, blk = 0;
  p.cta_begin[0] = 0;
  for (int i = 0; i < p.count && c < grid; ++i) {
    const GemvItem& it = p.item[i];
    const int64_t nblk = (it.rows + kGemvRows - 1) / kGemvRows;
    for (int64_t b = 0; b < nblk; ++b, ++blk) {
      const int64_t r = it.rows - b * kGemvRows < kGemvRows ? it.rows - b * kGemvRows : kGemvRows;
      done += r * it.cols;
      // close CTA c's range once its share is reached
      while (c + 1 < grid && done * grid >= (c + 1) * total) p.cta_begin[++c] = blk + 1;
    }
  }
  while (c < grid) p.cta_begin[++c] = p.total_blocks;
  p.cta_begin[grid] = p.total_blocks;
}

constexpr int kMaxGemvBatch = 8;   // activation rows (tokens) per call

// One matrix of a prefill launch: Y = A bf16(W~)^T on the tensor cores, with
// bf16(W~) the prefix-k reconstruction formed from the package in the
// kernel.  A matrix is cut into tiles of kPrefillBM weight rows by
// kPrefillBN tokens.  `cluster` CTAs (1, 2 or 4) with the same row tile and
// consecutive token tiles form a cluster that shares the weight tiles (each
// forms 1/cluster of the rows); token tiles are padded to a multiple of
// `cluster`.  The tiles of all matrices of a launch are numbered
// consecutively (one CTA each, clusters in token-tile-major order: the CTAs
// that run together share activation tiles) and tile_begin is this matrix's
// first.
struct PrefillItem {
  const uint8_t* codes[kMaxStages];
  const void* scales[kMaxStages];  // float or binary16
  const float* zeros[kMaxStages];  // asymmetric grid only
  float* Y;                        // [tokens, rows]
  int64_t rows, cols;
  int64_t tile_begin;
  int32_t row_tiles;
};

constexpr int kPrefillBM = 128;       // weight rows per tile (TMEM lanes, MMA M)
constexpr int kPrefillMmaN = 256;     // tokens per MMA (MMA N; also the activation box)
constexpr int kPrefillBN = 512;       // tokens per tile: two accumulators, all 512 TMEM columns
constexpr int kPrefillBK = 64;        // columns per pipeline stage (one 128-byte swizzle row)
constexpr int kMaxPrefillBatch = 16;  // matrices per launch

struct PrefillBatch {  // (64-byte aligned through its tensor maps)
  CUtensorMap act[kMaxPrefillBatch];  // activations [tokens, cols] bf16: box 64 x kPrefillMmaN, 128-byte swizzle
  // codes of stage i [rows, cols/4] bytes: box 16 x (kPrefillBM / cluster)
  // (the codes of one 64-column stage of a CTA's share of a row tile); used
  // when codes_tma != 0
  CUtensorMap codes[kMaxPrefillBatch][kMaxStages];
  PrefillItem item[kMaxPrefillBatch];
  int cluster;                        // CTAs per cluster (1, 2, 4; 1 with per-stage widths)
  int bits[kMaxStages];               // per-stage code widths (kAsymBits)
  int codes_tma;                      // every matrix has cols % 64 == 0
  int scale_blocks;                   // every matrix has 16-byte rows of scales (and zeros)
  int count;
  int log2g;                          // group = 1 << log2g
  int64_t tokens;
  int64_t total_tiles;
  uint32_t wait_limit_us;
  unsigned* status;
};

cudaError_t prefill_launch_asym_f32(int k, const PrefillBatch& p, cudaStream_t stream);
cudaError_t prefill_launch_sym_f32(int k, const PrefillBatch& p, cudaStream_t stream);
cudaError_t prefill_launch_sym_f16(int k, const PrefillBatch& p, cudaStream_t stream);
cudaError_t prefill_launch_asym_bits(int k, const PrefillBatch& p, cudaStream_t stream);

inline cudaError_t prefill_launch(Format fmt, int k, const PrefillBatch& p, cudaStream_t stream) {
  switch (fmt) {
    case kAsymF32: return prefill_launch_asym_f32(k, p, stream);
    case kSymF32: return prefill_launch_sym_f32(k, p, stream);
    case kSymF16: return prefill_launch_sym_f16(k, p, stream);
    case kAsymBits: return prefill_launch_asym_bits(k, p, stream);
    default: return cudaErrorInvalidValue;
  }
}

// One matrix of a group peak-to-mean ratio launch.
struct PmrItem {
  const uint16_t* W;               // bf16, n elements
  float* pmr;                      // n/group
  float* stats;                    // [2] max and mean over the groups, or null
  int64_t n;
  int64_t chunk_begin;
};

struct PmrBatch {
  int count;
  int group;
  int64_t total_chunks;
  PmrItem item[kMaxBatch];
};

cudaError_t pmr_launch(int group, const PmrBatch& p, cudaStream_t stream, int sms);

// One-time per-device set-up of kernel attributes (dynamic shared memory).
cudaError_t quantize_prepare();
cudaError_t quantize_prepare_base();
cudaError_t quantize_prepare_emit();
cudaError_t reconstruct_prepare_asym_f32();
cudaError_t reconstruct_prepare_sym_f32();
cudaError_t reconstruct_prepare_sym_f16();
cudaError_t reconstruct_prepare_asym_bits();

// Launch on `stream`; `sms` = multiprocessor count of the current device.
cudaError_t quantize_launch(int group, Format fmt, const QuantizeBatch& p, cudaStream_t stream, int sms);
// Stage 0 given (item codes[0], scales[0], zeros[0] are inputs); stages
// 1..n_stages-1 computed.
cudaError_t quantize_launch_base(int group, Format fmt, const QuantizeBatch& p, cudaStream_t stream,
                                 int sms);
// Every stage computed, and the bf16 reconstruction after stage k written to
// item out[k].
cudaError_t quantize_launch_emit(int group, Format fmt, const QuantizeBatch& p, cudaStream_t stream,
                                 int sms);
// all_prefixes: write prefixes 1..k to out[0..k-1] (else prefix k to out[0]).
// One translation unit per format (they compile in parallel).
cudaError_t reconstruct_launch_asym_f32(int group, int k, bool all_prefixes, const ReconstructBatch& p,
                                        cudaStream_t stream, int sms);
cudaError_t reconstruct_launch_sym_f32(int group, int k, bool all_prefixes, const ReconstructBatch& p,
                                       cudaStream_t stream, int sms);
cudaError_t reconstruct_launch_sym_f16(int group, int k, bool all_prefixes, const ReconstructBatch& p,
                                       cudaStream_t stream, int sms);
cudaError_t reconstruct_launch_asym_bits(int group, int k, bool all_prefixes, const ReconstructBatch& p,
                                         cudaStream_t stream, int sms);

// Activation rows one launch can hold in shared memory for matrices of up to
// max_cols columns with k stages and groups of `group` (0: too wide).
int gemv_rows_per_launch(Format fmt, int k, int64_t max_cols, int group);
// nb activation rows (1..kMaxGemvBatch, within gemv_rows_per_launch); one
// translation unit per format.
cudaError_t gemv_launch_asym_f32(int k, int nb, int64_t max_cols, GemvBatch& p, cudaStream_t stream, int sms);
cudaError_t gemv_launch_sym_f32(int k, int nb, int64_t max_cols, GemvBatch& p, cudaStream_t stream, int sms);
cudaError_t gemv_launch_sym_f16(int k, int nb, int64_t max_cols, GemvBatch& p, cudaStream_t stream, int sms);
cudaError_t gemv_launch_asym_bits(int k, int nb, int64_t max_cols, GemvBatch& p, cudaStream_t stream, int sms);

// Once per device: the decode product's kernels may take the shared memory
// their largest launch needs.
// the tensor-core form (groups of 64 and more, 2-bit stages), one unit per format
cudaError_t gemv_mma_launch_asym_f32(int group, int k, int nb, int64_t max_cols, GemvBatch& p, cudaStream_t stream,
                                     int sms);
cudaError_t gemv_mma_launch_sym_f32(int group, int k, int nb, int64_t max_cols, GemvBatch& p, cudaStream_t stream,
                                    int sms);
cudaError_t gemv_mma_launch_sym_f16(int group, int k, int nb, int64_t max_cols, GemvBatch& p, cudaStream_t stream,
                                    int sms);
cudaError_t gemv_mma_prepare_asym_f32();
cudaError_t gemv_mma_prepare_sym_f32();
cudaError_t gemv_mma_prepare_sym_f16();
cudaError_t gemv_prepare_asym_f32();
cudaError_t gemv_prepare_sym_f32();
cudaError_t gemv_prepare_sym_f16();
cudaError_t gemv_prepare_asym_bits();

inline cudaError_t gemv_prepare() {
  cudaError_t e;
  if ((e = gemv_prepare_asym_f32())) return e;
  if ((e = gemv_prepare_sym_f32())) return e;
  if ((e = gemv_prepare_sym_f16())) return e;
  return gemv_prepare_asym_bits();
}

inline cudaError_t gemv_launch(Format fmt, int k, int nb, int64_t max_cols, GemvBatch& p,
                               cudaStream_t stream, int sms) {
  switch (fmt) {
    case kAsymF32: return gemv_launch_asym_f32(k, nb, max_cols, p, stream, sms);
    case kSymF32: return gemv_launch_sym_f32(k, nb, max_cols, p, stream, sms);
    case kSymF16: return gemv_launch_sym_f16(k, nb, max_cols, p, stream, sms);
    case kAsymBits: return gemv_launch_asym_bits(k, nb, max_cols, p, stream, sms);
  }
  return cudaErrorInvalidValue;
}

inline cudaError_t reconstruct_prepare() {
  cudaError_t e;
  if ((e = reconstruct_prepare_asym_f32())) return e;
  if ((e = reconstruct_prepare_sym_f32())) return e;
  if ((e = reconstruct_prepare_sym_f16())) return e;
  return reconstruct_prepare_asym_bits();
}

inline cudaError_t reconstruct_launch(int group, Format fmt, int k, bool all_prefixes,
                                      const ReconstructBatch& p, cudaStream_t stream, int sms) {
  switch (fmt) {
    case kAsymF32: return reconstruct_launch_asym_f32(group, k, all_prefixes, p, stream, sms);
    case kSymF32: return reconstruct_launch_sym_f32(group, k, all_prefixes, p, stream, sms);
    case kSymF16: return reconstruct_launch_sym_f16(group, k, all_prefixes, p, stream, sms);
    case kAsymBits: return reconstruct_launch_asym_bits(group, k, all_prefixes, p, stream, sms);
  }
  return cudaErrorInvalidValue;
}

}  // namespace rrq
