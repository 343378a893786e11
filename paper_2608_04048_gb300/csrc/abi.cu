// C ABI of the RRQ library (declared in include/rrq.h): argument checks,
// per-device set-up and kernel launches.  Every check runs before anything is
// launched, so a rejected call has no effect on the device.
#include <algorithm>
#include <atomic>
#include <cstdint>
#include <cstring>
#include <map>
#include <mutex>
#include <vector>

#include <cuda_runtime.h>

#include "rrq.h"
#include "rrq_internal.h"

// Per-device status word: bit kStatusTimeout is set by a kernel that gave up
// on a bounded wait.  Read and cleared by rrq_get_device_status.
__device__ unsigned int rrq_device_status;
// The value rrq_get_device_status took out of the status word.
__device__ unsigned int rrq_device_status_taken;

// Reads and clears the status word in one atomic step, so that a bit set by
// a kernel on another stream in the meantime is kept for the next read.
__global__ void rrq_take_status_kernel() { rrq_device_status_taken = atomicExch(&rrq_device_status, 0u); }

namespace {

std::atomic<uint32_t> g_wait_limit_us{1000000u};
std::atomic<uint32_t> g_debug_flags{0u};
thread_local int t_last_cuda_error = 0;

struct DeviceState {
  bool ready = false;
  int sms = 0;
  unsigned* status = nullptr;  // device address of rrq_device_status
};
constexpr int kMaxDevices = 64;
std::mutex g_mu;
DeviceState g_devices[kMaxDevices];

rrq_status fail_cuda(cudaError_t e) {
  t_last_cuda_error = static_cast<int>(e);
  return RRQ_ERR_CUDA;
}

// Set-up of the current device, once: multiprocessor count, the device
// address of the status word, kernel attributes.
rrq_status current_device(int* dev_out, DeviceState** state) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail_cuda(e);
  if (dev < 0 || dev >= kMaxDevices) return RRQ_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_mu);
  DeviceState& d = g_devices[dev];
  if (!d.ready) {
    if ((e = cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, dev))) return fail_cuda(e);
    void* addr = nullptr;
    if ((e = cudaGetSymbolAddress(&addr, rrq_device_status))) return fail_cuda(e);
    d.status = static_cast<unsigned*>(addr);
    if ((e = rrq::quantize_prepare())) return fail_cuda(e);
    if ((e = rrq::quantize_prepare_base())) return fail_cuda(e);
    if ((e = rrq::quantize_prepare_emit())) return fail_cuda(e);
    if ((e = rrq::reconstruct_prepare())) return fail_cuda(e);
    if ((e = rrq::gemv_prepare())) return fail_cuda(e);
    d.ready = true;
  }
  *dev_out = dev;
  *state = &d;
  return RRQ_OK;
}

bool group_supported(int g) { return g == 32 || g == 64 || g == 128 || g == 256; }

bool shape_ok(int64_t rows, int64_t cols) {
  return rows >= 1 && cols >= 1 && rows < (int64_t(1) << 40) && cols < (int64_t(1) << 40) &&
         rows <= (int64_t(1) << 40) / cols;
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

// The driver's cuPointerGetAttributes, looked up once through the runtime
// (no link against the driver library).
using PointerAttrsFn = CUresult (*)(unsigned int, CUpointer_attribute*, void**, CUdeviceptr);

PointerAttrsFn pointer_attrs() {
  static PointerAttrsFn fn = [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuPointerGetAttributes", &ptr, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return static_cast<PointerAttrsFn>(nullptr);
    return reinterpret_cast<PointerAttrsFn>(ptr);
  }();
  return fn;
}

// Whether byte ranges lie in device memory of device `dev` (or in managed
// memory): every byte of [lo, hi) must belong to allocations the driver
// reports as such, walked allocation by allocation (a buffer may span
// several contiguously mapped allocations).  Answers are kept for the
// length of one call only: memory freed and reused between calls is looked
// up again.
class BufferCheck {
 public:
  explicit BufferCheck(int dev) : dev_(dev) {}

  bool ok(uintptr_t lo, uintptr_t hi) {
    if (hi < lo) return false;
    while (lo < hi) {
      uintptr_t end = 0;
      if (!known(lo, &end) && !lookup(lo, &end)) return false;
      lo = end;
    }
    return true;
  }

 private:
  bool known(uintptr_t a, uintptr_t* end) const {
    auto it = seen_.upper_bound(a);  // the first allocation starting after a
    if (it == seen_.begin()) return false;
    --it;
    if (a >= it->second) return false;
    *end = it->second;
    return true;
  }
  bool lookup(uintptr_t a, uintptr_t* end) {
    PointerAttrsFn fn = pointer_attrs();
    if (!fn) return false;
    unsigned int type = 0;
    int ordinal = -1, managed = 0;
    CUdeviceptr start = 0;
    size_t size = 0;
    CUpointer_attribute attrs[5] = {CU_POINTER_ATTRIBUTE_MEMORY_TYPE, CU_POINTER_ATTRIBUTE_DEVICE_ORDINAL,
                                    CU_POINTER_ATTRIBUTE_IS_MANAGED, CU_POINTER_ATTRIBUTE_RANGE_START_ADDR,
                                    CU_POINTER_ATTRIBUTE_RANGE_SIZE};
    void* data[5] = {&type, &ordinal, &managed, &start, &size};
    if (fn(5, attrs, data, static_cast<CUdeviceptr>(a)) != CUDA_SUCCESS) return false;
    const bool device = managed || (type == CU_MEMORYTYPE_DEVICE && ordinal == dev_);
    const uintptr_t s = static_cast<uintptr_t>(start), e = s + size;
    if (!device || size == 0 || a < s || a >= e) return false;
    seen_[s] = e;
    *end = e;
    return true;
  }

  int dev_;
  std::map<uintptr_t, uintptr_t> seen_;  // allocation start -> end (disjoint)
};

// Byte ranges touched by a call; outputs may not overlap anything else.
struct Range {
  uintptr_t lo, hi;
  bool output;
};

bool ranges_disjoint(std::vector<Range>& r) {
  std::sort(r.begin(), r.end(), [](const Range& a, const Range& b) { return a.lo < b.lo; });
  uintptr_t max_hi_any = 0, max_hi_out = 0;
  for (const Range& x : r) {
    if (x.hi == x.lo) continue;
    if (x.output ? x.lo < max_hi_any : x.lo < max_hi_out) return false;
    max_hi_any = std::max(max_hi_any, x.hi);
    if (x.output) max_hi_out = std::max(max_hi_out, x.hi);
  }
  return true;
}

// Every non-empty range of a call in device memory of the current device.
bool ranges_on_device(const std::vector<Range>& r, int dev) {
  BufferCheck check(dev);
  for (const Range& x : r)
    if (x.hi != x.lo && !check.ok(x.lo, x.hi)) return false;
  return true;
}

Range range_of(const void* p, uint64_t bytes, bool output) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(p);
  return {a, a + bytes, output};
}

// A validated package format.
struct Fmt {
  int group = 0;
  int n_stages = 0;
  rrq::Format kind = rrq::kAsymF32;
  int bits[RRQ_MAX_STAGES] = {2, 2, 2, 2};
  bool sym() const { return kind == rrq::kSymF32 || kind == rrq::kSymF16; }
  uint64_t scale_bytes() const { return kind == rrq::kSymF16 ? 2 : 4; }
  uint64_t code_bytes(uint64_t n, int k) const { return n * static_cast<uint64_t>(bits[k]) / 8; }
};

rrq_status parse_format(const rrq_format* f, Fmt* out) {
  if (!f || f->n_stages < 1 || f->n_stages > RRQ_MAX_STAGES) return RRQ_ERR_INVALID_ARG;
  if (f->grid != RRQ_GRID_ASYM && f->grid != RRQ_GRID_SYM) return RRQ_ERR_INVALID_ARG;
  if (f->scale_type != RRQ_SCALE_F32 && f->scale_type != RRQ_SCALE_F16) return RRQ_ERR_INVALID_ARG;
  bool two_bit = true;
  for (int k = 0; k < f->n_stages; ++k) {
    if (f->bits[k] < 0 || f->bits[k] > 4) return RRQ_ERR_INVALID_ARG;
    out->bits[k] = f->bits[k] == 0 ? 2 : f->bits[k];
    two_bit = two_bit && out->bits[k] == 2;
  }
  if (!group_supported(f->group)) return RRQ_ERR_UNSUPPORTED;
  out->group = f->group;
  out->n_stages = f->n_stages;
  if (f->grid == RRQ_GRID_ASYM) {
    if (f->scale_type != RRQ_SCALE_F32) return RRQ_ERR_UNSUPPORTED;
    out->kind = two_bit ? rrq::kAsymF32 : rrq::kAsymBits;
  } else {
    if (!two_bit) return RRQ_ERR_UNSUPPORTED;  // other widths: asymmetric grid only
    out->kind = f->scale_type == RRQ_SCALE_F16 ? rrq::kSymF16 : rrq::kSymF32;
  }
  return RRQ_OK;
}

Fmt asym_format(int group, int n_stages) {
  Fmt f;
  f.group = group;
  f.n_stages = n_stages;
  return f;
}

// ---------------------------------------------------------------------------
// quantize
// ---------------------------------------------------------------------------
// A quantize request for one matrix, from either descriptor type; out is
// all-null except for the build with prefixes.
struct QView {
  const uint16_t* W_bf16;
  int64_t rows, cols;
  uint8_t* codes[RRQ_MAX_STAGES];
  void* scales[RRQ_MAX_STAGES];
  float* zeros[RRQ_MAX_STAGES];
  uint16_t* out[RRQ_MAX_STAGES];
};

QView view_of(const rrq_quantize_desc& d) {
  QView v{};
  v.W_bf16 = d.W_bf16;
  v.rows = d.rows;
  v.cols = d.cols;
  for (int k = 0; k < RRQ_MAX_STAGES; ++k) {
    v.codes[k] = d.codes[k];
    v.scales[k] = d.scales[k];
    v.zeros[k] = d.zeros[k];
  }
  return v;
}

QView view_of(const rrq_quantize_prefixes_desc& d) {
  QView v{};
  v.W_bf16 = d.W_bf16;
  v.rows = d.rows;
  v.cols = d.cols;
  for (int k = 0; k < RRQ_MAX_STAGES; ++k) {
    v.codes[k] = d.codes[k];
    v.scales[k] = d.scales[k];
    v.zeros[k] = d.zeros[k];
    v.out[k] = d.out_bf16[k];
  }
  return v;
}

enum QMode { kBuild, kFromBase, kEmit };

rrq_status check_quantize_item(const QView& it, const Fmt& f, QMode mode) {
  if (!it.W_bf16 || !shape_ok(it.rows, it.cols)) return RRQ_ERR_INVALID_ARG;
  if (it.cols % f.group != 0) return RRQ_ERR_INVALID_ARG;
  for (int k = 0; k < f.n_stages; ++k)
    if (!it.codes[k] || !it.scales[k] || (!f.sym() && !it.zeros[k])) return RRQ_ERR_INVALID_ARG;
  if (!aligned(it.W_bf16, 16)) return RRQ_ERR_MISALIGNED;
  for (int k = 0; k < f.n_stages; ++k)
    if (!aligned(it.codes[k], 16) || !aligned(it.scales[k], 16) || (!f.sym() && !aligned(it.zeros[k], 16)))
      return RRQ_ERR_MISALIGNED;
  if (mode == kEmit) {
    for (int k = 0; k < f.n_stages; ++k)
      if (!it.out[k]) return RRQ_ERR_INVALID_ARG;
    for (int k = 0; k < f.n_stages; ++k)
      if (!aligned(it.out[k], 16)) return RRQ_ERR_MISALIGNED;
  }
  return RRQ_OK;
}

// kFromBase: stage 0 is an input (Algorithm 1 with a base checkpoint).
void add_quantize_ranges(const QView& it, const Fmt& f, QMode mode, std::vector<Range>& r) {
  const bool from_base = mode == kFromBase;
  const uint64_t n = static_cast<uint64_t>(it.rows * it.cols);
  r.push_back(range_of(it.W_bf16, 2 * n, false));
  if (mode == kEmit)
    for (int k = 0; k < f.n_stages; ++k) r.push_back(range_of(it.out[k], 2 * n, true));
  for (int k = 0; k < f.n_stages; ++k) {
    const bool out = !(from_base && k == 0);
    r.push_back(range_of(it.codes[k], f.code_bytes(n, k), out));
    r.push_back(range_of(it.scales[k], f.scale_bytes() * (n / f.group), out));
    if (!f.sym()) r.push_back(range_of(it.zeros[k], 4 * (n / f.group), out));
  }
}

rrq_status quantize_batch(const QView* items, int count, const Fmt& f, rrq_stream_t stream, QMode mode) {
  if (!items || count < 1) return RRQ_ERR_INVALID_ARG;
  const bool from_base = mode == kFromBase;
  if (from_base && f.n_stages < 2) return RRQ_ERR_INVALID_ARG;
  if (mode == kEmit && f.kind == rrq::kAsymBits) return RRQ_ERR_UNSUPPORTED;
  const int n_stages = f.n_stages;
  std::vector<Range> ranges;
  ranges.reserve(static_cast<size_t>(count) * (1 + 4 * n_stages));
  for (int i = 0; i < count; ++i) {
    if (rrq_status rc = check_quantize_item(items[i], f, mode)) return rc;
    add_quantize_ranges(items[i], f, mode, ranges);
  }
  if (!ranges_disjoint(ranges)) return RRQ_ERR_INVALID_ARG;

  int dev = 0;
  DeviceState* st = nullptr;
  if (rrq_status rc = current_device(&dev, &st)) return rc;
  if (!ranges_on_device(ranges, dev)) return RRQ_ERR_INVALID_ARG;

  static thread_local rrq::QuantizeBatch p;  // ~8 KiB: kept off the stack
  for (int base = 0; base < count; base += rrq::kMaxBatch) {
    const int m = std::min(rrq::kMaxBatch, count - base);
    std::memset(&p, 0, sizeof p);
    p.count = m;
    p.n_stages = n_stages;
    for (int k = 0; k < RRQ_MAX_STAGES; ++k) p.bits[k] = f.bits[k];
    p.wait_limit_us = g_wait_limit_us.load(std::memory_order_relaxed);
    p.flags = g_debug_flags.load(std::memory_order_relaxed);
    p.status = st->status;
    int64_t chunks = 0;
    for (int i = 0; i < m; ++i) {
      const QView& it = items[base + i];
      rrq::QuantizeItem& q = p.item[i];
      q.W = it.W_bf16;
      q.n = it.rows * it.cols;
      q.chunk_begin = chunks;
      chunks += (q.n + rrq::kChunkElems - 1) / rrq::kChunkElems;
      for (int k = 0; k < rrq::kMaxStages; ++k) {
        const int kk = k < n_stages ? k : n_stages - 1;
        q.codes[k] = it.codes[kk];
        q.scales[k] = it.scales[kk];
        q.zeros[k] = f.sym() ? nullptr : it.zeros[kk];
        q.out[k] = mode == kEmit ? it.out[kk] : nullptr;
      }
    }
    p.total_chunks = chunks;
    const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t e = mode == kFromBase ? rrq::quantize_launch_base(f.group, f.kind, p, s, st->sms)
                    : mode == kEmit   ? rrq::quantize_launch_emit(f.group, f.kind, p, s, st->sms)
                                      : rrq::quantize_launch(f.group, f.kind, p, s, st->sms);
    if (e != cudaSuccess) return fail_cuda(e);
  }
  return RRQ_OK;
}

// ---------------------------------------------------------------------------
// reconstruct
// ---------------------------------------------------------------------------
// A reconstruct request for one matrix: k stages in, n_out outputs
// (n_out = 1: the prefix with k stages; n_out = k: every prefix).
struct ReconView {
  const uint8_t* const* codes;
  const void* const* scales;
  const float* const* zeros;
  int64_t rows, cols;
  uint16_t* const* out;
};

rrq_status check_reconstruct_item(const ReconView& it, const Fmt& f, int k, int n_out) {
  if (!shape_ok(it.rows, it.cols)) return RRQ_ERR_INVALID_ARG;
  if (it.cols % f.group != 0) return RRQ_ERR_INVALID_ARG;
  for (int i = 0; i < k; ++i)
    if (!it.codes[i] || !it.scales[i] || (!f.sym() && !it.zeros[i])) return RRQ_ERR_INVALID_ARG;
  for (int j = 0; j < n_out; ++j)
    if (!it.out[j]) return RRQ_ERR_INVALID_ARG;
  for (int j = 0; j < n_out; ++j)
    if (!aligned(it.out[j], 16)) return RRQ_ERR_MISALIGNED;
  for (int i = 0; i < k; ++i)
    if (!aligned(it.codes[i], 16) || !aligned(it.scales[i], 16) || (!f.sym() && !aligned(it.zeros[i], 16)))
      return RRQ_ERR_MISALIGNED;
  return RRQ_OK;
}

rrq_status reconstruct_views(const ReconView* items, int count, const Fmt& f, int k, bool all_prefixes,
                             rrq_stream_t stream) {
  if (!items || count < 1 || k < 1 || k > RRQ_MAX_STAGES || k > f.n_stages) return RRQ_ERR_INVALID_ARG;
  const int group = f.group;
  const int n_out = all_prefixes ? k : 1;
  std::vector<Range> ranges;
  ranges.reserve(static_cast<size_t>(count) * (n_out + 3 * k));
  for (int i = 0; i < count; ++i) {
    const ReconView& it = items[i];
    if (rrq_status rc = check_reconstruct_item(it, f, k, n_out)) return rc;
    const uint64_t n = static_cast<uint64_t>(it.rows * it.cols);
    for (int j = 0; j < n_out; ++j) ranges.push_back(range_of(it.out[j], 2 * n, true));
    for (int j = 0; j < k; ++j) {
      ranges.push_back(range_of(it.codes[j], f.code_bytes(n, j), false));
      ranges.push_back(range_of(it.scales[j], f.scale_bytes() * (n / group), false));
      if (!f.sym()) ranges.push_back(range_of(it.zeros[j], 4 * (n / group), false));
    }
  }
  if (!ranges_disjoint(ranges)) return RRQ_ERR_INVALID_ARG;

  int dev = 0;
  DeviceState* st = nullptr;
  if (rrq_status rc = current_device(&dev, &st)) return rc;
  if (!ranges_on_device(ranges, dev)) return RRQ_ERR_INVALID_ARG;

  static thread_local rrq::ReconstructBatch p;
  for (int base = 0; base < count; base += rrq::kMaxBatch) {
    const int m = std::min(rrq::kMaxBatch, count - base);
    std::memset(&p, 0, sizeof p);
    p.count = m;
    for (int j = 0; j < RRQ_MAX_STAGES; ++j) p.bits[j] = f.bits[j];
    p.wait_limit_us = g_wait_limit_us.load(std::memory_order_relaxed);
    p.status = st->status;
    int64_t chunks = 0;
    for (int i = 0; i < m; ++i) {
      const ReconView& it = items[base + i];
      rrq::ReconstructItem& q = p.item[i];
      for (int j = 0; j < rrq::kMaxStages; ++j) {
        const int jj = j < k ? j : k - 1;
        q.codes[j] = it.codes[jj];
        q.scales[j] = it.scales[jj];
        q.zeros[j] = f.sym() ? nullptr : it.zeros[jj];
        q.out[j] = it.out[j < n_out ? j : n_out - 1];
      }
      q.n = it.rows * it.cols;
      q.chunk_begin = chunks;
      chunks += (q.n + rrq::kChunkElems - 1) / rrq::kChunkElems;
    }
    p.total_chunks = chunks;
    cudaError_t e = rrq::reconstruct_launch(group, f.kind, k, all_prefixes, p,
                                            reinterpret_cast<cudaStream_t>(stream), st->sms);
    if (e != cudaSuccess) return fail_cuda(e);
  }
  return RRQ_OK;
}

// ---------------------------------------------------------------------------
// stage-wise product
// ---------------------------------------------------------------------------
// Checks shared by the two products: shapes, pointers, alignment, no output
// overlapping an input or another output (act_rows activation rows per
// matrix), and every pointer on the current device; returns the device state.
rrq_status check_product_items(const rrq_gemv_desc* items, int count, const Fmt& f, int k, uint64_t act_rows,
                               DeviceState** st_out) {
  const int group = f.group;
  std::vector<Range> ranges;
  ranges.reserve(static_cast<size_t>(count) * (2 + 3 * k));
  for (int i = 0; i < count; ++i) {
    const rrq_gemv_desc& it = items[i];
    if (!shape_ok(it.rows, it.cols) || it.cols % group != 0 || !it.A_bf16 || !it.Y) return RRQ_ERR_INVALID_ARG;
    for (int j = 0; j < k; ++j)
      if (!it.codes[j] || !it.scales[j] || (!f.sym() && !it.zeros[j])) return RRQ_ERR_INVALID_ARG;
    if (!aligned(it.A_bf16, 16) || !aligned(it.Y, 16)) return RRQ_ERR_MISALIGNED;
    for (int j = 0; j < k; ++j)
      if (!aligned(it.codes[j], 16) || !aligned(it.scales[j], 16) || (!f.sym() && !aligned(it.zeros[j], 16)))
        return RRQ_ERR_MISALIGNED;
    const uint64_t n = static_cast<uint64_t>(it.rows * it.cols);
    ranges.push_back(range_of(it.A_bf16, 2 * act_rows * it.cols, false));
    ranges.push_back(range_of(it.Y, 4 * act_rows * it.rows, true));
    for (int j = 0; j < k; ++j) {
      ranges.push_back(range_of(it.codes[j], f.code_bytes(n, j), false));
      ranges.push_back(range_of(it.scales[j], f.scale_bytes() * (n / group), false));
      if (!f.sym()) ranges.push_back(range_of(it.zeros[j], 4 * (n / group), false));
    }
  }
  if (!ranges_disjoint(ranges)) return RRQ_ERR_INVALID_ARG;

  int dev = 0;
  DeviceState* st = nullptr;
  if (rrq_status rc = current_device(&dev, &st)) return rc;
  if (!ranges_on_device(ranges, dev)) return RRQ_ERR_INVALID_ARG;

  *st_out = st;
  return RRQ_OK;
}

rrq_status gemv_batch(const rrq_gemv_desc* items, int count, const Fmt& f, int k, int batch,
                      rrq_stream_t stream) {
  if (!items || count < 1 || k < 1 || k > f.n_stages) return RRQ_ERR_INVALID_ARG;
  if (batch < 1 || batch > rrq::kMaxGemvBatch) return RRQ_ERR_INVALID_ARG;
  const int group = f.group;
  DeviceState* st = nullptr;
  if (rrq_status rc = check_product_items(items, count, f, k, static_cast<uint64_t>(batch), &st)) return rc;

  // activation rows one launch holds for each matrix (shared memory); the
  // matrices that take the same number go together, so that a wide matrix
  // does not split the batch of the narrower ones
  std::vector<int> per(count), order(count);
  for (int i = 0; i < count; ++i) {
    if (items[i].cols > RRQ_MAX_GEMV_COLS) return RRQ_ERR_UNSUPPORTED;  // the stated limit of every form
    const int cap = rrq::gemv_rows_per_launch(f.kind, k, items[i].cols, group);
    if (cap < 1) return RRQ_ERR_UNSUPPORTED;
    per[i] = std::min(cap, batch);
    order[i] = i;
  }
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return per[a] > per[b]; });

  int log2g = 0;
  while ((1 << log2g) < group) ++log2g;
  static thread_local rrq::GemvBatch p;
  for (int base = 0; base < count;) {
    // up to kMaxBatch matrices with the same rows per launch
    int m = 1;
    while (m < rrq::kMaxBatch && base + m < count && per[order[base + m]] == per[order[base]]) ++m;
    const int rows_per = per[order[base]];
    std::memset(&p, 0, sizeof p);
    p.count = m;
    p.log2g = log2g;
    for (int j = 0; j < rrq::kMaxStages; ++j) p.bits[j] = f.bits[j];
    int64_t blocks = 0, max_cols = 0;
    for (int i = 0; i < m; ++i) {
      const rrq_gemv_desc& it = items[order[base + i]];
      rrq::GemvItem& q = p.item[i];
      for (int j = 0; j < rrq::kMaxStages; ++j) {
        const int jj = j < k ? j : k - 1;
        q.codes[j] = it.codes[jj];
        q.scales[j] = it.scales[jj];
        q.zeros[j] = f.sym() ? nullptr : it.zeros[jj];
      }
      q.rows = it.rows;
      q.cols = it.cols;
      q.blk_begin = blocks;
      blocks += (it.rows + rrq::kGemvRows - 1) / rrq::kGemvRows;
      max_cols = std::max(max_cols, it.cols);
    }
    p.total_blocks = blocks;
    for (int b0 = 0; b0 < batch; b0 += rows_per) {
      const int nb = std::min(rows_per, batch - b0);
      for (int i = 0; i < m; ++i) {
        const rrq_gemv_desc& it = items[order[base + i]];
        p.item[i].A = it.A_bf16 + static_cast<int64_t>(b0) * it.cols;
        p.item[i].Y = it.Y + static_cast<int64_t>(b0) * it.rows;
      }
      cudaError_t e = rrq::gemv_launch(f.kind, k, nb, max_cols, p, reinterpret_cast<cudaStream_t>(stream), st->sms);
      if (e != cudaSuccess) return fail_cuda(e);
    }
    base += m;
  }
  return RRQ_OK;
}

// The driver's tensor-map encoder, looked up once through the runtime (no
// link against the driver library).
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_tiled() {
  static EncodeTiledFn fn = [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return static_cast<EncodeTiledFn>(nullptr);
    return reinterpret_cast<EncodeTiledFn>(ptr);
  }();
  return fn;
}

// Activations [tokens, cols] bf16 as a 2-D tensor map: boxes of 64 columns x
// kPrefillMmaN tokens, 128-byte swizzle (the MMA's K-major operand layout),
// zeros outside the matrix.
bool encode_activations(CUtensorMap* map, const uint16_t* A, int64_t tokens, int64_t cols) {
  EncodeTiledFn fn = encode_tiled();
  if (!fn) return false;
  const cuuint64_t dim[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(tokens)};
  const cuuint64_t stride[1] = {static_cast<cuuint64_t>(cols) * 2};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(rrq::kPrefillBK), static_cast<cuuint32_t>(rrq::kPrefillMmaN)};
  const cuuint32_t estride[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<uint16_t*>(A), dim, stride, box, estride,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Codes of one stage [rows, cols/4] bytes as a 2-D tensor map: boxes of 16
// bytes (64 weights) x box_rows rows, no swizzle, zeros outside (needs
// cols % 64 == 0 for 16-byte row strides).
bool encode_codes(CUtensorMap* map, const uint8_t* codes, int64_t rows, int64_t cols, int box_rows) {
  EncodeTiledFn fn = encode_tiled();
  if (!fn) return false;
  const cuuint64_t dim[2] = {static_cast<cuuint64_t>(cols / 4), static_cast<cuuint64_t>(rows)};
  const cuuint64_t stride[1] = {static_cast<cuuint64_t>(cols / 4)};
  const cuuint32_t box[2] = {16, static_cast<cuuint32_t>(box_rows)};
  const cuuint32_t estride[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t*>(codes), dim, stride, box, estride,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool rrq::encode_lane_tiles(CUtensorMap* map, const uint16_t* W, int64_t n, int lw) {
  EncodeTiledFn fn = encode_tiled();
  if (!fn || (lw != 32 && lw != 64) || n % lw != 0 || n / lw >= (int64_t{1} << 31)) return false;
  const cuuint64_t dim[2] = {static_cast<cuuint64_t>(lw), static_cast<cuuint64_t>(n / lw)};
  const cuuint64_t stride[1] = {static_cast<cuuint64_t>(lw) * 2};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(lw), 32};
  const cuuint32_t estride[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<uint16_t*>(W), dim, stride, box, estride,
            CU_TENSOR_MAP_INTERLEAVE_NONE, lw == 64 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

namespace {

rrq_status prefill_batch(const rrq_gemv_desc* items, int count, const Fmt& f, int k, int64_t tokens,
                         rrq_stream_t stream) {
  if (!items || count < 1 || k < 1 || k > f.n_stages) return RRQ_ERR_INVALID_ARG;
  if (tokens < 1 || tokens > RRQ_MAX_PREFILL_TOKENS) return RRQ_ERR_INVALID_ARG;
  const bool widths = f.kind == rrq::kAsymBits;
  const int group = f.group;
  for (int i = 0; i < count; ++i)
    if (items[i].cols > (int64_t{1} << 31) - rrq::kPrefillBK) return RRQ_ERR_INVALID_ARG;  // TMA coordinates
  DeviceState* st = nullptr;
  if (rrq_status rc = check_product_items(items, count, f, k, static_cast<uint64_t>(tokens), &st)) return rc;

  int log2g = 0;
  while ((1 << log2g) < group) ++log2g;
  const int64_t token_tiles = (tokens + rrq::kPrefillBN - 1) / rrq::kPrefillBN;
  // clusters share weight tiles across token tiles: 4 CTAs for the longer
  // prefixes (forming weights costs most there), else 2 (measured best on
  // Qwen3-8B-shaped layers at 2048 tokens)
  // (per-stage widths: one CTA, each thread forming whole 32-weight words)
  const int cluster = widths ? 1 : (k >= 3 && token_tiles >= 3) ? 4 : token_tiles >= 2 ? 2 : 1;
  const int64_t token_tiles_padded = (token_tiles + cluster - 1) / cluster * cluster;
  static thread_local rrq::PrefillBatch p;
  for (int base = 0; base < count; base += rrq::kMaxPrefillBatch) {
    const int m = std::min(rrq::kMaxPrefillBatch, count - base);
    std::memset(&p, 0, sizeof p);
    p.count = m;
    p.log2g = log2g;
    p.tokens = tokens;
    p.cluster = cluster;
    p.wait_limit_us = g_wait_limit_us.load(std::memory_order_relaxed);
    p.status = st->status;
    int64_t tiles = 0;
    p.codes_tma = widths ? 0 : 1;
    p.scale_blocks = 1;
    for (int j = 0; j < rrq::kMaxStages; ++j) p.bits[j] = f.bits[j];
    for (int i = 0; i < m; ++i) {
      if (items[base + i].cols % 64 != 0) p.codes_tma = 0;
      if ((items[base + i].cols / group) % (16 / f.scale_bytes()) != 0) p.scale_blocks = 0;
    }
    // longest rows first: their tiles start in the first waves instead of
    // forming a long last wave (the tile order is the launch's)
    int order[rrq::kMaxPrefillBatch];
    for (int i = 0; i < m; ++i) order[i] = base + i;
    std::stable_sort(order, order + m, [&](int a, int b) { return items[a].cols > items[b].cols; });
    for (int i = 0; i < m; ++i) {
      const rrq_gemv_desc& it = items[order[i]];
      rrq::PrefillItem& q = p.item[i];
      for (int j = 0; j < rrq::kMaxStages; ++j) {
        const int jj = j < k ? j : k - 1;
        q.codes[j] = it.codes[jj];
        q.scales[j] = it.scales[jj];
        q.zeros[j] = f.sym() ? nullptr : it.zeros[jj];
      }
      q.Y = it.Y;
      q.rows = it.rows;
      q.cols = it.cols;
      const int64_t row_tiles = (it.rows + rrq::kPrefillBM - 1) / rrq::kPrefillBM;
      q.tile_begin = tiles;
      q.row_tiles = static_cast<int32_t>(row_tiles);
      tiles += row_tiles * token_tiles_padded;
      if (!encode_activations(&p.act[i], it.A_bf16, tokens, it.cols)) return RRQ_ERR_UNSUPPORTED;
      if (p.codes_tma)
        for (int j = 0; j < k; ++j)
          if (!encode_codes(&p.codes[i][j], it.codes[j], it.rows, it.cols, rrq::kPrefillBM / cluster))
            return RRQ_ERR_UNSUPPORTED;
    }
    if (tiles > 0x7fffffff) return RRQ_ERR_INVALID_ARG;
    p.total_tiles = tiles;
    cudaError_t e = rrq::prefill_launch(f.kind, k, p, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return fail_cuda(e);
  }
  return RRQ_OK;
}

rrq_status pmr_batch(const rrq_pmr_desc* items, int count, int group, rrq_stream_t stream) {
  if (!items || count < 1) return RRQ_ERR_INVALID_ARG;
  if (!group_supported(group)) return RRQ_ERR_UNSUPPORTED;
  std::vector<Range> ranges;
  for (int i = 0; i < count; ++i) {
    const rrq_pmr_desc& it = items[i];
    if (!it.W_bf16 || !it.pmr || !shape_ok(it.rows, it.cols) || it.cols % group != 0) return RRQ_ERR_INVALID_ARG;
    if (!aligned(it.W_bf16, 16) || !aligned(it.pmr, 16) || (it.stats && !aligned(it.stats, 4)))
      return RRQ_ERR_MISALIGNED;
    const uint64_t n = static_cast<uint64_t>(it.rows * it.cols);
    ranges.push_back(range_of(it.W_bf16, 2 * n, false));
    ranges.push_back(range_of(it.pmr, 4 * (n / group), true));
    if (it.stats) ranges.push_back(range_of(it.stats, 8, true));
  }
  if (!ranges_disjoint(ranges)) return RRQ_ERR_INVALID_ARG;
  int dev = 0;
  DeviceState* st = nullptr;
  if (rrq_status rc = current_device(&dev, &st)) return rc;
  if (!ranges_on_device(ranges, dev)) return RRQ_ERR_INVALID_ARG;
  static thread_local rrq::PmrBatch p;
  for (int base = 0; base < count; base += rrq::kMaxBatch) {
    const int m = std::min(rrq::kMaxBatch, count - base);
    std::memset(&p, 0, sizeof p);
    p.count = m;
    p.group = group;
    int64_t chunks = 0;
    for (int i = 0; i < m; ++i) {
      const rrq_pmr_desc& it = items[base + i];
      rrq::PmrItem& q = p.item[i];
      q.W = it.W_bf16;
      q.pmr = it.pmr;
      q.stats = it.stats;
      q.n = it.rows * it.cols;
      q.chunk_begin = chunks;
      chunks += (q.n + rrq::kChunkElems - 1) / rrq::kChunkElems;
    }
    p.total_chunks = chunks;
    cudaError_t e = rrq::pmr_launch(group, p, reinterpret_cast<cudaStream_t>(stream), st->sms);
    if (e != cudaSuccess) return fail_cuda(e);
  }
  return RRQ_OK;
}

template <typename Desc>
rrq_status quantize_descs(const Desc* items, int count, const rrq_format* fmt, rrq_stream_t stream, QMode mode) {
  Fmt f;
  if (rrq_status rc = parse_format(fmt, &f)) return rc;
  if (!items || count < 1) return RRQ_ERR_INVALID_ARG;
  std::vector<QView> v(static_cast<size_t>(count));
  for (int i = 0; i < count; ++i) v[i] = view_of(items[i]);
  return quantize_batch(v.data(), count, f, stream, mode);
}

}  // namespace

extern "C" {

rrq_status rrq_group_pmr(const rrq_pmr_desc* items, int count, int group, rrq_stream_t stream) {
  return pmr_batch(items, count, group, stream);
}

size_t rrq_codes_bytes(int64_t rows, int64_t cols) {
  if (!shape_ok(rows, cols)) return 0;
  return static_cast<size_t>(rows * cols / 4);
}

size_t rrq_meta_count(int64_t rows, int64_t cols, int group) {
  if (!shape_ok(rows, cols) || group < 1 || cols % group != 0) return 0;
  return static_cast<size_t>(rows * cols / group);
}

size_t rrq_package_bytes(int64_t rows, int64_t cols, int group, int n_stages) {
  if (n_stages < 1 || n_stages > RRQ_MAX_STAGES) return 0;
  const size_t m = rrq_meta_count(rows, cols, group);
  if (m == 0) return 0;
  return static_cast<size_t>(n_stages) * (rrq_codes_bytes(rows, cols) + 8 * m);
}

rrq_status rrq_quantize(const uint16_t* W_bf16, int64_t rows, int64_t cols, int group,
                        int n_stages, uint8_t* const out_codes[], float* const out_scales[],
                        float* const out_zeros[], rrq_stream_t stream) {
  if (!out_codes || !out_scales || !out_zeros || n_stages < 1 || n_stages > RRQ_MAX_STAGES)
    return RRQ_ERR_INVALID_ARG;
  if (!group_supported(group)) return RRQ_ERR_UNSUPPORTED;
  QView it{};
  it.W_bf16 = W_bf16;
  it.rows = rows;
  it.cols = cols;
  for (int k = 0; k < n_stages; ++k) {
    it.codes[k] = out_codes[k];
    it.scales[k] = out_scales[k];
    it.zeros[k] = out_zeros[k];
  }
  return quantize_batch(&it, 1, asym_format(group, n_stages), stream, kBuild);
}

rrq_status rrq_quantize_batch(const rrq_quantize_item* items, int count, int group, int n_stages,
                              rrq_stream_t stream) {
  if (!items || count < 1 || n_stages < 1 || n_stages > RRQ_MAX_STAGES) return RRQ_ERR_INVALID_ARG;
  if (!group_supported(group)) return RRQ_ERR_UNSUPPORTED;
  std::vector<QView> d(static_cast<size_t>(count));
  for (int i = 0; i < count; ++i) {
    d[i] = QView{};
    d[i].W_bf16 = items[i].W_bf16;
    d[i].rows = items[i].rows;
    d[i].cols = items[i].cols;
    for (int k = 0; k < RRQ_MAX_STAGES; ++k) {
      d[i].codes[k] = items[i].codes[k];
      d[i].scales[k] = items[i].scales[k];
      d[i].zeros[k] = items[i].zeros[k];
    }
  }
  return quantize_batch(d.data(), count, asym_format(group, n_stages), stream, kBuild);
}

rrq_status rrq_quantize_ex(const rrq_quantize_desc* items, int count, const rrq_format* fmt,
                           rrq_stream_t stream) {
  return quantize_descs(items, count, fmt, stream, kBuild);
}

rrq_status rrq_quantize_prefixes(const rrq_quantize_prefixes_desc* items, int count, const rrq_format* fmt,
                                 rrq_stream_t stream) {
  return quantize_descs(items, count, fmt, stream, kEmit);
}

rrq_status rrq_reconstruct(const uint8_t* const codes[], const float* const scales[],
                           const float* const zeros[], int64_t rows, int64_t cols, int group,
                           int k, uint16_t* out_bf16, rrq_stream_t stream) {
  if (!codes || !scales || !zeros || !out_bf16 || k < 1 || k > RRQ_MAX_STAGES) return RRQ_ERR_INVALID_ARG;
  if (!group_supported(group)) return RRQ_ERR_UNSUPPORTED;
  uint16_t* const outs[1] = {out_bf16};
  const void* sc[RRQ_MAX_STAGES] = {};
  for (int i = 0; i < k; ++i) sc[i] = scales[i];
  const ReconView v{codes, sc, zeros, rows, cols, outs};
  return reconstruct_views(&v, 1, asym_format(group, k), k, false, stream);
}

rrq_status rrq_reconstruct_batch(const rrq_reconstruct_item* items, int count, int group, int k,
                                 rrq_stream_t stream) {
  if (!items || count < 1 || k < 1 || k > RRQ_MAX_STAGES) return RRQ_ERR_INVALID_ARG;
  if (!group_supported(group)) return RRQ_ERR_UNSUPPORTED;
  std::vector<ReconView> v(static_cast<size_t>(count));
  std::vector<const void*> sc(static_cast<size_t>(count) * RRQ_MAX_STAGES);
  for (int i = 0; i < count; ++i) {
    for (int j = 0; j < RRQ_MAX_STAGES; ++j) sc[i * RRQ_MAX_STAGES + j] = items[i].scales[j];
    v[i] = {items[i].codes, &sc[i * RRQ_MAX_STAGES], items[i].zeros, items[i].rows, items[i].cols,
            &items[i].out_bf16};
  }
  return reconstruct_views(v.data(), count, asym_format(group, k), k, false, stream);
}

rrq_status rrq_reconstruct_prefixes(const uint8_t* const codes[], const float* const scales[],
                                    const float* const zeros[], int64_t rows, int64_t cols,
                                    int group, int k, uint16_t* const out_bf16[],
                                    rrq_stream_t stream) {
  if (!codes || !scales || !zeros || !out_bf16 || k < 1 || k > RRQ_MAX_STAGES) return RRQ_ERR_INVALID_ARG;
  if (!group_supported(group)) return RRQ_ERR_UNSUPPORTED;
  const void* sc[RRQ_MAX_STAGES] = {};
  for (int i = 0; i < k; ++i) sc[i] = scales[i];
  const ReconView v{codes, sc, zeros, rows, cols, out_bf16};
  return reconstruct_views(&v, 1, asym_format(group, k), k, true, stream);
}

rrq_status rrq_reconstruct_prefixes_batch(const rrq_prefixes_item* items, int count, int group,
                                          int k, rrq_stream_t stream) {
  if (!items || count < 1 || k < 1 || k > RRQ_MAX_STAGES) return RRQ_ERR_INVALID_ARG;
  if (!group_supported(group)) return RRQ_ERR_UNSUPPORTED;
  std::vector<ReconView> v(static_cast<size_t>(count));
  std::vector<const void*> sc(static_cast<size_t>(count) * RRQ_MAX_STAGES);
  for (int i = 0; i < count; ++i) {
    for (int j = 0; j < RRQ_MAX_STAGES; ++j) sc[i * RRQ_MAX_STAGES + j] = items[i].scales[j];
    v[i] = {items[i].codes, &sc[i * RRQ_MAX_STAGES], items[i].zeros, items[i].rows, items[i].cols,
            items[i].out_bf16};
  }
  return reconstruct_views(v.data(), count, asym_format(group, k), k, true, stream);
}

rrq_status rrq_quantize_from_base(const rrq_quantize_desc* items, int count, const rrq_format* fmt,
                                  rrq_stream_t stream) {
  return quantize_descs(items, count, fmt, stream, kFromBase);
}

rrq_status rrq_gemv(const rrq_gemv_desc* items, int count, const rrq_format* fmt, int k, int batch,
                    rrq_stream_t stream) {
  Fmt f;
  if (rrq_status rc = parse_format(fmt, &f)) return rc;
  return gemv_batch(items, count, f, k, batch, stream);
}

rrq_status rrq_prefill(const rrq_gemv_desc* items, int count, const rrq_format* fmt, int k, int64_t tokens,
                       rrq_stream_t stream) {
  Fmt f;
  if (rrq_status rc = parse_format(fmt, &f)) return rc;
  return prefill_batch(items, count, f, k, tokens, stream);
}

rrq_status rrq_reconstruct_ex(const rrq_reconstruct_desc* items, int count, const rrq_format* fmt,
                              int k, int all_prefixes, rrq_stream_t stream) {
  Fmt f;
  if (rrq_status rc = parse_format(fmt, &f)) return rc;
  if (!items || count < 1) return RRQ_ERR_INVALID_ARG;
  std::vector<ReconView> v(static_cast<size_t>(count));
  for (int i = 0; i < count; ++i)
    v[i] = {items[i].codes, items[i].scales, items[i].zeros, items[i].rows, items[i].cols, items[i].out_bf16};
  return reconstruct_views(v.data(), count, f, k, all_prefixes != 0, stream);
}

size_t rrq_stage_codes_bytes(int64_t rows, int64_t cols, int bits) {
  if (!shape_ok(rows, cols) || bits < 1 || bits > 4) return 0;
  return static_cast<size_t>(rows * cols) * static_cast<size_t>(bits) / 8;
}

size_t rrq_scales_bytes(int64_t rows, int64_t cols, const rrq_format* fmt) {
  Fmt f;
  if (parse_format(fmt, &f) != RRQ_OK) return 0;
  return rrq_meta_count(rows, cols, f.group) * static_cast<size_t>(f.scale_bytes());
}

size_t rrq_package_bytes_ex(int64_t rows, int64_t cols, const rrq_format* fmt) {
  Fmt f;
  if (parse_format(fmt, &f) != RRQ_OK) return 0;
  const size_t m = rrq_meta_count(rows, cols, f.group);
  if (m == 0) return 0;
  size_t total = 0;
  for (int k = 0; k < f.n_stages; ++k)
    total += rrq_stage_codes_bytes(rows, cols, f.bits[k]) + m * (f.scale_bytes() + (f.sym() ? 0 : 4));
  return total;
}

rrq_status rrq_get_device_status(rrq_stream_t stream) {
  int dev = 0;
  DeviceState* st = nullptr;
  if (rrq_status rc = current_device(&dev, &st)) return rc;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return fail_cuda(e);
  rrq_take_status_kernel<<<1, 1, 0, s>>>();
  if ((e = cudaGetLastError())) return fail_cuda(e);
  unsigned word = 0;
  if ((e = cudaMemcpyFromSymbolAsync(&word, rrq_device_status_taken, sizeof word, 0, cudaMemcpyDeviceToHost, s)))
    return fail_cuda(e);
  if ((e = cudaStreamSynchronize(s))) return fail_cuda(e);
  return (word & rrq::kStatusTimeout) ? RRQ_ERR_TIMEOUT : RRQ_OK;
}

rrq_status rrq_check_buffer(const void* p, size_t bytes) {
  if (!p) return RRQ_ERR_INVALID_ARG;
  int dev = 0;
  DeviceState* st = nullptr;
  if (rrq_status rc = current_device(&dev, &st)) return rc;
  const uintptr_t a = reinterpret_cast<uintptr_t>(p);
  BufferCheck check(dev);
  return check.ok(a, a + (bytes ? bytes : 1)) ? RRQ_OK : RRQ_ERR_INVALID_ARG;
}

void rrq_set_wait_limit_us(uint32_t microseconds) {
  g_wait_limit_us.store(microseconds, std::memory_order_relaxed);
}

void rrq_set_debug_flags(uint32_t flags) { g_debug_flags.store(flags, std::memory_order_relaxed); }

const char* rrq_status_string(rrq_status status) {
  switch (status) {
    case RRQ_OK: return "RRQ_OK";
    case RRQ_ERR_INVALID_ARG: return "RRQ_ERR_INVALID_ARG: invalid argument";
    case RRQ_ERR_UNSUPPORTED: return "RRQ_ERR_UNSUPPORTED: unsupported group size";
    case RRQ_ERR_MISALIGNED: return "RRQ_ERR_MISALIGNED: pointer alignment";
    case RRQ_ERR_CUDA: return "RRQ_ERR_CUDA: CUDA runtime error";
    case RRQ_ERR_TIMEOUT: return "RRQ_ERR_TIMEOUT: a kernel gave up on a bounded wait";
  }
  return "unknown rrq_status";
}

int rrq_last_cuda_error(void) { return t_last_cuda_error; }

}  // extern "C"
