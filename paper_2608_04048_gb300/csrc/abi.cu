// C ABI of the RRQ library (declared in include/rrq.h): argument checks,
// per-device set-up and kernel launches.  Every check runs before anything is
// launched, so a rejected call has no effect on the device.
#include <atomic>
#include <cstdint>
#include <cstring>
#include <mutex>

#include <cuda_runtime.h>

#include "rrq.h"
#include "rrq_internal.h"

// Per-device status word: bit kStatusTimeout is set by a kernel that gave up
// on a bounded wait.  Read and cleared by rrq_get_device_status.
__device__ unsigned int rrq_device_status;

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
    if ((e = rrq::reconstruct_prepare())) return fail_cuda(e);
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

// Device (or managed) memory that the current device can address.
bool on_device(const void* p, int dev) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();  // clear the sticky-free error of an unknown pointer
    return false;
  }
  if (a.type == cudaMemoryTypeManaged) return true;
  return a.type == cudaMemoryTypeDevice && a.device == dev;
}

struct Range {
  uintptr_t lo, hi;
};
bool overlap(Range a, Range b) { return a.lo < b.hi && b.lo < a.hi; }

}  // namespace

extern "C" {

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
  if (!W_bf16 || !out_codes || !out_scales || !out_zeros) return RRQ_ERR_INVALID_ARG;
  if (!shape_ok(rows, cols) || n_stages < 1 || n_stages > RRQ_MAX_STAGES) return RRQ_ERR_INVALID_ARG;
  if (!group_supported(group)) return RRQ_ERR_UNSUPPORTED;
  if (cols % group != 0) return RRQ_ERR_INVALID_ARG;
  for (int k = 0; k < n_stages; ++k)
    if (!out_codes[k] || !out_scales[k] || !out_zeros[k]) return RRQ_ERR_INVALID_ARG;
  if (!aligned(W_bf16, 16)) return RRQ_ERR_MISALIGNED;
  for (int k = 0; k < n_stages; ++k)
    if (!aligned(out_codes[k], 8) || !aligned(out_scales[k], 4) || !aligned(out_zeros[k], 4))
      return RRQ_ERR_MISALIGNED;

  const int64_t n = rows * cols;
  const size_t code_bytes = static_cast<size_t>(n / 4);
  const size_t meta_bytes = static_cast<size_t>(n / group) * sizeof(float);
  Range ranges[1 + 3 * RRQ_MAX_STAGES];
  int nr = 0;
  ranges[nr++] = {reinterpret_cast<uintptr_t>(W_bf16), reinterpret_cast<uintptr_t>(W_bf16) + 2 * n};
  for (int k = 0; k < n_stages; ++k) {
    const uintptr_t c = reinterpret_cast<uintptr_t>(out_codes[k]);
    const uintptr_t s = reinterpret_cast<uintptr_t>(out_scales[k]);
    const uintptr_t z = reinterpret_cast<uintptr_t>(out_zeros[k]);
    ranges[nr++] = {c, c + code_bytes};
    ranges[nr++] = {s, s + meta_bytes};
    ranges[nr++] = {z, z + meta_bytes};
  }
  for (int a = 0; a < nr; ++a)
    for (int b = a + 1; b < nr; ++b)
      if (overlap(ranges[a], ranges[b])) return RRQ_ERR_INVALID_ARG;

  int dev = 0;
  DeviceState* st = nullptr;
  if (rrq_status rc = current_device(&dev, &st)) return rc;
  if (!on_device(W_bf16, dev)) return RRQ_ERR_INVALID_ARG;
  for (int k = 0; k < n_stages; ++k)
    if (!on_device(out_codes[k], dev) || !on_device(out_scales[k], dev) || !on_device(out_zeros[k], dev))
      return RRQ_ERR_INVALID_ARG;

  rrq::QuantizeParams p{};
  p.W = W_bf16;
  p.n = n;
  for (int k = 0; k < rrq::kMaxStages; ++k) {
    const int kk = k < n_stages ? k : n_stages - 1;
    p.codes[k] = out_codes[kk];
    p.scales[k] = out_scales[kk];
    p.zeros[k] = out_zeros[kk];
  }
  p.n_stages = n_stages;
  p.wait_limit_us = g_wait_limit_us.load(std::memory_order_relaxed);
  p.flags = g_debug_flags.load(std::memory_order_relaxed);
  p.status = st->status;
  cudaError_t e = rrq::quantize_launch(group, p, reinterpret_cast<cudaStream_t>(stream), st->sms);
  if (e != cudaSuccess) return fail_cuda(e);
  return RRQ_OK;
}

rrq_status rrq_reconstruct(const uint8_t* const codes[], const float* const scales[],
                           const float* const zeros[], int64_t rows, int64_t cols, int group,
                           int k, uint16_t* out_bf16, rrq_stream_t stream) {
  if (!codes || !scales || !zeros || !out_bf16) return RRQ_ERR_INVALID_ARG;
  if (!shape_ok(rows, cols) || k < 1 || k > RRQ_MAX_STAGES) return RRQ_ERR_INVALID_ARG;
  if (!group_supported(group)) return RRQ_ERR_UNSUPPORTED;
  if (cols % group != 0) return RRQ_ERR_INVALID_ARG;
  for (int i = 0; i < k; ++i)
    if (!codes[i] || !scales[i] || !zeros[i]) return RRQ_ERR_INVALID_ARG;
  if (!aligned(out_bf16, 16)) return RRQ_ERR_MISALIGNED;
  for (int i = 0; i < k; ++i)
    if (!aligned(codes[i], 8) || !aligned(scales[i], 4) || !aligned(zeros[i], 4)) return RRQ_ERR_MISALIGNED;

  const int64_t n = rows * cols;
  const Range out{reinterpret_cast<uintptr_t>(out_bf16), reinterpret_cast<uintptr_t>(out_bf16) + 2 * n};
  for (int i = 0; i < k; ++i) {
    const uintptr_t c = reinterpret_cast<uintptr_t>(codes[i]);
    const uintptr_t s = reinterpret_cast<uintptr_t>(scales[i]);
    const uintptr_t z = reinterpret_cast<uintptr_t>(zeros[i]);
    const size_t mb = static_cast<size_t>(n / group) * sizeof(float);
    if (overlap(out, {c, c + static_cast<size_t>(n / 4)}) || overlap(out, {s, s + mb}) ||
        overlap(out, {z, z + mb}))
      return RRQ_ERR_INVALID_ARG;
  }

  int dev = 0;
  DeviceState* st = nullptr;
  if (rrq_status rc = current_device(&dev, &st)) return rc;
  if (!on_device(out_bf16, dev)) return RRQ_ERR_INVALID_ARG;
  for (int i = 0; i < k; ++i)
    if (!on_device(codes[i], dev) || !on_device(scales[i], dev) || !on_device(zeros[i], dev))
      return RRQ_ERR_INVALID_ARG;

  rrq::ReconstructParams p{};
  for (int i = 0; i < rrq::kMaxStages; ++i) {
    const int ii = i < k ? i : k - 1;
    p.codes[i] = codes[ii];
    p.scales[i] = scales[ii];
    p.zeros[i] = zeros[ii];
  }
  p.n = n;
  p.out = out_bf16;
  p.wait_limit_us = g_wait_limit_us.load(std::memory_order_relaxed);
  p.status = st->status;
  cudaError_t e = rrq::reconstruct_launch(group, k, p, reinterpret_cast<cudaStream_t>(stream), st->sms);
  if (e != cudaSuccess) return fail_cuda(e);
  return RRQ_OK;
}

rrq_status rrq_get_device_status(rrq_stream_t stream) {
  int dev = 0;
  DeviceState* st = nullptr;
  if (rrq_status rc = current_device(&dev, &st)) return rc;
  cudaError_t e = cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return fail_cuda(e);
  unsigned word = 0;
  if ((e = cudaMemcpyFromSymbol(&word, rrq_device_status, sizeof word))) return fail_cuda(e);
  if (word != 0) {
    const unsigned zero = 0;
    if ((e = cudaMemcpyToSymbol(rrq_device_status, &zero, sizeof zero))) return fail_cuda(e);
  }
  return (word & rrq::kStatusTimeout) ? RRQ_ERR_TIMEOUT : RRQ_OK;
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
