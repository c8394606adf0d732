// acid_drift_signal_noalloc: the drift reduction for callers that cannot
// allocate device memory at all, not even a workspace to hand to
// acid_drift_signal.  Examples: a plugin that only receives its input and
// output buffers from a host framework, or an inference process whose device
// memory is entirely reserved by another allocator.
//
// The reduction's scratch (one fp64 partial pair per thread block plus the
// three results) lives in the file-scope array below instead of a
// caller-provided workspace.  Every GPU that loads this library holds the
// array until the process exits.
#include <mutex>
#include <string>

#include "common.cuh"
#include "internal.h"

namespace acid {

bool is_device_pointer(const void* p);

namespace {

constexpr size_t kNoAllocScratchBytes = 16 * 1024;
// Largest element count accepted: the grid is capped at a fixed number of
// thread blocks, so each thread's fp32 partial sums cover at most about 55,000
// values at this size, which keeps their rounding far below the 1e-3 drift
// tolerance.
constexpr int64_t kNoAllocMaxElems = int64_t(1) << 33;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device, looked up once
// per device (host code cannot use the symbol itself as a device pointer).
acid_status scratch_address(void** out) {
  int dev = 0;
  ACID_CUDA(cudaGetDevice(&dev));
  ACID_REQUIRE(dev >= 0 && dev < kMaxDevices, ACID_ERR_UNSUPPORTED, "drift_noalloc: device index too large");
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    ACID_CUDA(cudaGetSymbolAddress(&p, g_noalloc_scratch));
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return ACID_OK;
}

}  // namespace
}  // namespace acid

using namespace acid;

extern "C" acid_status acid_drift_signal_noalloc(const void* prev, const void* cur, int64_t n, int32_t dtype,
                                                 double* out_rel_l1, double* out_sums, acid_stream_t stream) {
  clear_error();
  ACID_REQUIRE(dtype == ACID_BF16 || dtype == ACID_FP32, ACID_ERR_INVALID_ARG, "drift_noalloc: unknown dtype");
  ACID_REQUIRE(n >= 0, ACID_ERR_INVALID_ARG, "drift_noalloc: n must be >= 0");
  ACID_REQUIRE(n <= kNoAllocMaxElems, ACID_ERR_UNSUPPORTED,
               "drift_noalloc: n = " + std::to_string(n) + " exceeds the maximum of " +
                   std::to_string(kNoAllocMaxElems) + " elements; use acid_drift_signal with a workspace");
  ACID_REQUIRE(out_rel_l1 != nullptr, ACID_ERR_INVALID_ARG, "drift_noalloc: out_rel_l1 is null");
  ACID_REQUIRE(n == 0 || (prev && cur), ACID_ERR_INVALID_ARG, "drift_noalloc: null input");
  ACID_REQUIRE(n == 0 || (aligned(prev, 16) && aligned(cur, 16)), ACID_ERR_UNSUPPORTED,
               "drift_noalloc: inputs must be 16-byte aligned");
  const size_t part_bytes = drift_workspace_bytes(n);
  ACID_REQUIRE(part_bytes + 3 * sizeof(double) <= kNoAllocScratchBytes, ACID_ERR_UNSUPPORTED,
               "drift_noalloc: scratch array too small for this build");
  void* scratch = nullptr;
  ACID_TRY(scratch_address(&scratch));
  cudaStream_t s = (cudaStream_t)stream;
  double* result = reinterpret_cast<double*>(static_cast<uint8_t*>(scratch) + part_bytes);
  // Every partial slot the final pass reads is written earlier in the same
  // call, and the results are overwritten, so nothing needs clearing here.
  if (n == 0) {
    ACID_CUDA(cudaMemsetAsync(result, 0, 3 * sizeof(double), s));
  } else {
    ACID_TRY(drift_launch(dtype, prev, cur, nullptr, nullptr, n, result, scratch, part_bytes, s));
  }
  const bool rel_dev = is_device_pointer(out_rel_l1);
  const bool sums_dev = out_sums ? is_device_pointer(out_sums) : true;
  if (rel_dev) ACID_CUDA(cudaMemcpyAsync(out_rel_l1, result, sizeof(double), cudaMemcpyDeviceToDevice, s));
  if (out_sums && sums_dev)
    ACID_CUDA(cudaMemcpyAsync(out_sums, result + 1, 2 * sizeof(double), cudaMemcpyDeviceToDevice, s));
  if (!rel_dev || !sums_dev) {
    double h[3];
    ACID_CUDA(cudaMemcpyAsync(h, result, sizeof(h), cudaMemcpyDeviceToHost, s));
    ACID_CUDA(cudaStreamSynchronize(s));
    if (!rel_dev) *out_rel_l1 = h[0];
    if (out_sums && !sums_dev) {
      out_sums[0] = h[1];
      out_sums[1] = h[2];
    }
  }
  return ACID_OK;
}
