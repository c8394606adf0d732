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
#include <cudaTypedefs.h>

#include <mutex>
#include <string>

#include "common.cuh"
#include "internal.h"

namespace acid {

bool is_device_pointer(const void* p);

namespace {

constexpr size_t kNoAllocScratchBytes = 16 * 1024;
// Largest element count accepted.  The reduction runs a fixed grid of 608
// blocks of 256 threads, and each thread sums |cur - prev| and |prev| into
// two fp32 accumulators each, so at n = 2^31 an accumulator adds at most
// 2^31 / (608 * 256 * 2) < 6,900 terms.  Summing non-negative terms one by one
// in fp32 has a relative error of at most (terms - 1) * 2^-24 < 4.2e-4, and
// the fp64 stages after it add nothing at that scale, so the ratio of the two
// sums stays within about 8.4e-4 of exact even in the worst case: inside the
// 1e-3 drift tolerance.  (The expected error, which grows with the square
// root of the term count, is far smaller.)
constexpr int64_t kNoAllocMaxElems = int64_t(1) << 31;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_mu;
struct ScratchSlot {
  CUcontext ctx;  // context the address belongs to
  void* addr;
};
ScratchSlot g_slot[kMaxDevices] = {};

// cuCtxGetCurrent through the runtime's driver entry-point query (the library
// does not link the driver API).
PFN_cuCtxGetCurrent_v4000 ctx_get_current() {
  static PFN_cuCtxGetCurrent_v4000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p);
  });
  return fn;
}

// Device address of the scratch array in the current device's context (host
// code cannot use the symbol itself as a device pointer).  Looked up once per
// device and looked up again if that device's context has changed since, as
// after cudaDeviceReset, which reloads the module at a new address.
acid_status scratch_address(void** out) {
  int dev = 0;
  ACID_CUDA(cudaGetDevice(&dev));
  ACID_REQUIRE(dev >= 0 && dev < kMaxDevices, ACID_ERR_UNSUPPORTED, "drift_noalloc: device index too large");
  auto get_ctx = ctx_get_current();
  ACID_REQUIRE(get_ctx != nullptr, ACID_ERR_CUDA, "drift_noalloc: cuCtxGetCurrent entry point unavailable");
  std::lock_guard<std::mutex> lk(g_mu);
  ScratchSlot& sl = g_slot[dev];
  CUcontext ctx = nullptr;
  if (sl.addr != nullptr && get_ctx(&ctx) == CUDA_SUCCESS && ctx == sl.ctx) {
    *out = sl.addr;
    return ACID_OK;
  }
  // first call on this device, or its context was replaced: the lookup also
  // makes the device's primary context current, so the context is read after it
  void* p = nullptr;
  ACID_CUDA(cudaGetSymbolAddress(&p, g_noalloc_scratch));
  ctx = nullptr;
  ACID_REQUIRE(get_ctx(&ctx) == CUDA_SUCCESS && ctx != nullptr, ACID_ERR_CUDA, "drift_noalloc: no current context");
  sl.ctx = ctx;
  sl.addr = p;
  *out = p;
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
