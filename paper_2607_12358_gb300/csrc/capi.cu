// C-ABI entry points for the drift signal and cache apply, plus the
// library-wide status plumbing.
#include <math.h>

#include <atomic>
#include <mutex>
#include <string>
#include <vector>

#include "common.cuh"
#include "internal.h"

namespace acid {

unsigned int take_device_error_gemm();
unsigned int take_device_error_attention();
BoundsRecord take_bounds_elementwise();
BoundsRecord take_bounds_gemm();
BoundsRecord take_bounds_attention();

namespace {
thread_local std::string t_last_error;

std::atomic<long long> g_launches{0};

struct ProfRec {
  cudaEvent_t a = nullptr, b = nullptr;
  int kind = 0;
  double work = 0.0;
};
std::mutex g_prof_mu;
bool g_prof_on = false;
std::vector<ProfRec> g_prof;
}  // namespace

void set_error(const std::string& msg) { t_last_error = msg; }
void clear_error() { t_last_error.clear(); }
void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

ProfScope::ProfScope(int kind, double work, cudaStream_t s) : s_(s) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  if (!g_prof_on) return;
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &cap) != cudaSuccess || cap != cudaStreamCaptureStatusNone) return;  // not in graphs
  ProfRec r;
  r.kind = kind;
  r.work = work;
  if (cudaEventCreate(&r.a) != cudaSuccess || cudaEventCreate(&r.b) != cudaSuccess) return;
  cudaEventRecord(r.a, s);
  slot_ = (int)g_prof.size();
  g_prof.push_back(r);
}

ProfScope::~ProfScope() {
  if (slot_ < 0) return;
  std::lock_guard<std::mutex> lk(g_prof_mu);
  if (slot_ < (int)g_prof.size()) cudaEventRecord(g_prof[slot_].b, s_);
}

static void prof_clear() {
  for (auto& r : g_prof) {
    if (r.a) cudaEventDestroy(r.a);
    if (r.b) cudaEventDestroy(r.b);
  }
  g_prof.clear();
}

bool is_device_pointer(const void* p) {
  cudaPointerAttributes attr;
  if (cudaPointerGetAttributes(&attr, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return attr.type == cudaMemoryTypeDevice || attr.type == cudaMemoryTypeManaged;
}

// Runs the drift reduction (and the fused apply when resid != null) and
// delivers the results to device or host outputs.
static acid_status drift_entry(const void* prev, const void* cur, const void* resid, void* out, int64_t n,
                               int32_t dtype, double* out_rel, double* out_sums, void* ws, size_t ws_bytes,
                               cudaStream_t s) {
  ACID_REQUIRE(dtype == ACID_BF16 || dtype == ACID_FP32, ACID_ERR_INVALID_ARG, "drift: unknown dtype");
  ACID_REQUIRE(n >= 0, ACID_ERR_INVALID_ARG, "drift: n must be >= 0");
  ACID_REQUIRE(out_rel != nullptr, ACID_ERR_INVALID_ARG, "drift: out_rel_l1 is null");
  ACID_REQUIRE(n == 0 || (prev && cur), ACID_ERR_INVALID_ARG, "drift: null input");
  ACID_REQUIRE(n == 0 || (aligned(prev, 16) && aligned(cur, 16)), ACID_ERR_UNSUPPORTED,
               "drift: inputs must be 16-byte aligned");
  if (resid) {
    ACID_REQUIRE(n == 0 || out != nullptr, ACID_ERR_INVALID_ARG, "drift_apply: out is null");
    ACID_REQUIRE(n == 0 || (aligned(resid, 16) && aligned(out, 16)), ACID_ERR_UNSUPPORTED,
                 "drift_apply: residual and output must be 16-byte aligned");
  }
  ACID_REQUIRE(ws != nullptr && aligned(ws, 16), ACID_ERR_WORKSPACE, "drift: workspace null or not 16-byte aligned");
  const size_t need = drift_workspace_bytes(n) + 64;
  ACID_REQUIRE(ws_bytes >= need, ACID_ERR_WORKSPACE, "drift: workspace too small (need " + std::to_string(need) + ")");
  double* result = reinterpret_cast<double*>(static_cast<uint8_t*>(ws) + drift_workspace_bytes(n));
  if (n == 0) {
    ACID_CUDA(cudaMemsetAsync(result, 0, 3 * sizeof(double), s));
  } else {
    ACID_TRY(drift_launch(dtype, prev, cur, resid, out, n, result, ws, drift_workspace_bytes(n), s));
  }
  const bool rel_dev = is_device_pointer(out_rel);
  const bool sums_dev = out_sums ? is_device_pointer(out_sums) : true;
  if (rel_dev) ACID_CUDA(cudaMemcpyAsync(out_rel, result, sizeof(double), cudaMemcpyDeviceToDevice, s));
  if (out_sums && sums_dev)
    ACID_CUDA(cudaMemcpyAsync(out_sums, result + 1, 2 * sizeof(double), cudaMemcpyDeviceToDevice, s));
  if (!rel_dev || !sums_dev) {
    double h[3];
    ACID_CUDA(cudaMemcpyAsync(h, result, sizeof(h), cudaMemcpyDeviceToHost, s));
    ACID_CUDA(cudaStreamSynchronize(s));
    if (!rel_dev) *out_rel = h[0];
    if (out_sums && !sums_dev) {
      out_sums[0] = h[1];
      out_sums[1] = h[2];
    }
  }
  return ACID_OK;
}

}  // namespace acid

using namespace acid;

extern "C" const char* acid_last_error(void) { return t_last_error.c_str(); }

extern "C" const char* acid_version(void) { return "acid-gb300 0.1 (sm_103a)"; }

namespace acid {
namespace {
// One thread waits on an mbarrier that no thread arrives on, through the
// kernels' bounded wait with a short budget: the wait runs out, raises this
// unit's device flag and the kernel returns.
__global__ void wait_selftest_kernel(long long limit) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    mbar_fence_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) (void)mbar_wait_limit(&bar, 0, limit);
}

// Evaluates one index check one past the end of an extent of n, with no
// memory access behind it: a debug build records {kSiteSelftest, n, n}.
__global__ void bounds_selftest_kernel(long long n, int* sink) {
  if (threadIdx.x == 0 && !ACID_IN_BOUNDS(kSiteSelftest, n, n) && sink != nullptr) *sink = 1;
}
}  // namespace
ACID_DEVICE_FLAG_READER(take_device_error_capi)
ACID_BOUNDS_READER(take_bounds_capi)
}  // namespace acid

extern "C" acid_status acid_bounds_report(int32_t* checked, int64_t* site, int64_t* index, int64_t* extent) {
  clear_error();
  ACID_REQUIRE(checked && site && index && extent, ACID_ERR_INVALID_ARG, "acid_bounds_report: null argument");
  ACID_CUDA(cudaDeviceSynchronize());
  const BoundsRecord recs[4] = {take_bounds_elementwise(), take_bounds_gemm(), take_bounds_attention(),
                                take_bounds_capi()};
  *checked = kBoundsChecked ? 1 : 0;
  *site = *index = *extent = 0;
  for (const BoundsRecord& r : recs) {
    ACID_REQUIRE(r.site >= 0, ACID_ERR_CUDA, "acid_bounds_report: record not readable");
    if (r.site != 0 && *site == 0) {
      *site = r.site;
      *index = r.index;
      *extent = r.extent;
    }
  }
  return ACID_OK;
}

extern "C" acid_status acid_selftest_bounds(acid_stream_t stream) {
  clear_error();
  cudaStream_t s = (cudaStream_t)stream;
  bounds_selftest_kernel<<<1, 32, 0, s>>>(1000, nullptr);
  ACID_CHECK_LAUNCH();
  ACID_CUDA(cudaStreamSynchronize(s));
  return ACID_OK;
}

extern "C" acid_status acid_selftest_wait_timeout(int64_t budget_cycles, acid_stream_t stream) {
  clear_error();
  ACID_REQUIRE(budget_cycles >= 1000 && budget_cycles <= 10000000000LL, ACID_ERR_INVALID_ARG,
               "acid_selftest_wait_timeout: budget must be 1e3..1e10 cycles");
  cudaStream_t s = (cudaStream_t)stream;
  wait_selftest_kernel<<<1, 32, 0, s>>>((long long)budget_cycles);
  ACID_CHECK_LAUNCH();
  ACID_CUDA(cudaStreamSynchronize(s));
  return ACID_OK;
}

extern "C" acid_status acid_check_device_error(void) {
  clear_error();
  ACID_CUDA(cudaDeviceSynchronize());
  const unsigned int flag = take_device_error_gemm() | take_device_error_attention() | take_device_error_capi();
  if (flag) {
    set_error("a bounded device-side wait timed out");
    return ACID_ERR_TIMEOUT;
  }
  return ACID_OK;
}

extern "C" acid_status acid_drift_workspace_size(int64_t n, size_t* bytes) {
  clear_error();
  ACID_REQUIRE(bytes != nullptr && n >= 0, ACID_ERR_INVALID_ARG, "acid_drift_workspace_size: bad argument");
  *bytes = drift_workspace_bytes(n) + 64;
  return ACID_OK;
}

extern "C" acid_status acid_temni_drift(const float* h_prev, const float* h_cur, const float* mod_prev,
                                        const float* mod_cur, int64_t rows, int32_t d, float eps, double* out_rel,
                                        double* out_sums, void* ws, size_t ws_bytes, acid_stream_t stream) {
  clear_error();
  cudaStream_t s = (cudaStream_t)stream;
  ACID_REQUIRE(rows >= 0 && d > 0, ACID_ERR_INVALID_ARG, "temni_drift: rows must be >= 0 and d > 0");
  ACID_REQUIRE(d % 8 == 0 && d <= 3072, ACID_ERR_UNSUPPORTED, "temni_drift: d must be a multiple of 8, <= 3072");
  ACID_REQUIRE(out_rel != nullptr, ACID_ERR_INVALID_ARG, "temni_drift: out_rel_l1 is null");
  ACID_REQUIRE(rows == 0 || (h_prev && h_cur && mod_prev && mod_cur), ACID_ERR_INVALID_ARG, "temni_drift: null input");
  ACID_REQUIRE(rows == 0 || (aligned(h_prev, 16) && aligned(h_cur, 16) && aligned(mod_prev, 16) && aligned(mod_cur, 16)),
               ACID_ERR_UNSUPPORTED, "temni_drift: inputs must be 16-byte aligned");
  ACID_REQUIRE(ws != nullptr && aligned(ws, 16), ACID_ERR_WORKSPACE, "temni_drift: workspace null or not 16-byte aligned");
  const int64_t n = rows * (int64_t)d;
  const size_t need = drift_workspace_bytes(n) + 64;
  ACID_REQUIRE(ws_bytes >= need, ACID_ERR_WORKSPACE,
               "temni_drift: workspace too small (need " + std::to_string(need) + ")");
  double* result = reinterpret_cast<double*>(static_cast<uint8_t*>(ws) + drift_workspace_bytes(n));
  if (rows == 0) {
    ACID_CUDA(cudaMemsetAsync(result, 0, 3 * sizeof(double), s));
  } else {
    ACID_TRY(temni_drift(h_cur, h_prev, mod_cur, mod_prev, nullptr, 1, rows, d, eps, result, ws,
                         drift_workspace_bytes(n), s));
  }
  const bool rel_dev = is_device_pointer(out_rel);
  const bool sums_dev = out_sums ? is_device_pointer(out_sums) : true;
  if (rel_dev) ACID_CUDA(cudaMemcpyAsync(out_rel, result, sizeof(double), cudaMemcpyDeviceToDevice, s));
  if (out_sums && sums_dev)
    ACID_CUDA(cudaMemcpyAsync(out_sums, result + 1, 2 * sizeof(double), cudaMemcpyDeviceToDevice, s));
  if (!rel_dev || !sums_dev) {
    double h[3];
    ACID_CUDA(cudaMemcpyAsync(h, result, sizeof(h), cudaMemcpyDeviceToHost, s));
    ACID_CUDA(cudaStreamSynchronize(s));
    if (!rel_dev) *out_rel = h[0];
    if (out_sums && !sums_dev) {
      out_sums[0] = h[1];
      out_sums[1] = h[2];
    }
  }
  return ACID_OK;
}

extern "C" acid_status acid_drift_signal(const void* prev, const void* cur, int64_t n, int32_t dtype,
                                         double* out_rel_l1, double* out_sums, void* workspace, size_t workspace_bytes,
                                         acid_stream_t stream) {
  clear_error();
  return drift_entry(prev, cur, nullptr, nullptr, n, dtype, out_rel_l1, out_sums, workspace, workspace_bytes,
                     (cudaStream_t)stream);
}

extern "C" acid_status acid_drift_apply(const void* prev, const void* cur, const void* cached_residual, void* out,
                                        int64_t n, int32_t dtype, double* out_rel_l1, double* out_sums,
                                        void* workspace, size_t workspace_bytes, acid_stream_t stream) {
  clear_error();
  ACID_REQUIRE(n == 0 || cached_residual != nullptr, ACID_ERR_INVALID_ARG, "acid_drift_apply: residual is null");
  return drift_entry(prev, cur, cached_residual, out, n, dtype, out_rel_l1, out_sums, workspace, workspace_bytes,
                     (cudaStream_t)stream);
}

extern "C" acid_status acid_cache_apply(const void* x, const void* cached_residual, void* out, int64_t n,
                                        int32_t dtype, acid_stream_t stream) {
  clear_error();
  ACID_REQUIRE(dtype == ACID_BF16 || dtype == ACID_FP32, ACID_ERR_INVALID_ARG, "acid_cache_apply: unknown dtype");
  ACID_REQUIRE(n >= 0, ACID_ERR_INVALID_ARG, "acid_cache_apply: n must be >= 0");
  if (n == 0) return ACID_OK;
  ACID_REQUIRE(x && cached_residual && out, ACID_ERR_INVALID_ARG, "acid_cache_apply: null pointer");
  ACID_REQUIRE(aligned(x, 16) && aligned(cached_residual, 16) && aligned(out, 16), ACID_ERR_UNSUPPORTED,
               "acid_cache_apply: pointers must be 16-byte aligned");
  return add_same(dtype, x, cached_residual, out, n, (cudaStream_t)stream);
}

extern "C" acid_status acid_linear_forward(int32_t dtype, const void* A, int64_t lda, int64_t M, int32_t K,
                                           const void* W, const float* bias, int32_t N, void* out, int64_t ldo,
                                           int32_t epilogue, const float* gate, const void* residual, int64_t ldr,
                                           int32_t out_fp32, acid_stream_t stream) {
  clear_error();
  ACID_REQUIRE(dtype == ACID_BF16 || dtype == ACID_FP32, ACID_ERR_INVALID_ARG, "acid_linear_forward: unknown dtype");
  ACID_REQUIRE(epilogue == ACID_EPI_BIAS || epilogue == ACID_EPI_GELU || epilogue == ACID_EPI_GATED_RES ||
                   epilogue == ACID_EPI_RES,
               ACID_ERR_INVALID_ARG, "acid_linear_forward: unknown epilogue");
  ACID_REQUIRE(epilogue != ACID_EPI_GATED_RES || gate != nullptr, ACID_ERR_INVALID_ARG,
               "acid_linear_forward: gated residual needs a gate");
  ACID_REQUIRE(lda >= K && ldo >= N, ACID_ERR_INVALID_ARG, "acid_linear_forward: row stride smaller than the row");
  Epilogue e;
  e.kind = epilogue;
  e.bias = bias;
  e.gate_video = gate;
  e.residual = residual;
  e.ldr = ldr;
  e.out_fp32 = out_fp32 != 0 || dtype == ACID_FP32;
  e.res_fp32 = e.out_fp32;  // the residual has the output's dtype
  return linear_forward(dtype, A, lda, M, K, W, N, out, ldo, e, (cudaStream_t)stream);
}

extern "C" acid_status acid_attention_forward(int32_t dtype, const void* q, int64_t ldq, const void* k, int64_t ldk,
                                              const void* v, int64_t ldv, void* out, int64_t ldo, int64_t nq,
                                              int64_t nk, int32_t heads, int32_t head_dim, void* workspace,
                                              size_t workspace_bytes, acid_stream_t stream) {
  clear_error();
  ACID_REQUIRE(workspace == nullptr || aligned(workspace, 16), ACID_ERR_WORKSPACE,
               "acid_attention_forward: workspace must be 16-byte aligned");
  ACID_REQUIRE(dtype == ACID_BF16 || dtype == ACID_FP32, ACID_ERR_INVALID_ARG, "acid_attention_forward: unknown dtype");
  ACID_REQUIRE(heads > 0 && head_dim > 0, ACID_ERR_INVALID_ARG, "acid_attention_forward: bad heads / head_dim");
  const int64_t w = (int64_t)heads * head_dim;
  ACID_REQUIRE(ldq >= w && ldk >= w && ldv >= w && ldo >= w, ACID_ERR_INVALID_ARG,
               "acid_attention_forward: row stride smaller than heads * head_dim");
  ACID_REQUIRE(nq >= 0 && nk >= 1, ACID_ERR_INVALID_ARG, "acid_attention_forward: need nq >= 0 and nk >= 1");
  AttnArgs a;
  a.q = q; a.ldq = ldq;
  a.k = k; a.ldk = ldk;
  a.v = v; a.ldv = ldv;
  a.out = out; a.ldo = ldo;
  a.nq = nq; a.nk = nk;
  a.heads = heads; a.head_dim = head_dim;
  a.part = workspace;
  a.part_bytes = workspace ? workspace_bytes : 0;
  return attention_forward(dtype, a, (cudaStream_t)stream);
}

extern "C" acid_status acid_attention_workspace_size(int32_t head_dim, size_t* bytes) {
  clear_error();
  ACID_REQUIRE(bytes != nullptr && head_dim > 0, ACID_ERR_INVALID_ARG, "acid_attention_workspace_size: bad argument");
  *bytes = attn_part_bytes(head_dim);
  return ACID_OK;
}

extern "C" acid_status acid_layernorm_mod(int32_t x_dtype, const void* x, int32_t y_dtype, void* y, int64_t rows,
                                          int32_t d, const float* shift, const float* scale, float eps,
                                          acid_stream_t stream) {
  clear_error();
  ACID_REQUIRE((x_dtype == ACID_BF16 || x_dtype == ACID_FP32) && (y_dtype == ACID_BF16 || y_dtype == ACID_FP32),
               ACID_ERR_INVALID_ARG, "acid_layernorm_mod: unknown dtype");
  ACID_REQUIRE(rows >= 0 && d > 0, ACID_ERR_INVALID_ARG, "acid_layernorm_mod: bad shape");
  ACID_REQUIRE((shift == nullptr) == (scale == nullptr), ACID_ERR_INVALID_ARG,
               "acid_layernorm_mod: shift and scale must both be given or both be NULL");
  if (rows == 0) return ACID_OK;
  ACID_REQUIRE(x && y && aligned(x, 16) && aligned(y, 16), ACID_ERR_UNSUPPORTED,
               "acid_layernorm_mod: x and y must be 16-byte aligned device pointers");
  return ln_mod(x_dtype, x, y_dtype, y, rows, d, shift, scale, nullptr, nullptr, 0, eps, (cudaStream_t)stream);
}

extern "C" int64_t acid_launch_count(void) { return (int64_t)g_launches.load(); }

extern "C" acid_status acid_profile_enable(int32_t on) {
  clear_error();
  std::lock_guard<std::mutex> lk(g_prof_mu);
  if (on) {
    ACID_CUDA(cudaDeviceSynchronize());
    prof_clear();
  }
  g_prof_on = on != 0;
  return ACID_OK;
}

extern "C" acid_status acid_profile_read(int32_t kind, int64_t* launches, double* total_ms, double* work) {
  clear_error();
  ACID_REQUIRE(kind >= 0 && kind < PROF_KINDS && launches && total_ms && work, ACID_ERR_INVALID_ARG,
               "acid_profile_read: bad argument");
  ACID_CUDA(cudaDeviceSynchronize());
  std::lock_guard<std::mutex> lk(g_prof_mu);
  int64_t n = 0;
  double ms = 0.0, wk = 0.0;
  for (auto& r : g_prof) {
    if (r.kind != kind) continue;
    float t = 0.f;
    ACID_CUDA(cudaEventElapsedTime(&t, r.a, r.b));
    ++n;
    ms += t;
    wk += r.work;
  }
  *launches = n;
  *total_ms = ms;
  *work = wk;
  return ACID_OK;
}
