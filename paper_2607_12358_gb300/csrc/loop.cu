// The sampling loop of Algorithm 1 (Sec. 3.3) around an Euler flow-matching
// sampler, with TeaCache, EasyCache or DiCache (Sec. 2) as the wrapped
// method, with or without classifier-free guidance.  All tensor work runs in
// the library's kernels.  The host-driven loop keeps only the scalar
// controller state and takes one decision per non-warmup step from the drift
// value it reads back; the graph-launched loop takes it on the device.
#include <math.h>
#include <string.h>

#include <cmath>

#include <string>
#include <utility>

#include "block.h"
#include "common.cuh"
#include "internal.h"

namespace acid {

namespace {

size_t es(int dt) { return dt == ACID_BF16 ? 2 : 4; }

struct LoopWs {
  float* sinus;
  float* temb_h;
  float* temb;
  float* mod0[2];   // block 0 shift / scale (TEMNI) of the even / odd steps
  float* fmod;      // final layer shift / scale
  uint8_t* tokens;  // [N, P] fp32 patch vectors, or [N, 2P] bf16 hi / lo parts (patch_split)
  float* h_in[2];   // [N, d] patch embedding (fp32) of the even / odd steps
  float* temni[2];  // [N, d] DiCache probe features of the even / odd steps
  float* resid;     // [N, d] TeaCache residual H_out - H_in
  uint8_t* xbuf;    // [L + N, d] block-stack state (model dtype)
  uint8_t* text;    // [L, d] text context / text tokens (model dtype)
  uint8_t* ctx_kv;  // WAN with text: [blocks, L, 2d] cross-attention keys and values (model dtype)
  uint8_t* y;       // [N, d] final LayerNorm output
  float* vtok;      // [N, P] final layer output
  float* v[2];      // latent-sized velocity, current / previous (EasyCache)
  float* x_prev;    // latent-sized previous input (EasyCache)
  float* offset;    // latent-sized v_c - x_c (EasyCache)
  // DiCache: probe features of the current / previous step are temni[], the
  // deep part D_1 = H_out - P of the last computed step is resid
  float* dc_p1;     // [N, d] probe features of the last computed step
  float* dc_p2;     // [N, d] probe features of the computed step before
  float* dc_d2;     // [N, d] deep part of the computed step before
  int* dc_count;    // computed steps cached (0, 1, 2)
  double* dres;     // [8] device drift results
  uint8_t* drift_ws;
  unsigned int* drift_done;  // TEMNI drift: CTAs finished (zero between launches)
  // bf16 models with P % 8 == 0: the patch embedding runs on tensor cores
  // against the patch weights repeated along K, [d, 2P] bf16
  bool patch_split;
  uint8_t* patch_w2;
  float2* rope;
  uint8_t* block_base;
  // device-side loop state for graph-launched generations
  struct DevLoop* dev;      // controller state and configuration
  double* sig;              // [kMaxGraphSteps + 1] noise levels
  int8_t* forced;           // [kMaxGraphSteps]
  double* tau_sched;        // [kMaxGraphSteps] fixed thresholds (NaN: delta rule)
  acid_step_log* dlog;      // [kMaxGraphSteps]
  size_t bytes;
};

constexpr int kMaxGraphSteps = 1024;

// Algorithm 1's state and inputs as the device controller sees them.
struct DevLoop {
  int step;  // first member: the kernels read the step index through &dev->step
  int have_prev, have_cache, have_rate;
  int n_steps, warmup, method, force_last, use_forced, use_tau_sched;
  int compute;
  double sigma_acc, s_prev, k_rate;
  double tau_low, tau_high, delta;
  double latent_n;
  int poly_n;
  double poly[8];
};

struct Shape {
  int64_t N, L, P, latent;
  int d;
};

Shape shape_of(const acid_model& m) {
  Shape s;
  const int64_t gf = m.latent_f / m.pt, gh = m.latent_h / m.ph, gw = m.latent_w / m.pw;
  s.N = gf * gh * gw;
  s.L = m.block.n_text;
  s.P = (int64_t)m.latent_c * m.pt * m.ph * m.pw;
  s.latent = (int64_t)m.latent_c * m.latent_f * m.latent_h * m.latent_w;
  s.d = m.block.d;
  return s;
}

acid_block_desc desc_for(const acid_model& m, int i) {
  acid_block_desc d = m.block;
  if (m.block.kind == ACID_BLOCK_HV_DUAL || m.block.kind == ACID_BLOCK_HV_SINGLE)
    d.kind = i < m.n_blocks ? ACID_BLOCK_HV_DUAL : ACID_BLOCK_HV_SINGLE;
  return d;
}

int total_blocks(const acid_model& m) {
  const bool hv = m.block.kind == ACID_BLOCK_HV_DUAL || m.block.kind == ACID_BLOCK_HV_SINGLE;
  return m.n_blocks + (hv ? m.n_single : 0);
}

LoopWs loop_layout(const acid_model& m, void* base) {
  Bump b{static_cast<uint8_t*>(base)};
  const Shape s = shape_of(m);
  const int dt = m.block.dtype;
  LoopWs w;
  w.sinus = b.take<float>(m.time_freq_dim);
  w.temb_h = b.take<float>(s.d);
  w.temb = b.take<float>(s.d);
  w.mod0[0] = b.take<float>(2 * s.d);
  w.mod0[1] = b.take<float>(2 * s.d);
  w.fmod = b.take<float>(2 * s.d);
  w.tokens = b.take<uint8_t>(s.N * s.P * sizeof(float));
  w.h_in[0] = b.take<float>(s.N * s.d);
  w.h_in[1] = b.take<float>(s.N * s.d);
  w.temni[0] = b.take<float>(s.N * s.d);
  w.temni[1] = b.take<float>(s.N * s.d);
  w.resid = b.take<float>(s.N * s.d);
  const int64_t xrows = m.block.kind == ACID_BLOCK_WAN ? s.N : s.N + s.L;
  w.xbuf = b.take<uint8_t>(xrows * s.d * es(dt));
  w.text = b.take<uint8_t>(std::max<int64_t>(s.L, 1) * s.d * es(dt));
  const bool wan_text = m.block.kind == ACID_BLOCK_WAN && s.L > 0;
  w.ctx_kv = b.take<uint8_t>(wan_text ? (size_t)total_blocks(m) * s.L * 2 * s.d * es(dt) : 0);
  w.y = b.take<uint8_t>(s.N * s.d * es(dt));
  w.vtok = b.take<float>(s.N * s.P);
  w.v[0] = b.take<float>(s.latent);
  w.v[1] = b.take<float>(s.latent);
  w.x_prev = b.take<float>(s.latent);
  w.offset = b.take<float>(s.latent);
  w.dc_p1 = b.take<float>(s.N * s.d);
  w.dc_p2 = b.take<float>(s.N * s.d);
  w.dc_d2 = b.take<float>(s.N * s.d);
  w.dc_count = b.take<int>(1);
  w.dres = b.take<double>(8);
  w.drift_ws = b.take<uint8_t>(drift_workspace_bytes(0));
  w.drift_done = b.take<unsigned int>(1);
  w.patch_split = dt == ACID_BF16 && s.P % 8 == 0;
  w.patch_w2 = b.take<uint8_t>(w.patch_split ? (size_t)s.d * 2 * s.P * 2 : 0);
  RopeTable rt = rope_layout(m.block.grid_f, m.block.grid_h, m.block.grid_w, m.block.d / std::max(1, m.block.heads));
  w.rope = b.take<float2>((size_t)rt.elems());
  // one block workspace, sized for the larger of the first and last block kinds
  size_t blk = block_ws_layout(desc_for(m, 0), nullptr).bytes;
  blk = std::max(blk, block_ws_layout(desc_for(m, total_blocks(m) - 1), nullptr).bytes);
  w.block_base = b.take<uint8_t>(blk);
  w.dev = b.take<DevLoop>(1);
  w.sig = b.take<double>(kMaxGraphSteps + 1);
  w.forced = b.take<int8_t>(kMaxGraphSteps);
  w.tau_sched = b.take<double>(kMaxGraphSteps);
  w.dlog = b.take<acid_step_log>(kMaxGraphSteps);
  w.bytes = b.off + 1024;
  return w;
}

acid_status validate_model(const acid_model& m) {
  ACID_REQUIRE(m.blocks != nullptr && m.n_blocks > 0, ACID_ERR_INVALID_ARG, "model: no blocks");
  ACID_TRY(validate_block_desc(m.block));
  ACID_REQUIRE(m.latent_c > 0 && m.pt > 0 && m.ph > 0 && m.pw > 0 && m.latent_f % m.pt == 0 &&
                   m.latent_h % m.ph == 0 && m.latent_w % m.pw == 0,
               ACID_ERR_INVALID_ARG, "model: latent shape not divisible by the patch size");
  ACID_REQUIRE(m.block.grid_f == m.latent_f / m.pt && m.block.grid_h == m.latent_h / m.ph &&
                   m.block.grid_w == m.latent_w / m.pw,
               ACID_ERR_INVALID_ARG, "model: block grid does not match latent / patch");
  ACID_REQUIRE(m.time_freq_dim > 0 && m.time_freq_dim % 16 == 0, ACID_ERR_INVALID_ARG,
               "model: time_freq_dim must be a positive multiple of 16");
  ACID_REQUIRE(m.patch.w && m.time1.w && m.time2.w && m.final_mod.w && m.final_out.w, ACID_ERR_INVALID_ARG,
               "model: missing patch / time / final weights");
  const int64_t P = (int64_t)m.latent_c * m.pt * m.ph * m.pw;
  ACID_REQUIRE(P % 64 == 0 || m.block.dtype == ACID_FP32, ACID_ERR_UNSUPPORTED,
               "model bf16: patch dimension C*pt*ph*pw must be a multiple of 64");
  if (m.block.kind == ACID_BLOCK_WAN && m.block.n_text > 0)
    ACID_REQUIRE(m.text.w != nullptr && m.d_text > 0 && m.d_text % 64 == 0, ACID_ERR_INVALID_ARG,
                 "model: WAN with text needs the text projection (d_text % 64 == 0)");
  if (m.block.kind != ACID_BLOCK_WAN)
    ACID_REQUIRE(m.d_text == m.block.d || m.block.n_text == 0, ACID_ERR_INVALID_ARG,
                 "model: joint text tokens must be given at width d");
  for (int i = 0; i < total_blocks(m); ++i) ACID_TRY(validate_block_weights(desc_for(m, i), m.blocks[i]));
  return ACID_OK;
}

acid_status validate_cfg(const acid_loop_cfg& c) {
  ACID_REQUIRE(c.n_steps > 0 && c.warmup >= 0, ACID_ERR_INVALID_ARG, "loop: n_steps must be > 0, warmup >= 0");
  ACID_REQUIRE(c.method == ACID_METHOD_TEACACHE || c.method == ACID_METHOD_EASYCACHE ||
                   c.method == ACID_METHOD_DICACHE,
               ACID_ERR_INVALID_ARG, "loop: unknown method");
  ACID_REQUIRE(c.method != ACID_METHOD_DICACHE || c.probe_blocks >= 1, ACID_ERR_INVALID_ARG,
               "loop: DiCache needs probe_blocks >= 1");
  ACID_REQUIRE(c.method == ACID_METHOD_EASYCACHE || c.warmup >= 1, ACID_ERR_INVALID_ARG,
               "loop: TeaCache and DiCache need warmup >= 1 (the first signal compares two steps)");
  ACID_REQUIRE(c.method != ACID_METHOD_EASYCACHE || c.warmup >= 2, ACID_ERR_INVALID_ARG,
               "loop: EasyCache needs warmup >= 2 (k is defined after two computed steps)");
  ACID_REQUIRE(c.shift > 0.0, ACID_ERR_INVALID_ARG, "loop: shift must be > 0");
  ACID_REQUIRE(c.signal_poly_n >= 0 && c.signal_poly_n <= 8 && (c.signal_poly_n == 0 || c.signal_poly != nullptr),
               ACID_ERR_INVALID_ARG, "loop: signal_poly_n must be 0..8 with coefficients given");
  return ACID_OK;
}

double sigma_at(const acid_loop_cfg& c, int i) {
  const double s = 1.0 - (double)i / c.n_steps;
  if (c.shift == 1.0) return s;
  return c.shift * s / (1.0 + (c.shift - 1.0) * s);
}

// Optional rescaling of the raw signal, s' = sum_j c_j s^j (Horner).
__host__ __device__ inline double rescale_signal(double s, const double* c, int n) {
  if (n <= 0) return s;
  double r = c[n - 1];
  for (int j = n - 2; j >= 0; --j) r = r * s + c[j];
  return r;
}

// One non-warmup step of Algorithm 1 on (Sigma, s_prev), shared by the host
// and device controllers: accumulate, pick the threshold from the signal's
// rate of change, compare, reset Sigma on compute; s_prev always updated.  tau_fix: a finite value replaces the threshold the
// delta rule would pick (a fixed threshold schedule, Sec. 3.2's transition
// experiment); NaN keeps the rule.  forced >= 0 replaces the decision.
// Returns true when the step computes.
__host__ __device__ inline bool algorithm1_step(double& sigma_acc, double& s_prev, int& have_prev, double s,
                                                double tau_low, double tau_high, double delta, double tau_fix,
                                                int forced, acid_step_log* lg) {
  sigma_acc += s;
  double tau, ds = NAN;
  if (have_prev) {
    ds = fabs(s - s_prev);
    tau = ds <= delta ? tau_high : tau_low;
  } else {
    tau = tau_low;
  }
  if (tau_fix == tau_fix) tau = tau_fix;
  const double seen = sigma_acc;
  bool skip = seen <= tau;
  if (forced >= 0) skip = forced == 0;
  if (!skip) sigma_acc = 0.0;
  s_prev = s;
  have_prev = 1;
  lg->signal = s;
  lg->dsignal = ds;
  lg->tau = tau;
  lg->sigma = seen;
  lg->forced = forced >= 0;
  return !skip;
}

bool controller_step(acid_loop_state& st, const acid_loop_cfg& c, int i, double s_raw, int forced,
                     acid_step_log* lg) {
  const double s = rescale_signal(s_raw, c.signal_poly, c.signal_poly_n);
  const double tau_fix = c.tau_schedule ? c.tau_schedule[i] : NAN;
  int have_prev = st.have_prev_signal;
  acid_step_log tmp;
  const bool compute = algorithm1_step(st.sigma_acc, st.s_prev, have_prev, s, c.tau_low, c.tau_high, c.delta,
                                       tau_fix, forced, lg ? lg : &tmp);
  st.have_prev_signal = have_prev;
  return compute;
}

double ratio_or_inf(double num, double den) {
  if (den == 0.0) return num == 0.0 ? 0.0 : INFINITY;
  return num / den;
}

acid_status read_results(double* host, const double* dev, int n, cudaStream_t s) {
  ACID_CUDA(cudaMemcpyAsync(host, dev, sizeof(double) * n, cudaMemcpyDeviceToHost, s));
  ACID_CUDA(cudaStreamSynchronize(s));
  return ACID_OK;
}

// Runs every block on the state in w.xbuf.
acid_status run_blocks(const acid_model& m, const LoopWs& w, cudaStream_t s, int b0 = 0, int b1 = -1) {
  const RopeTable base_rope = [&] {
    RopeTable t = rope_layout(m.block.grid_f, m.block.grid_h, m.block.grid_w, m.block.d / m.block.heads);
    t.table = w.rope;
    return t;
  }();
  const bool wan_text = m.block.kind == ACID_BLOCK_WAN && m.block.n_text > 0;
  const void* ctx = wan_text ? w.text : nullptr;
  const size_t kv_bytes = (size_t)m.block.n_text * 2 * m.block.d * es(m.block.dtype);
  if (b1 < 0) b1 = total_blocks(m);
  for (int i = b0; i < b1; ++i) {
    const acid_block_desc d = desc_for(m, i);
    const BlockWs bws = block_ws_layout(d, w.block_base);
    const void* kv = wan_text ? w.ctx_kv + i * kv_bytes : nullptr;
    ACID_TRY(block_forward_impl(d, w.xbuf, w.temb, ctx, kv, m.blocks[i], bws, &base_rope, s));
  }
  return ACID_OK;
}

// ---------------------------------------------------------------- DiCache
// After a computed step: D = H_out - P_t; the caches shift
// (P_2, D_2) <- (P_1, D_1), (P_1, D_1) <- (P_t, D); on the first computed
// step both slots get (P_t, D), so the trajectory term vanishes.
template <typename T>
__global__ void dicache_update_kernel(const T* __restrict__ h_out, const float* __restrict__ p_t, float* d1,
                                      float* d2, float* p1, float* p2, int64_t n, const int* count) {
  const int c = *count;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    const float p = p_t[i];
    const float d = io<T>::ld(h_out + i) - p;
    if (c >= 1) {
      d2[i] = d1[i];
      p2[i] = p1[i];
    } else {
      d2[i] = d;
      p2[i] = p;
    }
    d1[i] = d;
    p1[i] = p;
  }
}

__global__ void dicache_count_kernel(int* count) { *count = min(*count + 1, 2); }

// Reuse: H_out = P_t + D_1 + g (D_1 - D_2), g = sum|P_t - P_1| / sum|P_1 - P_2|
// (0 when the denominator is 0); the sums are read from device memory.
template <typename T>
__global__ void dicache_reuse_kernel(T* out, const float* __restrict__ p_t, const float* __restrict__ d1,
                                     const float* __restrict__ d2, int64_t n, const double* num, const double* den) {
  const double dn = *den;
  const float g = dn > 0.0 ? (float)(*num / dn) : 0.0f;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    const float a = d1[i];
    io<T>::st(out + i, p_t[i] + a + g * (a - d2[i]));
  }
}

int elem_grid(int64_t n) { return (int)std::min<int64_t>(152 * 16, std::max<int64_t>(1, (n + 255) / 256)); }

acid_status dicache_update(int dt, const void* h_out, const float* p_t, const LoopWs& w, int64_t n, cudaStream_t s) {
  if (dt == ACID_BF16)
    dicache_update_kernel<__nv_bfloat16><<<elem_grid(n), 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(h_out), p_t, w.resid, w.dc_d2, w.dc_p1, w.dc_p2, n, w.dc_count);
  else
    dicache_update_kernel<float><<<elem_grid(n), 256, 0, s>>>(static_cast<const float*>(h_out), p_t, w.resid,
                                                              w.dc_d2, w.dc_p1, w.dc_p2, n, w.dc_count);
  ACID_CHECK_LAUNCH();
  dicache_count_kernel<<<1, 1, 0, s>>>(w.dc_count);
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

// Reuse into out (the block-stack state's video rows, model dtype).  Uses
// w.dres[0..5] for the two trajectory sums.
acid_status dicache_reuse(int dt, void* out, const float* p_t, const LoopWs& w, int64_t n, cudaStream_t s) {
  ACID_TRY(drift_launch(ACID_FP32, w.dc_p1, p_t, nullptr, nullptr, n, w.dres, w.drift_ws, drift_workspace_bytes(0), s));
  ACID_TRY(drift_launch(ACID_FP32, w.dc_p2, w.dc_p1, nullptr, nullptr, n, w.dres + 3, w.drift_ws,
                        drift_workspace_bytes(0), s));
  if (dt == ACID_BF16)
    dicache_reuse_kernel<__nv_bfloat16><<<elem_grid(n), 256, 0, s>>>(static_cast<__nv_bfloat16*>(out), p_t, w.resid,
                                                                     w.dc_d2, n, w.dres + 1, w.dres + 4);
  else
    dicache_reuse_kernel<float><<<elem_grid(n), 256, 0, s>>>(static_cast<float*>(out), p_t, w.resid, w.dc_d2, n,
                                                            w.dres + 1, w.dres + 4);
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

// Final layer + unpatchify: v (optional) and the Euler update of the latent.
acid_status final_layer(const acid_model& m, const LoopWs& w, const void* h_out, float* v_out, float* latent,
                        float dsig, cudaStream_t s) {
  const Shape sh = shape_of(m);
  const int dt = m.block.dtype;
  ACID_TRY(gemv(dt, m.final_mod.w, m.final_mod.b, w.temb, w.fmod, 2 * sh.d, sh.d, true, s));
  ACID_TRY(ln_mod(dt, h_out, dt, w.y, sh.N, sh.d, w.fmod, w.fmod + sh.d, nullptr, nullptr, 0, m.block.ln_eps, s));
  Epilogue e;
  e.bias = m.final_out.b;
  e.out_fp32 = true;
  ACID_TRY(linear_forward(dt, w.y, sh.d, sh.N, sh.d, m.final_out.w, (int)sh.P, w.vtok, sh.P, e, s));
  return unpatchify_euler(w.vtok, v_out, latent, m.latent_c, m.latent_f, m.latent_h, m.latent_w, m.pt, m.ph, m.pw,
                          dsig, s);
}

}  // namespace

}  // namespace acid

using namespace acid;

extern "C" acid_status acid_loop_workspace_size(const acid_model* m, size_t* bytes) {
  clear_error();
  ACID_REQUIRE(m && bytes, ACID_ERR_INVALID_ARG, "acid_loop_workspace_size: null argument");
  ACID_TRY(validate_model(*m));
  *bytes = loop_layout(*m, nullptr).bytes;
  return ACID_OK;
}

static acid_status check_ws(const acid_model& m, void* ws, size_t bytes, LoopWs* out) {
  ACID_REQUIRE(ws != nullptr && aligned(ws, 1024), ACID_ERR_WORKSPACE, "loop: workspace null or not 1024-aligned");
  *out = loop_layout(m, ws);
  ACID_REQUIRE(bytes >= out->bytes, ACID_ERR_WORKSPACE,
               "loop: workspace too small (need " + std::to_string(out->bytes) + " bytes)");
  return ACID_OK;
}

extern "C" acid_status acid_loop_begin(const acid_model* m, const acid_loop_cfg* cfg, const void* text,
                                       acid_loop_state* state, void* workspace, size_t workspace_bytes,
                                       acid_stream_t stream) {
  clear_error();
  ACID_REQUIRE(m && cfg && state, ACID_ERR_INVALID_ARG, "acid_loop_begin: null argument");
  ACID_TRY(validate_model(*m));
  ACID_TRY(validate_cfg(*cfg));
  LoopWs w;
  ACID_TRY(check_ws(*m, workspace, workspace_bytes, &w));
  cudaStream_t s = (cudaStream_t)stream;
  memset(state, 0, sizeof(*state));
  const Shape sh = shape_of(*m);
  const int dt = m->block.dtype;
  if (sh.L > 0) {
    ACID_REQUIRE(text != nullptr && aligned(text, 16), ACID_ERR_INVALID_ARG,
                 "acid_loop_begin: text must be a 16-byte aligned device pointer");
    if (m->block.kind == ACID_BLOCK_WAN) {
      Epilogue e;
      e.bias = m->text.b;
      ACID_TRY(linear_forward(dt, text, m->d_text, sh.L, m->d_text, m->text.w, sh.d, w.text, sh.d, e, s));
      // every block's cross-attention keys and values, once per generation
      // (the same GEMM the block would run on each step)
      const size_t kv_bytes = (size_t)sh.L * 2 * sh.d * es(dt);
      for (int i = 0; i < total_blocks(*m); ++i) {
        Epilogue ekv;
        ekv.bias = m->blocks[i].ckv.b;
        ACID_TRY(linear_forward(dt, w.text, sh.d, sh.L, sh.d, m->blocks[i].ckv.w, 2 * sh.d, w.ctx_kv + i * kv_bytes,
                                2 * sh.d, ekv, s));
      }
    } else {
      ACID_CUDA(cudaMemcpyAsync(w.text, text, sh.L * sh.d * es(dt), cudaMemcpyDeviceToDevice, s));
    }
  }
  RopeTable rt = rope_layout(m->block.grid_f, m->block.grid_h, m->block.grid_w, m->block.d / m->block.heads);
  ACID_TRY(rope_build(rt, w.rope, m->block.rope_theta, s));
  ACID_CUDA(cudaMemsetAsync(w.dc_count, 0, sizeof(int), s));
  ACID_CUDA(cudaMemsetAsync(w.drift_done, 0, sizeof(unsigned int), s));
  if (w.patch_split) {  // [W | W]: each row of the patch weights twice
    const size_t row = (size_t)sh.P * 2;
    for (int k = 0; k < 2; ++k)
      ACID_CUDA(cudaMemcpy2DAsync(w.patch_w2 + k * row, 2 * row, m->patch.w, row, row, sh.d, cudaMemcpyDeviceToDevice,
                                  s));
  }
  ACID_REQUIRE(cfg->method != ACID_METHOD_DICACHE || cfg->probe_blocks <= total_blocks(*m), ACID_ERR_INVALID_ARG,
               "acid_loop_begin: probe_blocks exceeds the number of blocks");
  return ACID_OK;
}

// CUDA-event timing of one step (only when a log is requested).
struct StepTimer {
  bool on;
  cudaStream_t s;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  StepTimer(bool on_, cudaStream_t s_) : on(on_), s(s_) {}
  ~StepTimer() {
    if (e0) cudaEventDestroy(e0);
    if (e1) cudaEventDestroy(e1);
  }
  acid_status start() {
    if (!on) return ACID_OK;
    ACID_CUDA(cudaEventCreate(&e0));
    ACID_CUDA(cudaEventCreate(&e1));
    ACID_CUDA(cudaEventRecord(e0, s));
    return ACID_OK;
  }
  // Milliseconds since start (or the previous lap); synchronises on the event.
  acid_status stop(double* ms) {
    ACID_CUDA(cudaEventRecord(e1, s));
    ACID_CUDA(cudaEventSynchronize(e1));
    float f = 0.f;
    ACID_CUDA(cudaEventElapsedTime(&f, e0, e1));
    *ms = f;
    std::swap(e0, e1);
    return ACID_OK;
  }
};

// Patch embedding H_in (fp32) of the latent.  bf16 models: the tokens as
// bf16 hi + lo parts against the weights repeated along K, one tcgen05 GEMM
// with fp32 accumulation (the fp32 tokens to within 2^-17 relative); fp32
// models: the fp32 SIMT GEMM.
static acid_status patch_embed(const acid_model& m, const LoopWs& w, const float* latent, float* h_in,
                               cudaStream_t s) {
  const Shape sh = shape_of(m);
  Epilogue e;
  e.bias = m.patch.b;
  e.out_fp32 = true;
  if (w.patch_split) {
    ACID_TRY(patchify_split(latent, w.tokens, m.latent_c, m.latent_f, m.latent_h, m.latent_w, m.pt, m.ph, m.pw, s));
    return linear_forward(ACID_BF16, w.tokens, 2 * sh.P, sh.N, (int)(2 * sh.P), w.patch_w2, sh.d, h_in, sh.d, e, s);
  }
  ACID_TRY(patchify(latent, ACID_FP32, w.tokens, m.latent_c, m.latent_f, m.latent_h, m.latent_w, m.pt, m.ph, m.pw, s));
  return linear_forward_f32(w.tokens, sh.P, sh.N, (int)sh.P, m.block.dtype, m.patch.w, sh.d, h_in, sh.d, e, s);
}

// One branch's model evaluation at step st->step: Algorithm 1's decision,
// then the base method's compute or reuse.  defer_euler = false applies the
// Euler update to the latent in place; defer_euler = true leaves the latent
// unchanged and points *v_out at the branch's velocity (fp32, latent layout,
// inside w).  Fills the step log's fields except ms; does not advance
// st->step.
static acid_status branch_step(const acid_model* m, const acid_loop_cfg* cfg, acid_loop_state* st, float* latent,
                               const LoopWs& w, bool defer_euler, const float** v_out, acid_step_log& lg,
                               cudaStream_t s) {
  const Shape sh = shape_of(*m);
  const int dt = m->block.dtype;
  const int i = st->step;
  const double sig = sigma_at(*cfg, i), sig_next = sigma_at(*cfg, i + 1);
  const double t = 1000.0 * sig;
  const float dsig = (float)(sig_next - sig);
  const bool warm = i < cfg->warmup;
  // buffers of this step and of the previous one alternate with the parity
  const int par = i & 1;
  float* h_in = w.h_in[par];
  int forced = cfg->forced ? cfg->forced[i] : -1;
  if (forced < 0 && cfg->force_last && i == cfg->n_steps - 1) forced = 1;
  memset(&lg, 0, sizeof(lg));
  lg.step = i;
  lg.warmup = warm;
  lg.t = t;
  lg.signal = lg.dsignal = lg.tau = lg.sigma = NAN;

  // timestep embedding: temb = W2 SiLU(W1 sinusoid(t) + b1) + b2
  ACID_TRY(timestep_sinusoid(w.sinus, t, m->time_freq_dim, s));
  ACID_TRY(gemv(dt, m->time1.w, m->time1.b, w.sinus, w.temb_h, sh.d, m->time_freq_dim, false, s));
  ACID_TRY(gemv(dt, m->time2.w, m->time2.b, w.temb_h, w.temb, sh.d, sh.d, true, s));
  // patch embedding H_in (fp32)
  // (fp32 tokens and accumulation: the drift signal compares consecutive H_in
  // that differ by a few percent, so it must not see bf16 input rounding)
  ACID_TRY(patch_embed(*m, w, latent, h_in, s));
  const int64_t vrow0 = m->block.kind == ACID_BLOCK_WAN ? 0 : sh.L;
  void* x_video = w.xbuf + vrow0 * sh.d * es(dt);
  auto run_model = [&]() -> acid_status {
    if (vrow0 > 0) ACID_CUDA(cudaMemcpyAsync(w.xbuf, w.text, sh.L * sh.d * es(dt), cudaMemcpyDeviceToDevice, s));
    ACID_TRY(add_mixed(ACID_FP32, h_in, ACID_FP32, h_in, dt, x_video, sh.N * sh.d, 0.0f, s));
    return run_blocks(*m, w, s);
  };

  bool compute = true;
  if (cfg->method == ACID_METHOD_TEACACHE) {
    // s_t: rel_l1 of block 0's modulated input (TEMNI) between consecutive
    // steps, both TEMNIs formed from this and the previous step's H_in and
    // block-0 modulation in one read-only pass
    ACID_TRY(gemv(dt, m->blocks[0].mod.w, m->blocks[0].mod.b, w.temb, w.mod0[par], 2 * sh.d, sh.d, true, s));
    ACID_TRY(temni_drift(h_in, w.h_in[par ^ 1], w.mod0[par], w.mod0[par ^ 1], nullptr, i, sh.N, sh.d,
                         m->block.ln_eps, w.dres, w.drift_ws, drift_workspace_bytes(0), s, w.drift_done));
    if (!warm) {
      ACID_REQUIRE(i > 0, ACID_ERR_INVALID_ARG, "TeaCache needs at least one warmup step");
      double h[3];
      ACID_TRY(read_results(h, w.dres, 3, s));
      compute = controller_step(*st, *cfg, i, h[0], forced, &lg);
    }
    if (compute || !st->have_cache) {
      compute = true;
      ACID_TRY(run_model());
      ACID_TRY(add_mixed(dt, x_video, ACID_FP32, h_in, ACID_FP32, w.resid, sh.N * sh.d, -1.0f, s));
      st->have_cache = 1;
    } else {
      ACID_TRY(add_mixed(ACID_FP32, h_in, ACID_FP32, w.resid, dt, x_video, sh.N * sh.d, 1.0f, s));
    }
    ACID_TRY(final_layer(*m, w, x_video, defer_euler ? w.v[0] : nullptr, defer_euler ? nullptr : latent, dsig, s));
    if (defer_euler) *v_out = w.v[0];
  } else if (cfg->method == ACID_METHOD_DICACHE) {
    // probe: the first probe_blocks blocks on every step; P_i (fp32) in temni[i & 1]
    const int pb = cfg->probe_blocks;
    float* p_cur = w.temni[par];
    float* p_prev = w.temni[par ^ 1];
    if (vrow0 > 0) ACID_CUDA(cudaMemcpyAsync(w.xbuf, w.text, sh.L * sh.d * es(dt), cudaMemcpyDeviceToDevice, s));
    ACID_TRY(add_mixed(ACID_FP32, h_in, ACID_FP32, h_in, dt, x_video, sh.N * sh.d, 0.0f, s));
    ACID_TRY(run_blocks(*m, w, s, 0, pb));
    ACID_TRY(add_mixed(dt, x_video, dt, x_video, ACID_FP32, p_cur, sh.N * sh.d, 0.0f, s));
    if (!warm) {
      ACID_REQUIRE(i > 0, ACID_ERR_INVALID_ARG, "DiCache needs at least one warmup step");
      ACID_TRY(drift_launch(ACID_FP32, p_prev, p_cur, nullptr, nullptr, sh.N * sh.d, w.dres, w.drift_ws,
                            drift_workspace_bytes(0), s));
      double h[3];
      ACID_TRY(read_results(h, w.dres, 3, s));
      compute = controller_step(*st, *cfg, i, h[0], forced, &lg);
    }
    if (compute || !st->have_cache) {
      compute = true;
      ACID_TRY(run_blocks(*m, w, s, pb, total_blocks(*m)));
      ACID_TRY(dicache_update(dt, x_video, p_cur, w, sh.N * sh.d, s));
      st->have_cache = 1;
    } else {
      ACID_TRY(dicache_reuse(dt, x_video, p_cur, w, sh.N * sh.d, s));
    }
    ACID_TRY(final_layer(*m, w, x_video, defer_euler ? w.v[0] : nullptr, defer_euler ? nullptr : latent, dsig, s));
    if (defer_euler) *v_out = w.v[0];
  } else {
    // EasyCache: s_t = k mean|x_t - x_{t-1}| / mean|v_{t-1}|
    float* v = w.v[i & 1];
    float* v_prev = w.v[(i & 1) ^ 1];
    if (!warm) {
      ACID_REQUIRE(st->have_rate, ACID_ERR_INVALID_ARG, "EasyCache: transformation rate undefined");
      ACID_TRY(drift_launch(ACID_FP32, w.x_prev, latent, nullptr, nullptr, sh.latent, w.dres, w.drift_ws,
                            drift_workspace_bytes(0), s));
      ACID_TRY(drift_launch(ACID_FP32, v_prev, v_prev, nullptr, nullptr, sh.latent, w.dres + 3, w.drift_ws,
                            drift_workspace_bytes(0), s));
      double h[6];
      ACID_TRY(read_results(h, w.dres, 6, s));
      const double sig_t = ratio_or_inf(st->k_rate * (h[1] / sh.latent), h[5] / sh.latent);
      compute = controller_step(*st, *cfg, i, sig_t, forced, &lg);
    }
    if (compute || !st->have_cache) {
      compute = true;
      ACID_TRY(run_model());
      ACID_TRY(final_layer(*m, w, x_video, v, nullptr, 0.0f, s));
      if (i > 0) {  // k = mean|v_c - v_{c-1}| / mean|x_c - x_{c-1}|
        ACID_TRY(drift_launch(ACID_FP32, v_prev, v, nullptr, nullptr, sh.latent, w.dres, w.drift_ws,
                              drift_workspace_bytes(0), s));
        ACID_TRY(drift_launch(ACID_FP32, w.x_prev, latent, nullptr, nullptr, sh.latent, w.dres + 3, w.drift_ws,
                              drift_workspace_bytes(0), s));
        double h[6];
        ACID_TRY(read_results(h, w.dres, 6, s));
        st->k_rate = ratio_or_inf(h[1] / sh.latent, h[4] / sh.latent);
        st->have_rate = 1;
      }
      ACID_TRY(add_mixed(ACID_FP32, v, ACID_FP32, latent, ACID_FP32, w.offset, sh.latent, -1.0f, s));
      st->have_cache = 1;
    } else {
      ACID_TRY(add_mixed(ACID_FP32, latent, ACID_FP32, w.offset, ACID_FP32, v, sh.latent, 1.0f, s));
    }
    ACID_CUDA(cudaMemcpyAsync(w.x_prev, latent, sh.latent * sizeof(float), cudaMemcpyDeviceToDevice, s));
    if (defer_euler)
      *v_out = v;
    else
      ACID_TRY(euler_update(latent, v, sh.latent, dsig, s));
  }
  lg.computed = compute;
  return ACID_OK;
}

extern "C" acid_status acid_denoise_step(const acid_model* m, const acid_loop_cfg* cfg, acid_loop_state* st,
                                         void* latent_v, acid_step_log* log, void* workspace, size_t workspace_bytes,
                                         acid_stream_t stream) {
  clear_error();
  ACID_REQUIRE(m && cfg && st && latent_v, ACID_ERR_INVALID_ARG, "acid_denoise_step: null argument");
  ACID_TRY(validate_cfg(*cfg));
  ACID_REQUIRE(st->step >= 0 && st->step < cfg->n_steps, ACID_ERR_INVALID_ARG, "acid_denoise_step: step out of range");
  ACID_REQUIRE(aligned(latent_v, 16), ACID_ERR_UNSUPPORTED, "acid_denoise_step: latent must be 16-byte aligned");
  LoopWs w;
  ACID_TRY(check_ws(*m, workspace, workspace_bytes, &w));
  cudaStream_t s = (cudaStream_t)stream;
  StepTimer tm(log != nullptr, s);
  ACID_TRY(tm.start());
  acid_step_log lg;
  ACID_TRY(branch_step(m, cfg, st, static_cast<float*>(latent_v), w, false, nullptr, lg, s));
  st->step += 1;
  if (log) {
    ACID_TRY(tm.stop(&lg.ms));
    *log = lg;
  }
  return ACID_OK;
}

extern "C" acid_status acid_denoise_loop(const acid_model* m, const acid_loop_cfg* cfg, void* latent, const void* text,
                                         acid_step_log* log, void* workspace, size_t workspace_bytes,
                                         acid_stream_t stream) {
  acid_loop_state st;
  ACID_TRY(acid_loop_begin(m, cfg, text, &st, workspace, workspace_bytes, stream));
  for (int i = 0; i < cfg->n_steps; ++i)
    ACID_TRY(acid_denoise_step(m, cfg, &st, latent, log ? log + i : nullptr, workspace, workspace_bytes, stream));
  return ACID_OK;
}

// ===========================================================================
// Classifier-free guidance: two branches (conditional and unconditional
// text), each with its own loop workspace, Algorithm 1 state and cache; the
// Euler step takes v = v_u + g (v_c - v_u).
// ===========================================================================

static size_t guided_half(const acid_model& m) { return (loop_layout(m, nullptr).bytes + 1023) / 1024 * 1024; }

static acid_status guided_check(const acid_model* m, const acid_loop_cfg* cc, const acid_loop_cfg* cu, void* ws,
                                size_t bytes, LoopWs* wc, LoopWs* wu) {
  ACID_REQUIRE(m && cc && cu, ACID_ERR_INVALID_ARG, "guided loop: null argument");
  ACID_TRY(validate_cfg(*cc));
  ACID_TRY(validate_cfg(*cu));
  ACID_REQUIRE(cc->n_steps == cu->n_steps && cc->shift == cu->shift, ACID_ERR_INVALID_ARG,
               "guided loop: both branches need the same n_steps and shift");
  ACID_REQUIRE(ws != nullptr && aligned(ws, 1024), ACID_ERR_WORKSPACE,
               "guided loop: workspace null or not 1024-aligned");
  const size_t half = guided_half(*m);
  ACID_REQUIRE(bytes >= 2 * half, ACID_ERR_WORKSPACE,
               "guided loop: workspace too small (need " + std::to_string(2 * half) + " bytes)");
  *wc = loop_layout(*m, ws);
  *wu = loop_layout(*m, static_cast<uint8_t*>(ws) + half);
  return ACID_OK;
}

extern "C" acid_status acid_guided_workspace_size(const acid_model* m, size_t* bytes) {
  clear_error();
  ACID_REQUIRE(m && bytes, ACID_ERR_INVALID_ARG, "acid_guided_workspace_size: null argument");
  ACID_TRY(validate_model(*m));
  *bytes = 2 * guided_half(*m);
  return ACID_OK;
}

extern "C" acid_status acid_guided_begin(const acid_model* m, const acid_loop_cfg* cfg_cond,
                                         const acid_loop_cfg* cfg_uncond, const void* text_cond,
                                         const void* text_uncond, acid_loop_state* state_cond,
                                         acid_loop_state* state_uncond, void* workspace, size_t workspace_bytes,
                                         acid_stream_t stream) {
  clear_error();
  ACID_REQUIRE(m, ACID_ERR_INVALID_ARG, "acid_guided_begin: null model");
  ACID_TRY(validate_model(*m));
  LoopWs wc, wu;
  ACID_TRY(guided_check(m, cfg_cond, cfg_uncond, workspace, workspace_bytes, &wc, &wu));
  const size_t half = guided_half(*m);
  ACID_TRY(acid_loop_begin(m, cfg_cond, text_cond, state_cond, workspace, half, stream));
  ACID_TRY(acid_loop_begin(m, cfg_uncond, text_uncond, state_uncond, static_cast<uint8_t*>(workspace) + half, half,
                           stream));
  return ACID_OK;
}

extern "C" acid_status acid_guided_step(const acid_model* m, const acid_loop_cfg* cfg_cond,
                                        const acid_loop_cfg* cfg_uncond, double guidance_scale,
                                        acid_loop_state* state_cond, acid_loop_state* state_uncond, void* latent_v,
                                        acid_step_log* log_cond, acid_step_log* log_uncond, void* workspace,
                                        size_t workspace_bytes, acid_stream_t stream) {
  clear_error();
  ACID_REQUIRE(state_cond && state_uncond && latent_v, ACID_ERR_INVALID_ARG, "acid_guided_step: null argument");
  LoopWs wc, wu;
  ACID_TRY(guided_check(m, cfg_cond, cfg_uncond, workspace, workspace_bytes, &wc, &wu));
  ACID_REQUIRE(state_cond->step == state_uncond->step && state_cond->step >= 0 &&
                   state_cond->step < cfg_cond->n_steps,
               ACID_ERR_INVALID_ARG, "acid_guided_step: branch steps differ or out of range");
  ACID_REQUIRE(aligned(latent_v, 16), ACID_ERR_UNSUPPORTED, "acid_guided_step: latent must be 16-byte aligned");
  ACID_REQUIRE(std::isfinite(guidance_scale), ACID_ERR_INVALID_ARG, "acid_guided_step: guidance scale not finite");
  cudaStream_t s = (cudaStream_t)stream;
  float* latent = static_cast<float*>(latent_v);
  const int i = state_cond->step;
  const float dsig = (float)(sigma_at(*cfg_cond, i + 1) - sigma_at(*cfg_cond, i));
  const bool timed = log_cond || log_uncond;
  StepTimer tm(timed, s);
  ACID_TRY(tm.start());
  acid_step_log lc, lu;
  const float *vc = nullptr, *vu = nullptr;
  ACID_TRY(branch_step(m, cfg_cond, state_cond, latent, wc, true, &vc, lc, s));
  if (timed) ACID_TRY(tm.stop(&lc.ms));
  ACID_TRY(branch_step(m, cfg_uncond, state_uncond, latent, wu, true, &vu, lu, s));
  ACID_TRY(guided_euler_update(latent, vc, vu, shape_of(*m).latent, (float)guidance_scale, dsig, s));
  if (timed) ACID_TRY(tm.stop(&lu.ms));
  state_cond->step += 1;
  state_uncond->step += 1;
  if (log_cond) *log_cond = lc;
  if (log_uncond) *log_uncond = lu;
  return ACID_OK;
}

extern "C" acid_status acid_denoise_loop_guided(const acid_model* m, const acid_loop_cfg* cfg_cond,
                                                const acid_loop_cfg* cfg_uncond, double guidance_scale,
                                                void* latent, const void* text_cond, const void* text_uncond,
                                                acid_step_log* log_cond, acid_step_log* log_uncond, void* workspace,
                                                size_t workspace_bytes, acid_stream_t stream) {
  acid_loop_state sc, su;
  ACID_TRY(acid_guided_begin(m, cfg_cond, cfg_uncond, text_cond, text_uncond, &sc, &su, workspace, workspace_bytes,
                             stream));
  for (int i = 0; i < cfg_cond->n_steps; ++i)
    ACID_TRY(acid_guided_step(m, cfg_cond, cfg_uncond, guidance_scale, &sc, &su, latent,
                              log_cond ? log_cond + i : nullptr, log_uncond ? log_uncond + i : nullptr, workspace,
                              workspace_bytes, stream));
  return ACID_OK;
}

// ===========================================================================
// The whole generation as one CUDA graph: a WHILE node whose body is one
// sampler step.  The drift signal, Algorithm 1's decision and the step index
// live in device memory; the decision selects the IF (compute) or ELSE
// (reuse) body of a conditional node, so no step waits for the host.
// ===========================================================================

namespace acid {
namespace {

__device__ double dev_ratio_or_inf(double num, double den) {
  if (den == 0.0) return num == 0.0 ? 0.0 : INFINITY;
  return num / den;
}

// Algorithm 1 on the device (one thread), through the same algorithm1_step.
// dres: TeaCache {rel, num, den}; EasyCache {., sum|x - x_prev|, .,
// ., ., sum|v_prev|}.
__global__ void controller_kernel(DevLoop* st, const double* dres, const double* sig, const int8_t* forced,
                                  const double* tau_sched, acid_step_log* log,
                                  cudaGraphConditionalHandle h_compute) {
  const int i = st->step;
  const bool warm = i < st->warmup;
  int f = st->use_forced ? forced[i] : -1;
  if (f < 0 && st->force_last && i == st->n_steps - 1) f = 1;
  acid_step_log lg;
  lg.step = i;
  lg.warmup = warm;
  lg.forced = 0;
  lg.t = 1000.0 * sig[i];
  lg.signal = lg.dsignal = lg.tau = lg.sigma = NAN;
  lg.ms = NAN;
  bool compute = true;
  if (!warm) {
    const double s_raw = st->method != ACID_METHOD_EASYCACHE
                             ? dres[0]
                             : dev_ratio_or_inf(st->k_rate * (dres[1] / st->latent_n), dres[5] / st->latent_n);
    const double s = rescale_signal(s_raw, st->poly, st->poly_n);
    const double tau_fix = st->use_tau_sched ? tau_sched[i] : NAN;
    compute = algorithm1_step(st->sigma_acc, st->s_prev, st->have_prev, s, st->tau_low, st->tau_high, st->delta,
                              tau_fix, f, &lg);
  }
  if (!st->have_cache) compute = true;
  if (compute) st->have_cache = 1;
  st->compute = compute;
  lg.computed = compute;
  log[i] = lg;
  cudaGraphSetConditional(h_compute, compute ? 1u : 0u);
}

// EasyCache k = mean|v_c - v_{c-1}| / mean|x_c - x_{c-1}| after a computed step i > 0.
__global__ void easycache_rate_kernel(DevLoop* st, const double* dres) {
  if (st->step == 0) return;
  st->k_rate = dev_ratio_or_inf(dres[1] / st->latent_n, dres[4] / st->latent_n);
  st->have_rate = 1;
}

// Next step: the step index of the branch (and of the second branch of a
// guided generation), and the WHILE condition.
__global__ void advance_kernel(DevLoop* st, DevLoop* st2, cudaGraphConditionalHandle h_loop) {
  st->step += 1;
  if (st2) st2->step += 1;
  cudaGraphSetConditional(h_loop, st->step < st->n_steps ? 1u : 0u);
}

acid_status add_conditional(cudaStream_t s, cudaGraphConditionalHandle h, cudaGraphConditionalNodeType type,
                            unsigned size, cudaGraph_t* bodies) {
  cudaStreamCaptureStatus status;
  cudaGraph_t g;
  const cudaGraphNode_t* deps = nullptr;
  size_t ndeps = 0;
  ACID_CUDA(cudaStreamGetCaptureInfo(s, &status, nullptr, &g, &deps, nullptr, &ndeps));
  ACID_REQUIRE(status == cudaStreamCaptureStatusActive, ACID_ERR_CUDA, "graph: stream is not capturing");
  cudaGraphNodeParams p = {};
  p.type = cudaGraphNodeTypeConditional;
  p.conditional.handle = h;
  p.conditional.type = type;
  p.conditional.size = size;
  cudaGraphNode_t node;
  ACID_CUDA(cudaGraphAddNode(&node, g, deps, nullptr, ndeps, &p));
  for (unsigned k = 0; k < size; ++k) bodies[k] = p.conditional.phGraph_out[k];
  ACID_CUDA(cudaStreamUpdateCaptureDependencies(s, &node, nullptr, 1, cudaStreamSetCaptureDependencies));
  return ACID_OK;
}

struct GraphCapture {
  cudaStream_t main = nullptr, side = nullptr;
  ~GraphCapture() {
    if (main) cudaStreamDestroy(main);
    if (side) cudaStreamDestroy(side);
  }
};

// Records, into the graph `body` that gc.main is capturing, one branch's part
// of a step of parity `par` (the buffers that alternate between steps are
// chosen here; the graph holds one such body per parity): its inputs, signal
// and Algorithm 1 decision, the compute or reuse body of an IF/ELSE node
// (captured on gc.side), and its velocity in w.v[0] together with the copies
// that keep the previous step's values.  The Euler update is left to the caller.
acid_status capture_branch(const acid_model& m, const acid_loop_cfg& cfg, LoopWs& w, float* latent,
                           GraphCapture& gc, cudaGraph_t body, int par) {
  const Shape sh = shape_of(m);
  const int dt = m.block.dtype;
  cudaStream_t s = gc.main, s2 = gc.side;
  const int* step = &w.dev->step;
  const int64_t vrow0 = m.block.kind == ACID_BLOCK_WAN ? 0 : sh.L;
  void* x_video = w.xbuf + vrow0 * sh.d * es(dt);
  float* h_in = w.h_in[par];
  cudaGraphConditionalHandle h_compute;
  ACID_CUDA(cudaGraphConditionalHandleCreate(&h_compute, body, 0, 0));

  // ---- step inputs: temb, patch embedding
  ACID_TRY(timestep_sinusoid_sig(w.sinus, w.sig, step, m.time_freq_dim, s));
  ACID_TRY(gemv(dt, m.time1.w, m.time1.b, w.sinus, w.temb_h, sh.d, m.time_freq_dim, false, s));
  ACID_TRY(gemv(dt, m.time2.w, m.time2.b, w.temb_h, w.temb, sh.d, sh.d, true, s));
  ACID_TRY(patch_embed(m, w, latent, h_in, s));
  // ---- signal and decision
  float* v = w.v[0];
  float* v_prev = w.v[1];
  // DiCache probe features of this step and of the previous one
  float* p_cur = w.temni[par];
  float* p_prev = w.temni[par ^ 1];
  const int pb = cfg.probe_blocks;
  if (cfg.method == ACID_METHOD_TEACACHE) {
    ACID_TRY(gemv(dt, m.blocks[0].mod.w, m.blocks[0].mod.b, w.temb, w.mod0[par], 2 * sh.d, sh.d, true, s));
    ACID_TRY(temni_drift(h_in, w.h_in[par ^ 1], w.mod0[par], w.mod0[par ^ 1], step, 0, sh.N, sh.d, m.block.ln_eps,
                         w.dres, w.drift_ws, drift_workspace_bytes(0), s, w.drift_done));
  } else if (cfg.method == ACID_METHOD_DICACHE) {
    if (vrow0 > 0) ACID_CUDA(cudaMemcpyAsync(w.xbuf, w.text, sh.L * sh.d * es(dt), cudaMemcpyDeviceToDevice, s));
    ACID_TRY(add_mixed(ACID_FP32, h_in, ACID_FP32, h_in, dt, x_video, sh.N * sh.d, 0.0f, s));
    ACID_TRY(run_blocks(m, w, s, 0, pb));
    ACID_TRY(add_mixed(dt, x_video, dt, x_video, ACID_FP32, p_cur, sh.N * sh.d, 0.0f, s));
    ACID_TRY(drift_launch(ACID_FP32, p_prev, p_cur, nullptr, nullptr, sh.N * sh.d, w.dres, w.drift_ws,
                          drift_workspace_bytes(0), s));
  } else {
    ACID_TRY(drift_launch(ACID_FP32, w.x_prev, latent, nullptr, nullptr, sh.latent, w.dres, w.drift_ws,
                          drift_workspace_bytes(0), s));
    ACID_TRY(drift_launch(ACID_FP32, v_prev, v_prev, nullptr, nullptr, sh.latent, w.dres + 3, w.drift_ws,
                          drift_workspace_bytes(0), s));
  }
  controller_kernel<<<1, 1, 0, s>>>(w.dev, w.dres, w.sig, w.forced, w.tau_sched, w.dlog, h_compute);
  ACID_CHECK_LAUNCH();
  cudaGraph_t br[2];
  ACID_TRY(add_conditional(s, h_compute, cudaGraphCondTypeIf, 2, br));

  // ---- compute body: the model
  ACID_CUDA(cudaStreamBeginCaptureToGraph(s2, br[0], nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed));
  if (cfg.method == ACID_METHOD_DICACHE) {
    ACID_TRY(run_blocks(m, w, s2, pb, total_blocks(m)));
    ACID_TRY(dicache_update(dt, x_video, p_cur, w, sh.N * sh.d, s2));
  } else {
    if (vrow0 > 0) ACID_CUDA(cudaMemcpyAsync(w.xbuf, w.text, sh.L * sh.d * es(dt), cudaMemcpyDeviceToDevice, s2));
    ACID_TRY(add_mixed(ACID_FP32, h_in, ACID_FP32, h_in, dt, x_video, sh.N * sh.d, 0.0f, s2));
    ACID_TRY(run_blocks(m, w, s2));
  }
  if (cfg.method == ACID_METHOD_DICACHE) {
  } else if (cfg.method == ACID_METHOD_TEACACHE) {
    ACID_TRY(add_mixed(dt, x_video, ACID_FP32, h_in, ACID_FP32, w.resid, sh.N * sh.d, -1.0f, s2));
  } else {
    ACID_TRY(final_layer(m, w, x_video, v, nullptr, 0.0f, s2));
    ACID_TRY(drift_launch(ACID_FP32, v_prev, v, nullptr, nullptr, sh.latent, w.dres, w.drift_ws,
                          drift_workspace_bytes(0), s2));
    ACID_TRY(drift_launch(ACID_FP32, w.x_prev, latent, nullptr, nullptr, sh.latent, w.dres + 3, w.drift_ws,
                          drift_workspace_bytes(0), s2));
    easycache_rate_kernel<<<1, 1, 0, s2>>>(w.dev, w.dres);
    ACID_CHECK_LAUNCH();
    ACID_TRY(add_mixed(ACID_FP32, v, ACID_FP32, latent, ACID_FP32, w.offset, sh.latent, -1.0f, s2));
  }
  cudaGraph_t tmp;
  ACID_CUDA(cudaStreamEndCapture(s2, &tmp));
  // ---- reuse body: cached residual / offset
  ACID_CUDA(cudaStreamBeginCaptureToGraph(s2, br[1], nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed));
  if (cfg.method == ACID_METHOD_TEACACHE)
    ACID_TRY(add_mixed(ACID_FP32, h_in, ACID_FP32, w.resid, dt, x_video, sh.N * sh.d, 1.0f, s2));
  else if (cfg.method == ACID_METHOD_DICACHE)
    ACID_TRY(dicache_reuse(dt, x_video, p_cur, w, sh.N * sh.d, s2));
  else
    ACID_TRY(add_mixed(ACID_FP32, latent, ACID_FP32, w.offset, ACID_FP32, v, sh.latent, 1.0f, s2));
  ACID_CUDA(cudaStreamEndCapture(s2, &tmp));

  // ---- output: the velocity, and the previous step's values
  if (cfg.method == ACID_METHOD_TEACACHE) {
    ACID_TRY(final_layer(m, w, x_video, v, nullptr, 0.0f, s));
  } else if (cfg.method == ACID_METHOD_DICACHE) {
    ACID_TRY(final_layer(m, w, x_video, v, nullptr, 0.0f, s));
  } else {
    ACID_CUDA(cudaMemcpyAsync(w.x_prev, latent, sh.latent * sizeof(float), cudaMemcpyDeviceToDevice, s));
    ACID_CUDA(cudaMemcpyAsync(v_prev, v, sh.latent * sizeof(float), cudaMemcpyDeviceToDevice, s));
  }
  return ACID_OK;
}

// Sets the parity conditional of the step about to run (1: odd step).
__global__ void parity_kernel(const DevLoop* st, cudaGraphConditionalHandle h_parity) {
  cudaGraphSetConditional(h_parity, (unsigned)(st->step & 1));
}

// Opens the parity switch of a step in `body` (captured on gc.main): an
// IF/ELSE node on the step's parity; returns its odd (bodies[0]) and even
// (bodies[1]) graphs.
acid_status capture_parity_switch(const LoopWs& w, GraphCapture& gc, cudaGraph_t body, cudaGraph_t* bodies) {
  cudaGraphConditionalHandle h_parity;
  ACID_CUDA(cudaGraphConditionalHandleCreate(&h_parity, body, 0, 0));
  parity_kernel<<<1, 1, 0, gc.main>>>(w.dev, h_parity);
  ACID_CHECK_LAUNCH();
  return add_conditional(gc.main, h_parity, cudaGraphCondTypeIf, 2, bodies);
}

// One sampler step into `body`: the branch (one capture per parity, under the
// parity switch), then the Euler update and the next step.
acid_status capture_step(const acid_model& m, const acid_loop_cfg& cfg, LoopWs& w, float* latent, GraphCapture& gc,
                         cudaGraph_t body, cudaGraphConditionalHandle h_loop) {
  cudaStream_t s = gc.main;
  cudaGraph_t tmp, pb[2];
  ACID_CUDA(cudaStreamBeginCaptureToGraph(s, body, nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed));
  ACID_TRY(capture_parity_switch(w, gc, body, pb));
  ACID_TRY(euler_update_sig(latent, w.v[0], shape_of(m).latent, w.sig, &w.dev->step, s));
  advance_kernel<<<1, 1, 0, s>>>(w.dev, nullptr, h_loop);
  ACID_CHECK_LAUNCH();
  ACID_CUDA(cudaStreamEndCapture(s, &tmp));
  for (int par = 0; par < 2; ++par) {
    cudaGraph_t g = pb[par == 1 ? 0 : 1];
    ACID_CUDA(cudaStreamBeginCaptureToGraph(s, g, nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed));
    ACID_TRY(capture_branch(m, cfg, w, latent, gc, g, par));
    ACID_CUDA(cudaStreamEndCapture(s, &tmp));
  }
  return ACID_OK;
}

// One guided step: both branches on x_i, then x_{i+1} = x_i + dsigma (v_u + g (v_c - v_u)).
acid_status capture_guided_step(const acid_model& m, const acid_loop_cfg& cc, const acid_loop_cfg& cu, float scale,
                                LoopWs& wc, LoopWs& wu, float* latent, GraphCapture& gc, cudaGraph_t body,
                                cudaGraphConditionalHandle h_loop) {
  cudaStream_t s = gc.main;
  cudaGraph_t tmp, pb[2];
  ACID_CUDA(cudaStreamBeginCaptureToGraph(s, body, nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed));
  ACID_TRY(capture_parity_switch(wc, gc, body, pb));
  ACID_TRY(guided_euler_update_sig(latent, wc.v[0], wu.v[0], shape_of(m).latent, scale, wc.sig, &wc.dev->step, s));
  advance_kernel<<<1, 1, 0, s>>>(wc.dev, wu.dev, h_loop);
  ACID_CHECK_LAUNCH();
  ACID_CUDA(cudaStreamEndCapture(s, &tmp));
  for (int par = 0; par < 2; ++par) {
    cudaGraph_t g = pb[par == 1 ? 0 : 1];
    ACID_CUDA(cudaStreamBeginCaptureToGraph(s, g, nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed));
    ACID_TRY(capture_branch(m, cc, wc, latent, gc, g, par));
    ACID_TRY(capture_branch(m, cu, wu, latent, gc, g, par));
    ACID_CUDA(cudaStreamEndCapture(s, &tmp));
  }
  return ACID_OK;
}

// Device-side loop state, noise levels, forced decisions and threshold
// schedule of one branch; `stream` is synchronised (host sources are stack memory).
acid_status setup_graph_state(const acid_model& m, const acid_loop_cfg& cfg, const LoopWs& w, cudaStream_t s) {
  const Shape sh = shape_of(m);
  DevLoop d = {};
  d.n_steps = cfg.n_steps;
  d.warmup = cfg.warmup;
  d.method = cfg.method;
  d.force_last = cfg.force_last;
  d.use_forced = cfg.forced != nullptr;
  d.use_tau_sched = cfg.tau_schedule != nullptr;
  d.tau_low = cfg.tau_low;
  d.tau_high = cfg.tau_high;
  d.delta = cfg.delta;
  d.latent_n = (double)sh.latent;
  d.poly_n = cfg.signal_poly_n;
  for (int j = 0; j < cfg.signal_poly_n; ++j) d.poly[j] = cfg.signal_poly[j];
  double sig[kMaxGraphSteps + 1];
  for (int i = 0; i <= cfg.n_steps; ++i) sig[i] = sigma_at(cfg, i);
  ACID_CUDA(cudaMemcpyAsync(w.dev, &d, sizeof(d), cudaMemcpyHostToDevice, s));
  ACID_CUDA(cudaMemcpyAsync(w.sig, sig, sizeof(double) * (cfg.n_steps + 1), cudaMemcpyHostToDevice, s));
  if (cfg.forced) ACID_CUDA(cudaMemcpyAsync(w.forced, cfg.forced, cfg.n_steps, cudaMemcpyHostToDevice, s));
  if (cfg.tau_schedule)
    ACID_CUDA(cudaMemcpyAsync(w.tau_sched, cfg.tau_schedule, sizeof(double) * cfg.n_steps, cudaMemcpyHostToDevice, s));
  ACID_CUDA(cudaStreamSynchronize(s));
  return ACID_OK;
}

// Builds the WHILE graph around `record` (which captures one step into the
// body), launches it on `stream`, synchronises and destroys it.
template <typename Record>
acid_status run_graph(cudaStream_t stream, Record record) {
  GraphCapture gc;
  ACID_CUDA(cudaStreamCreateWithFlags(&gc.main, cudaStreamNonBlocking));
  ACID_CUDA(cudaStreamCreateWithFlags(&gc.side, cudaStreamNonBlocking));
  cudaGraph_t g = nullptr;
  cudaGraphExec_t exec = nullptr;
  acid_status rc = ACID_OK;
  do {
    if (cudaGraphCreate(&g, 0) != cudaSuccess) { rc = ACID_ERR_CUDA; set_error("cudaGraphCreate failed"); break; }
    cudaGraphConditionalHandle h_loop;
    if (cudaGraphConditionalHandleCreate(&h_loop, g, 1, cudaGraphCondAssignDefault) != cudaSuccess) {
      rc = ACID_ERR_CUDA;
      set_error("cudaGraphConditionalHandleCreate failed");
      break;
    }
    cudaGraphNodeParams p = {};
    p.type = cudaGraphNodeTypeConditional;
    p.conditional.handle = h_loop;
    p.conditional.type = cudaGraphCondTypeWhile;
    p.conditional.size = 1;
    cudaGraphNode_t node;
    if (cudaGraphAddNode(&node, g, nullptr, nullptr, 0, &p) != cudaSuccess) {
      rc = ACID_ERR_CUDA;
      set_error("cudaGraphAddNode (while) failed");
      break;
    }
    rc = record(gc, p.conditional.phGraph_out[0], h_loop);
    if (rc != ACID_OK) {
      cudaGraph_t junk;
      cudaStreamEndCapture(gc.side, &junk);
      cudaStreamEndCapture(gc.main, &junk);
      break;
    }
    cudaError_t e = cudaGraphInstantiate(&exec, g, 0);
    if (e != cudaSuccess) {
      rc = ACID_ERR_CUDA;
      set_error(std::string("cudaGraphInstantiate: ") + cudaGetErrorString(e));
      break;
    }
    e = cudaGraphLaunch(exec, stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
    if (e != cudaSuccess) {
      rc = ACID_ERR_CUDA;
      set_error(std::string("graph launch: ") + cudaGetErrorString(e));
    }
  } while (false);
  if (exec) cudaGraphExecDestroy(exec);
  if (g) cudaGraphDestroy(g);
  return rc;
}

}  // namespace
}  // namespace acid

extern "C" acid_status acid_denoise_loop_graph(const acid_model* m, const acid_loop_cfg* cfg, void* latent_v,
                                               const void* text, acid_step_log* log, void* workspace,
                                               size_t workspace_bytes, acid_stream_t stream) {
  clear_error();
  ACID_REQUIRE(m && cfg && latent_v, ACID_ERR_INVALID_ARG, "acid_denoise_loop_graph: null argument");
  ACID_TRY(validate_cfg(*cfg));
  ACID_REQUIRE(cfg->n_steps <= kMaxGraphSteps, ACID_ERR_UNSUPPORTED,
               "acid_denoise_loop_graph: at most " + std::to_string(kMaxGraphSteps) + " steps");
  ACID_REQUIRE(aligned(latent_v, 16), ACID_ERR_UNSUPPORTED, "acid_denoise_loop_graph: latent must be 16-byte aligned");
  acid_loop_state st;
  ACID_TRY(acid_loop_begin(m, cfg, text, &st, workspace, workspace_bytes, stream));
  LoopWs w = loop_layout(*m, workspace);
  cudaStream_t s = (cudaStream_t)stream;
  ACID_TRY(setup_graph_state(*m, *cfg, w, s));
  float* latent = static_cast<float*>(latent_v);
  ACID_TRY(run_graph(s, [&](GraphCapture& gc, cudaGraph_t body, cudaGraphConditionalHandle h_loop) {
    return capture_step(*m, *cfg, w, latent, gc, body, h_loop);
  }));
  if (log) {
    ACID_CUDA(cudaMemcpyAsync(log, w.dlog, sizeof(acid_step_log) * cfg->n_steps, cudaMemcpyDeviceToHost, s));
    ACID_CUDA(cudaStreamSynchronize(s));
  }
  return ACID_OK;
}

extern "C" acid_status acid_denoise_loop_guided_graph(const acid_model* m, const acid_loop_cfg* cfg_cond,
                                                      const acid_loop_cfg* cfg_uncond, double guidance_scale,
                                                      void* latent_v, const void* text_cond, const void* text_uncond,
                                                      acid_step_log* log_cond, acid_step_log* log_uncond,
                                                      void* workspace, size_t workspace_bytes, acid_stream_t stream) {
  clear_error();
  ACID_REQUIRE(m && cfg_cond && cfg_uncond && latent_v, ACID_ERR_INVALID_ARG,
               "acid_denoise_loop_guided_graph: null argument");
  ACID_REQUIRE(cfg_cond->n_steps <= kMaxGraphSteps, ACID_ERR_UNSUPPORTED,
               "acid_denoise_loop_guided_graph: at most " + std::to_string(kMaxGraphSteps) + " steps");
  ACID_REQUIRE(aligned(latent_v, 16), ACID_ERR_UNSUPPORTED,
               "acid_denoise_loop_guided_graph: latent must be 16-byte aligned");
  ACID_REQUIRE(std::isfinite(guidance_scale), ACID_ERR_INVALID_ARG,
               "acid_denoise_loop_guided_graph: guidance scale not finite");
  acid_loop_state sc, su;
  ACID_TRY(acid_guided_begin(m, cfg_cond, cfg_uncond, text_cond, text_uncond, &sc, &su, workspace, workspace_bytes,
                             stream));
  LoopWs wc, wu;
  ACID_TRY(guided_check(m, cfg_cond, cfg_uncond, workspace, workspace_bytes, &wc, &wu));
  cudaStream_t s = (cudaStream_t)stream;
  ACID_TRY(setup_graph_state(*m, *cfg_cond, wc, s));
  ACID_TRY(setup_graph_state(*m, *cfg_uncond, wu, s));
  float* latent = static_cast<float*>(latent_v);
  ACID_TRY(run_graph(s, [&](GraphCapture& gc, cudaGraph_t body, cudaGraphConditionalHandle h_loop) {
    return capture_guided_step(*m, *cfg_cond, *cfg_uncond, (float)guidance_scale, wc, wu, latent, gc, body, h_loop);
  }));
  const int n = cfg_cond->n_steps;
  if (log_cond) ACID_CUDA(cudaMemcpyAsync(log_cond, wc.dlog, sizeof(acid_step_log) * n, cudaMemcpyDeviceToHost, s));
  if (log_uncond) ACID_CUDA(cudaMemcpyAsync(log_uncond, wu.dlog, sizeof(acid_step_log) * n, cudaMemcpyDeviceToHost, s));
  ACID_CUDA(cudaStreamSynchronize(s));
  return ACID_OK;
}
