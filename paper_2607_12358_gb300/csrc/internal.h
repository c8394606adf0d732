// Internal launch interface shared by the library's translation units.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "acid.h"

namespace acid {

// ----------------------------------------------------------------- rope
// 3D RoPE tables: for each axis a, pos < extent_a, pair j < pairs_a,
// float2(cos, sin) of pos * theta^(-2j / d_a).  Axes in order t, h, w;
// d_h = d_w = 2 floor(Dh/6), d_t = Dh - 2 d_h.
struct RopeTable {
  const float2* table = nullptr;  // [F*pt2 | H*ph2 | W*pw2]
  int grid_f = 0, grid_h = 0, grid_w = 0;
  int pairs_t = 0, pairs_h = 0, pairs_w = 0;
  float inv_hw = 0.f, inv_w = 0.f;  // 1 / (grid_h * grid_w), 1 / grid_w (position decomposition)
  int64_t elems() const {
    return (int64_t)grid_f * pairs_t + (int64_t)grid_h * pairs_h + (int64_t)grid_w * pairs_w;
  }
};
RopeTable rope_layout(int grid_f, int grid_h, int grid_w, int head_dim);
acid_status rope_build(RopeTable& t, float2* storage, float theta, cudaStream_t s);

// ----------------------------------------------------------------- GEMM
enum EpiKind : int {
  EPI_BIAS = 0,       // out = acc + b
  EPI_GELU = 1,       // out = gelu_tanh(acc + b)
  EPI_ROPE_QKV = 2,   // out = acc + b, then 3D RoPE on the q and k column blocks of video rows
  EPI_GATED_RES = 3,  // out = res + gate[col] * (acc + b); gate per stream
  EPI_RES = 4         // out = res + acc + b
};

struct Epilogue {
  int kind = EPI_BIAS;
  const float* bias = nullptr;     // [N] or null
  // gated residual: rows (global index) < gate_split use gate_text, else gate_video
  const float* gate_video = nullptr;
  const float* gate_text = nullptr;
  int64_t gate_split = 0;
  const void* residual = nullptr;  // [M, ldr] (may equal out)
  int64_t ldr = 0;
  bool res_fp32 = false;           // residual dtype fp32 (else the GEMM dtype)
  int64_t row_base = 0;            // global row index of GEMM row 0
  // rope: columns [0, 2d) hold q then k; video rows are global rows >= rope_first_video
  RopeTable rope;
  int64_t rope_first_video = 0;
  int d = 0, head_dim = 0;
  bool out_fp32 = false;           // output dtype fp32 (else the GEMM dtype)
  // optional device scratch for a split-K last round of the SM-pair GEMM
  // (long K only); without it the GEMM runs as one launch
  void* splitk_ws = nullptr;
  size_t splitk_bytes = 0;
};

// Scratch that lets a pair GEMM's split-K last round run (a bound for any
// shape: at most one 256 x 256 fp32 partial tile per resident CTA pair).
constexpr size_t kSplitKScratchBytes = (size_t)80 * 256 * 256 * 4;

// out[M, N] (row stride ldo) = epilogue(A[M, K] (row stride lda) * W[N, K]^T)
acid_status linear_forward(int dtype, const void* A, int64_t lda, int64_t M, int K, const void* W,
                           int N, void* out, int64_t ldo, const Epilogue& epi, cudaStream_t s);

// fp32 activations and output with fp32 or bf16 weights (FP32 pipes, fp32 accumulation)
acid_status linear_forward_f32(const void* A, int64_t lda, int64_t M, int K, int w_dtype, const void* W, int N,
                               void* out, int64_t ldo, const Epilogue& epi, cudaStream_t s);

// ----------------------------------------------------------------- attention
struct AttnArgs {
  const void* q = nullptr; int64_t ldq = 0; int q_col = 0;
  const void* k = nullptr; int64_t ldk = 0; int k_col = 0;
  const void* v = nullptr; int64_t ldv = 0; int v_col = 0;
  void* out = nullptr; int64_t ldo = 0; int o_col = 0;
  int64_t nq = 0, nk = 0;
  int heads = 0, head_dim = 0;
  // optional scratch for splitting the last partial wave along the key range
  void* part = nullptr;
  size_t part_bytes = 0;
};
acid_status attention_forward(int dtype, const AttnArgs& a, cudaStream_t s);
constexpr int kAttnSplitCtas = 160;  // at least the SM count of the target GPU
inline size_t attn_part_bytes(int head_dim) {
  return (size_t)kAttnSplitCtas * 256 * (size_t)(head_dim + 2) * sizeof(float);
}

// ----------------------------------------------------------------- elementwise
// y[r] = LN(x[r]) * (1 + scale) + shift; rows < split use (shift_t, scale_t).
// shift/scale may be null (plain LayerNorm).
acid_status ln_mod(int in_dtype, const void* x, int out_dtype, void* y, int64_t rows, int d,
                   const float* shift_v, const float* scale_v, const float* shift_t,
                   const float* scale_t, int64_t split, float eps, cudaStream_t s);

// TeaCache signal sums from the fp32 patch embeddings of two consecutive steps
// and their block-0 modulations (shift then scale, d each): TEMNI of both
// steps formed in registers, 8 bytes read per element.  Result {rel, num, den}
// in d_result as drift_launch.  step from step_dev (device) if non-null, else
// step_host; step 0 gives zero sums.  done: null, or a device counter that is
// zero on entry; then the kernel's last CTA forms the result (one launch) and
// leaves the counter at zero again.
acid_status temni_drift(const float* h_cur, const float* h_prev, const float* mod_cur, const float* mod_prev,
                        const int* step_dev, int step_host, int64_t rows, int d, float eps, double* d_result,
                        void* workspace, size_t ws_bytes, cudaStream_t s, unsigned int* done = nullptr);

// y[j] = sum_k W[j, k] act(x[k]) + b[j]; act = SiLU if silu_input.
acid_status gemv(int w_dtype, const void* W, const float* b, const float* x, float* y, int n_out,
                 int k, bool silu_input, cudaStream_t s);

acid_status timestep_sinusoid(float* out, double t, int dim, cudaStream_t s);

// drift partial sums (fixed-order two-pass reduction) and optional fused apply
size_t drift_workspace_bytes(int64_t n);
acid_status drift_launch(int dtype, const void* prev, const void* cur, const void* resid, void* out,
                         int64_t n, double* d_result /* device double[3]: rel, num, den */,
                         void* workspace, size_t ws_bytes, cudaStream_t s);

// out = a + b elementwise, one dtype, 16-byte vectors
acid_status add_same(int dtype, const void* a, const void* b, void* out, int64_t n, cudaStream_t s);

// out = a + b_scale * b elementwise with per-operand dtypes
acid_status add_mixed(int a_dtype, const void* a, int b_dtype, const void* b, int out_dtype,
                      void* out, int64_t n, float b_scale, cudaStream_t s);

acid_status patchify(const float* latent, int out_dtype, void* tokens, int C, int F, int H, int W,
                     int pt, int ph, int pw, cudaStream_t s);
// bf16 tokens [N, 2P]: each fp32 patch value x as hi = bf16(x) in column p and
// lo = bf16(x - hi) in column P + p (hi + lo = x to within 2^-17 |x|)
acid_status patchify_split(const float* latent, void* tokens, int C, int F, int H, int W, int pt, int ph, int pw,
                           cudaStream_t s);
// v (optional) = unpatchify(vtok); latent += dsigma * v
acid_status unpatchify_euler(const float* vtok, float* v_out, float* latent, int C, int F, int H,
                             int W, int pt, int ph, int pw, float dsigma, cudaStream_t s);
acid_status euler_update(float* latent, const float* v, int64_t n, float dsigma, cudaStream_t s);
acid_status guided_euler_update(float* latent, const float* v_cond, const float* v_uncond, int64_t n, float scale,
                               float dsigma, cudaStream_t s);
acid_status guided_euler_update_sig(float* latent, const float* v_cond, const float* v_uncond, int64_t n, float scale,
                                   const double* sig, const int* step, cudaStream_t s);
// Variants that read the step index from device memory (graph-launched loops):
// t = 1000 sig[*step]; dsigma = sig[*step + 1] - sig[*step].
acid_status euler_update_sig(float* latent, const float* v, int64_t n, const double* sig, const int* step,
                             cudaStream_t s);
acid_status timestep_sinusoid_sig(float* out, const double* sig, const int* step, int dim, cudaStream_t s);

}  // namespace acid
