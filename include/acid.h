/*
 * acid.h — C ABI of the GB300 (sm_103a) hot path behind ACID, adaptive
 * dual-threshold step caching for video diffusion transformers
 * (arXiv 2607.12358).
 *
 * The library computes, on one GPU, the per-step evaluation of a video DiT
 * denoiser and the cheap drift reductions that decide whether a step is
 * computed or reused (Sec. 2 "TeaCache" / "EasyCache" / "DiCache", Sec. 3.3,
 * Algorithm 1), around an Euler flow-matching sampler, with or without
 * classifier-free guidance.  Every call takes plain pointers and sizes.
 *
 * Conventions shared by all entry points
 *  - Pointers named "device" must point to memory on the current CUDA device.
 *    The caller owns every buffer, including workspaces; the library keeps no
 *    pointer after a call returns and allocates no device memory in any call.
 *  - Weight matrices are row-major [out, in] (the nn.Linear convention) in the
 *    block's dtype; biases are fp32 [out] and may be NULL (treated as zero).
 *  - Token rows are row-major [rows, d].  Joint (text + video) sequences hold
 *    the text rows first.
 *  - Unless stated otherwise a call is asynchronous on `stream` (NULL = the
 *    legacy default stream).  Argument errors are reported before anything is
 *    launched.  Every call returns an acid_status; on failure
 *    acid_last_error() gives a message (thread-local).
 *  - Device-side waits are bounded.  A wait that runs out sets a device flag
 *    that acid_check_device_error() reports as ACID_ERR_TIMEOUT.
 *  - One CUDA device per process.  The kernels' shared-memory attributes and
 *    the SM count used to size persistent grids are set up at the first call,
 *    for the device current then.  Several GPUs are served by one process
 *    each; a call on another device of the same process may fail with
 *    ACID_ERR_CUDA.  Calls that share a workspace must be ordered by their
 *    streams.
 */
#ifndef ACID_H_
#define ACID_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* acid_stream_t; /* a cudaStream_t */

typedef enum {
  ACID_OK = 0,
  ACID_ERR_INVALID_ARG = 1,  /* NULL pointer, bad size, inconsistent shape */
  ACID_ERR_UNSUPPORTED = 2,  /* shape or alignment the kernels do not cover */
  ACID_ERR_WORKSPACE = 3,    /* workspace missing or smaller than required */
  ACID_ERR_CUDA = 4,         /* a CUDA runtime/driver call failed */
  ACID_ERR_TIMEOUT = 5       /* a bounded device-side wait ran out */
} acid_status;

typedef enum { ACID_BF16 = 0, ACID_FP32 = 1 } acid_dtype;

typedef enum {
  ACID_BLOCK_WAN = 0,       /* self-attn (3D RoPE) + cross-attn to text + FFN; n_text = 0: no cross-attn */
  ACID_BLOCK_COG = 1,       /* joint [text; video] attention, shared weights, per-stream modulation */
  ACID_BLOCK_HV_DUAL = 2,   /* joint attention, separate text/video weights */
  ACID_BLOCK_HV_SINGLE = 3  /* joint single stream, parallel attention + MLP */
} acid_block_kind;

typedef enum {
  ACID_METHOD_TEACACHE = 0,   /* Sec. 2 "TeaCache": drift of block 0's modulated input */
  ACID_METHOD_EASYCACHE = 1,  /* Sec. 2 "EasyCache": k * input change / output magnitude */
  ACID_METHOD_DICACHE = 2     /* Sec. 2 "DiCache": drift of shallow probe-block features */
} acid_method;

/* Message of the last failed call on this thread ("" if none). */
const char* acid_last_error(void);
/* Library version string. */
const char* acid_version(void);
/* Synchronises the current device and reports (then clears) the flag set by a
 * timed-out device wait: ACID_OK or ACID_ERR_TIMEOUT.  Synchronous. */
acid_status acid_check_device_error(void);

/* Diagnostic of the failure path: launches one CTA whose thread waits on an
 * mbarrier that nothing arrives on, through the same bounded wait as the
 * kernels but with a budget of `budget_cycles` SM clocks (1e3..1e10).  The
 * wait runs out, raises the device flag and the kernel returns normally, so
 * the next acid_check_device_error() reports ACID_ERR_TIMEOUT and the context
 * stays usable.  Synchronises `stream`. */
acid_status acid_selftest_wait_timeout(int64_t budget_cycles, acid_stream_t stream);

/* Memory-index checks of the debug build.  The library built with
 * `python -m paper_2607_12358_gb300.build --debug` (libacid_gb300_debug.so,
 * compiled with ACID_BOUNDS_CHECK) checks the global-memory index of every
 * hand-computed access in the element-wise, LayerNorm, drift, patch, GEMV,
 * GEMM-epilogue and attention-merge kernels against the extent the host
 * passed; an index outside it is not accessed and the first one per source
 * file is recorded.  Accesses by the TMA engine are bounded by their tensor
 * maps.  Synchronises the device and reports, then clears, the first
 * recorded violation: *site = 0 if there is none, else a kernel-site code,
 * with the index and the extent.  *checked = 1 in the debug build, 0 in the
 * release build (which records nothing). */
acid_status acid_bounds_report(int32_t* checked, int64_t* site, int64_t* index, int64_t* extent);

/* Diagnostic of the index checks: one thread evaluates a check one past the
 * end of an extent of 1000, with no memory access behind it.  In the debug
 * build the next acid_bounds_report gives site 99, index 1000, extent 1000.
 * Synchronises `stream`. */
acid_status acid_selftest_bounds(acid_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Tracing: launch counting and per-launch device timing                     */
/* ------------------------------------------------------------------------ */

typedef enum {
  ACID_PROF_ATTENTION = 0,   /* work = 4 nq nk head_dim heads FLOPs */
  ACID_PROF_LINEAR = 1,      /* work = 2 M N K FLOPs (tcgen05 GEMMs) */
  ACID_PROF_DRIFT = 2        /* work = algorithmic bytes read + written */
} acid_prof_kind;

/* Number of kernels this library has launched since it was loaded. */
int64_t acid_launch_count(void);
/* on != 0: synchronises the device, clears earlier records and starts
 * recording a CUDA event pair around every attention, tcgen05 linear and
 * drift launch, on the launching stream.  on == 0 stops recording. */
acid_status acid_profile_enable(int32_t on);
/* Synchronises the device and sums the recorded launches of `kind`:
 * launch count, total device milliseconds and total algorithmic work. */
acid_status acid_profile_read(int32_t kind, int64_t* launches, double* total_ms, double* work);

/* ------------------------------------------------------------------------ */
/* Drift signal and cache apply (Sec. 2 "TeaCache", "EasyCache")            */
/* ------------------------------------------------------------------------ */

/* Bytes of device workspace acid_drift_signal needs for n elements. */
acid_status acid_drift_workspace_size(int64_t n, size_t* bytes);

/* TeaCache drift between consecutive tensors (Sec. 2, "TeaCache": L1 distance
 * between consecutive modulated inputs, taken relative to the previous one):
 *     rel_l1 = sum_i |cur_i - prev_i| / sum_i |prev_i|
 * accumulated in fp32 per thread and fp64 across threads, in a fixed order
 * (deterministic).  A zero denominator gives 0 if the numerator is 0, else
 * +inf.
 *   prev, cur    device, n elements of `dtype`, 16-byte aligned.
 *   n            element count, >= 0 (n = 0 gives 0).
 *   out_rel_l1   device or host double.  A host pointer makes the call
 *                synchronous on `stream`.
 *   out_sums     optional (NULL), device or host double[2] =
 *                {sum|cur - prev|, sum|prev|}; same host rule.
 *   workspace    device, >= acid_drift_workspace_size(n) bytes, 16-aligned.
 */
acid_status acid_drift_signal(const void* prev, const void* cur, int64_t n, int32_t dtype,
                              double* out_rel_l1, double* out_sums, void* workspace,
                              size_t workspace_bytes, acid_stream_t stream);

/* TeaCache signal straight from two consecutive steps' patch embeddings
 * (Sec. 2, "TeaCache": the drift of the timestep-embedding-modulated noisy
 * input, TEMNI).  With TEMNI_t = LN(h_t) (1 + scale_t) + shift_t row by row
 * (LayerNorm without affine parameters, epsilon eps) it returns
 *     rel_l1 = sum |TEMNI_t - TEMNI_{t-1}| / sum |TEMNI_{t-1}|
 * as acid_drift_signal does, but forms both TEMNIs in registers in one
 * read-only pass over the two fp32 inputs (8 bytes read per element, nothing
 * written but the result): the step loop keeps each step's h and modulation
 * instead of a stored TEMNI.
 *   h_prev, h_cur      device fp32 [rows, d], row-major, 16-byte aligned.
 *   mod_prev, mod_cur  device fp32 [2 d] = {shift[d], scale[d]} of each step.
 *   rows >= 0; d % 8 == 0 and d <= 3072, else ACID_ERR_UNSUPPORTED.
 *   out_rel_l1, out_sums   as acid_drift_signal (device or host; host makes
 *                          the call synchronous).
 *   workspace  device, >= acid_drift_workspace_size(rows * d) bytes,
 *              16-byte aligned.
 * rows = 0 gives 0 (and zero sums). */
acid_status acid_temni_drift(const float* h_prev, const float* h_cur, const float* mod_prev, const float* mod_cur,
                             int64_t rows, int32_t d, float eps, double* out_rel_l1, double* out_sums,
                             void* workspace, size_t workspace_bytes, acid_stream_t stream);

/* Cached-residual reuse on a skipped step (Sec. 2 "TeaCache": previous output
 * reconstructed with a stored residual; "EasyCache": input plus the offset of
 * the last computed step):  out = x + cached_residual, elementwise, rounded
 * once to `dtype`.
 *   x, cached_residual, out   device, n elements, 16-byte aligned; out may
 *                             alias x or cached_residual.
 */
acid_status acid_cache_apply(const void* x, const void* cached_residual, void* out, int64_t n,
                             int32_t dtype, acid_stream_t stream);

/* acid_drift_signal without a workspace, for callers that cannot allocate
 * any device memory: for example a plugin that is handed only its input and
 * output buffers by a host framework, or a process whose device memory is
 * fully reserved by another allocator.  The paper has no counterpart: this is
 * a deployment variant of the drift reduction above, with the same result.
 *   Arguments and outputs as acid_drift_signal (device or host outputs).
 *   n          0 <= n <= 2^31; larger n fails with ACID_ERR_UNSUPPORTED (the
 *              limit keeps the worst-case fp32 rounding of the per-thread sums
 *              inside the 1e-3 drift tolerance).
 * Scratch: a 16 KiB array in the library's device memory, held by every GPU
 * that loads the library until the process exits.  No cudaMalloc, cudaFree
 * or allocating library call is made.  The first call on each device looks
 * up the array's device address (cudaGetSymbolAddress); make that first call
 * outside any stream capture.  The lookup is repeated when the device's
 * context has been replaced (cudaDeviceReset reloads the library's device
 * code at a new address); the first call after a reset is again a set-up
 * call.  All calls share the array and it keeps the last call's contents:
 * calls that overlap on the GPU (different streams without ordering) race and
 * give undefined results. */
acid_status acid_drift_signal_noalloc(const void* prev, const void* cur, int64_t n, int32_t dtype,
                                      double* out_rel_l1, double* out_sums, acid_stream_t stream);

/* Drift and reuse in one pass over HBM (the two calls above fused):
 * rel_l1(prev, cur) as acid_drift_signal and out = cur + cached_residual.
 * Same argument rules; out may alias cur or cached_residual. */
acid_status acid_drift_apply(const void* prev, const void* cur, const void* cached_residual,
                             void* out, int64_t n, int32_t dtype, double* out_rel_l1,
                             double* out_sums, void* workspace, size_t workspace_bytes,
                             acid_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Kernel-level entry points: the building blocks of acid_dit_block_forward, */
/* exposed for testing and for callers composing their own blocks.           */
/* ------------------------------------------------------------------------ */

typedef enum {
  ACID_EPI_BIAS = 0,         /* out = acc + b */
  ACID_EPI_GELU = 1,         /* out = gelu_tanh(acc + b) */
  ACID_EPI_GATED_RES = 3,    /* out = residual + gate[col] * (acc + b) */
  ACID_EPI_RES = 4           /* out = residual + acc + b */
} acid_epilogue;

/* Linear layer with a fused epilogue: out[M, N] = epi(A[M, K] W[N, K]^T + b).
 *   A          device [M, K] row stride lda (elements), dtype.
 *   W          device [N, K] contiguous, dtype; bias fp32 [N] or NULL.
 *   out        device [M, N] row stride ldo; fp32 if out_fp32 else dtype.
 *   gate       fp32 [N] (ACID_EPI_GATED_RES), residual [M, N] row stride ldr
 *              in the output dtype (may equal out: in place).
 * bf16 runs on tcgen05 (fp32 accumulation): N % 32 == 0, K % 8 == 0, rows
 * 16-byte aligned.  fp32 runs on the FP32 pipes: N even.  M = 0 returns
 * ACID_OK without a launch (the pointers may then be NULL). */
acid_status acid_linear_forward(int32_t dtype, const void* A, int64_t lda, int64_t M, int32_t K,
                                const void* W, const float* bias, int32_t N, void* out, int64_t ldo,
                                int32_t epilogue, const float* gate, const void* residual,
                                int64_t ldr, int32_t out_fp32, acid_stream_t stream);

/* Multi-head attention softmax(q k^T / sqrt(head_dim)) v, per head h reading
 * columns [h*head_dim, (h+1)*head_dim) of q (row stride ldq), k (ldk), v (ldv)
 * and writing the same columns of out (ldo).  nk >= 1 key rows; nq = 0
 * returns ACID_OK without a launch (q and out may then be NULL).  bf16 runs on
 * tcgen05 with head_dim 64 or 128; fp32 with head_dim a multiple of 32, <= 128.
 *   workspace  optional (NULL, 0): device scratch of
 *              acid_attention_workspace_size bytes.  With it, and a key range
 *              of more than 8 key tiles (1024 keys at head_dim 128, 512 at
 *              64), the work that would run as a last, partly filled wave of
 *              CTAs is split along the key range and merged (same result up
 *              to summation order).  Shorter key ranges run on persistent
 *              CTAs and do not use it. */
acid_status acid_attention_forward(int32_t dtype, const void* q, int64_t ldq, const void* k,
                                   int64_t ldk, const void* v, int64_t ldv, void* out, int64_t ldo,
                                   int64_t nq, int64_t nk, int32_t heads, int32_t head_dim,
                                   void* workspace, size_t workspace_bytes, acid_stream_t stream);
/* Bytes of the optional acid_attention_forward workspace for head_dim (the
 * partial results of a split last wave: kept for 160 CTAs of 256 rows, fp32
 * output rows plus the running max and sum). */
acid_status acid_attention_workspace_size(int32_t head_dim, size_t* bytes);

/* adaLN LayerNorm: y = LN(x) * (1 + scale) + shift per row of x [rows, d]
 * (no affine part, epsilon eps); shift / scale fp32 [d] or both NULL.
 * x and y may have different dtypes (x_dtype, y_dtype). */
acid_status acid_layernorm_mod(int32_t x_dtype, const void* x, int32_t y_dtype, void* y,
                               int64_t rows, int32_t d, const float* shift, const float* scale,
                               float eps, acid_stream_t stream);

/* ------------------------------------------------------------------------ */
/* DiT block forward: the denoiser f_theta the method skips (Sec. 3.1, Eq. 2;  */
/* Algorithm 1 runs it on computed steps).  The paper names the models         */
/* (Sec. 4.1) but not their blocks; the block definitions follow the          */
/* adaLN-zero DiT form:                                                       */
/*   WAN:  x += g1*O(Attn_RoPE(QKV(LNmod1 x))); x += O_c(Attn(Q_c(LN x),       */
/*         KV_c(ctx))); x += g2*W2 GELU(W1 LNmod2 x); mod = 6d                 */
/*   COG:  the same without cross-attention over [text; video], one weight    */
/*         set, mod = video 6d then text 6d                                   */
/*   HV_DUAL: as COG with separate text/video weights (t_* fields)            */
/*   HV_SINGLE: h = LNmod x; x += g*W2[Attn_RoPE(h W_qkv) | GELU(h W_mlp)];   */
/*         mod = 3d                                                           */
/* LayerNorm has no affine part; modulation vectors are W_mod SiLU(temb) + b. */
/* ------------------------------------------------------------------------ */

typedef struct {
  int32_t kind;        /* acid_block_kind */
  int32_t dtype;       /* acid_dtype of activations and weight matrices */
  int32_t d;           /* hidden width; d % 64 == 0 */
  int32_t heads;       /* head_dim = d / heads must be 64 or 128 */
  int32_t ffn;         /* FFN / MLP width; ffn % 64 == 0 */
  int32_t grid_f, grid_h, grid_w; /* video token grid (after patchify) */
  int64_t n_text;      /* WAN: cross-attention context rows (0: none); COG/HV: joint text rows */
  float rope_theta;    /* RoPE base, e.g. 10000 */
  float ln_eps;        /* LayerNorm epsilon, e.g. 1e-6 */
} acid_block_desc;

typedef struct {
  const void* w;       /* device [out, in], desc dtype */
  const float* b;      /* device fp32 [out] or NULL */
} acid_linear;

typedef struct {
  /* WAN / COG / HV_DUAL video stream / HV_SINGLE */
  acid_linear mod;     /* [6d|12d|6d|3d, d] */
  acid_linear qkv;     /* [3d, d] */
  acid_linear o;       /* [d, d]   (unused by HV_SINGLE) */
  acid_linear ff1;     /* [ffn, d] (HV_SINGLE: the MLP input W_mlp) */
  acid_linear ff2;     /* [d, ffn] (HV_SINGLE: W2 [d, d + ffn]) */
  /* WAN cross-attention (n_text > 0) */
  acid_linear cq;      /* [d, d] */
  acid_linear ckv;     /* [2d, d] */
  acid_linear co;      /* [d, d] */
  /* HV_DUAL text stream */
  acid_linear t_mod, t_qkv, t_o, t_ff1, t_ff2;
} acid_block_weights;

typedef struct {
  const float* temb;   /* device fp32 [d]: timestep embedding after the time MLP */
  const void* ctx;     /* WAN with n_text > 0: device [n_text, d] text context, desc dtype */
  const void* ctx_kv;  /* optional (NULL): WAN with n_text > 0: device [n_text, 2d], desc dtype,
                          16-byte aligned, this block's cross-attention keys and values
                          ctx W_ckv^T + b_ckv (keys in columns [0, d), values in [d, 2d)).
                          The text is fixed for a generation, so a caller running many
                          steps computes them once per block (acid_denoise_* do); given,
                          the block reads them and ctx may be NULL. */
} acid_cond;

/* Rows of x for a block: n_video (WAN) or n_text + n_video (COG/HV). */
acid_status acid_block_rows(const acid_block_desc* desc, int64_t* rows);
/* Bytes of device workspace acid_dit_block_forward needs. */
acid_status acid_block_workspace_size(const acid_block_desc* desc, size_t* bytes);

/* One DiT block, in place on x.
 *   x          device [rows, d] (acid_block_rows), desc dtype, updated in place.
 *   cond       host struct of device pointers.
 *   w          host struct of device pointers; fields the kind does not use
 *              are ignored.
 *   workspace  device, >= acid_block_workspace_size bytes, 1024-byte aligned.
 * bf16 runs on tcgen05 tensor cores (fp32 accumulation); fp32 runs on the
 * FP32 pipes.  Fails with ACID_ERR_UNSUPPORTED on head_dim not in {64, 128}
 * (bf16) or d, ffn not multiples of 64. */
acid_status acid_dit_block_forward(const acid_block_desc* desc, void* x, const acid_cond* cond,
                                   const acid_block_weights* w, void* workspace,
                                   size_t workspace_bytes, acid_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Denoising loop with the dual-threshold switch (Algorithm 1, Sec. 3.3)      */
/* ------------------------------------------------------------------------ */

typedef struct {
  acid_block_desc block;     /* shape shared by all blocks; kind = first block's kind */
  int32_t n_blocks;          /* WAN/COG: blocks; HV: dual-stream blocks */
  int32_t n_single;          /* HV: single-stream blocks after the dual ones */
  const acid_block_weights* blocks; /* host array [n_blocks + n_single] */
  int32_t latent_c, latent_f, latent_h, latent_w; /* latent [C, F, H, W] */
  int32_t pt, ph, pw;        /* patch size; grid = (F/pt, H/ph, W/pw) */
  int32_t time_freq_dim;     /* sinusoid width (256) */
  int32_t d_text;            /* raw text width (WAN: projected by `text`) */
  acid_linear patch;         /* [d, C*pt*ph*pw] */
  acid_linear time1;         /* [d, time_freq_dim] */
  acid_linear time2;         /* [d, d] */
  acid_linear text;          /* WAN: [d, d_text] */
  acid_linear final_mod;     /* [2d, d] -> shift, scale */
  acid_linear final_out;     /* [C*pt*ph*pw, d] */
} acid_model;

typedef struct {
  int32_t n_steps;           /* Euler steps N: sigma_i = 1 - i/N (shifted) */
  int32_t warmup;            /* steps that always run the model (M.warmup) */
  int32_t method;            /* acid_method */
  int32_t force_last;        /* 1: always compute the final step */
  double tau_low, tau_high;  /* thresholds; tau_low == tau_high is fixed-tau caching */
  double delta;              /* stability bound on |s_t - s_prev| */
  double shift;              /* sigma shift s (1 = none) */
  const int8_t* forced;      /* host [n_steps] or NULL: -1 controller, 0 reuse, 1 compute */
  int32_t probe_blocks;      /* DiCache: blocks run on every step as the probe (>= 1) */
  int32_t signal_poly_n;     /* 0: raw signal; else coefficients in signal_poly (<= 8) */
  const double* signal_poly; /* host [signal_poly_n], ascending powers: the controller
                                sees s' = sum_j c_j s^j (TeaCache's calibrated rescaling
                                of its raw drift; not part of Algorithm 1 itself) */
  const double* tau_schedule;/* host [n_steps] or NULL: a finite entry fixes the threshold
                                of that step (overriding the delta rule; a low-then-high
                                schedule is the fixed transition-point dual threshold of
                                Sec. 3.2); NaN entries keep the delta rule */
} acid_loop_cfg;

typedef struct {
  int32_t step, warmup, computed, forced;
  double t;                  /* timestep 1000 * sigma_i */
  double signal;             /* s_t (NaN on warmup steps) */
  double dsignal;            /* |s_t - s_prev| (NaN if s_prev is None) */
  double tau;                /* active threshold (NaN on warmup steps) */
  double sigma;              /* accumulated drift compared with tau */
  double ms;                 /* device time of the step */
} acid_step_log;

/* Controller and cache state carried between steps (plain data). */
typedef struct {
  int32_t step;              /* next step index */
  int32_t have_prev_signal;  /* s_prev != None */
  int32_t have_cache;        /* a residual / offset is stored */
  int32_t have_rate;         /* EasyCache k is defined */
  double sigma_acc;          /* accumulated drift */
  double s_prev;
  double k_rate;             /* EasyCache transformation rate */
} acid_loop_state;

acid_status acid_loop_workspace_size(const acid_model* m, size_t* bytes);

/* Prepares a generation: zeroes `state`, projects the text features (WAN) or
 * stores the text tokens (COG/HV) into the workspace.  WAN with text also
 * computes every block's cross-attention keys and values from the projected
 * text there, once; the steps read them (acid_cond.ctx_kv).  bf16 models also
 * get the patch weights repeated along K ([W | W]) for the tensor-core patch
 * embedding, and the TEMNI drift's CTA counter is zeroed.  The whole
 * workspace is the generation's state: to resume a generation elsewhere, copy
 * all of it (with `state`).
 *   text      device [n_text, d_text] in the model dtype, or NULL if n_text = 0.
 *   workspace device, >= acid_loop_workspace_size bytes, 1024-byte aligned;
 *             holds the caches between steps, so the same workspace must be
 *             passed to every step of the generation. */
acid_status acid_loop_begin(const acid_model* m, const acid_loop_cfg* cfg, const void* text,
                            acid_loop_state* state, void* workspace, size_t workspace_bytes,
                            acid_stream_t stream);

/* One sampler step i = state->step of Algorithm 1:
 *   t = 1000 sigma_i; temb; patch embedding H_in of the latent;
 *   on non-warmup steps s_t (TeaCache: rel_l1 of block 0's modulated input
 *   between consecutive steps; EasyCache: k mean|x_t - x_{t-1}| /
 *   mean|v_{t-1}|; DiCache: rel_l1 of the probe blocks' output P between
 *   consecutive steps), Sigma += s_t, tau by |s_t - s_prev| <= delta, reuse
 *   iff Sigma <= tau, else run all (remaining) blocks and reset Sigma.
 *   DiCache reuse (a reading; the paper describes it only in words):
 *   H_out = P_t + D_1 + g (D_1 - D_2), D = H_out - P at the last two computed
 *   steps, g = |P_t - P_1|_1 / |P_1 - P_2|_1 (0 when P_1 = P_2);
 *   final layer, x_{i+1} = x_i + (sigma_{i+1} - sigma_i) v.
 *   latent    device fp32 [C, F, H, W], updated in place.
 *   log       host, one entry written, or NULL.
 * Synchronises `stream` once per non-warmup step (the decision is taken on
 * the host from the drift value). */
acid_status acid_denoise_step(const acid_model* m, const acid_loop_cfg* cfg, acid_loop_state* state,
                              void* latent, acid_step_log* log, void* workspace,
                              size_t workspace_bytes, acid_stream_t stream);

/* acid_loop_begin followed by cfg->n_steps calls of acid_denoise_step.
 *   log   host [n_steps] or NULL. */
acid_status acid_denoise_loop(const acid_model* m, const acid_loop_cfg* cfg, void* latent,
                              const void* text, acid_step_log* log, void* workspace,
                              size_t workspace_bytes, acid_stream_t stream);

/* The same generation as acid_denoise_loop, launched as one CUDA graph: a
 * WHILE node whose body is one sampler step.  The drift signal (TeaCache:
 * block 0's modulated input and its relative L1 in one fused pass) and
 * Algorithm 1's decision are computed on the device; the decision selects the
 * compute or the reuse body of a conditional node, so no step waits for the
 * host.  Arithmetic and decisions are those of acid_denoise_loop.
 *   n_steps    <= 1024.
 *   log        host [n_steps] or NULL; entries as acid_denoise_step writes
 *              them, with ms = NaN (steps are not timed individually).
 * Builds, instantiates and launches the graph on `stream`, then synchronises
 * `stream` and destroys the graph.  CUDA graph objects are created by the
 * driver for the duration of the call; no device buffer is allocated. */
acid_status acid_denoise_loop_graph(const acid_model* m, const acid_loop_cfg* cfg, void* latent,
                                    const void* text, acid_step_log* log, void* workspace,
                                    size_t workspace_bytes, acid_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Classifier-free guidance (the paper is silent on guidance)                 */
/* ------------------------------------------------------------------------ */
/* Two branches share the latent: the conditional one (text_cond) and the
 * unconditional one (text_uncond).  Each branch has its own acid_loop_cfg
 * (thresholds, forced decisions, method; n_steps and shift must agree), its
 * own acid_loop_state and its own half of the workspace, so Algorithm 1's
 * Sigma and s_prev and the base method's cache are kept per branch and the
 * branches decide independently.  Step i evaluates both branches on x_i
 * (conditional first) and then x_{i+1} = x_i + (sigma_{i+1} - sigma_i)
 * (v_u + g (v_c - v_u)), g = guidance_scale.
 * Workspace: >= acid_guided_workspace_size bytes, 1024-byte aligned; the
 * unconditional half starts at the first 1024-byte boundary past the
 * single-branch loop workspace size. */
acid_status acid_guided_workspace_size(const acid_model* m, size_t* bytes);

/* acid_loop_begin for both branches (texts: device, as acid_loop_begin). */
acid_status acid_guided_begin(const acid_model* m, const acid_loop_cfg* cfg_cond,
                              const acid_loop_cfg* cfg_uncond, const void* text_cond,
                              const void* text_uncond, acid_loop_state* state_cond,
                              acid_loop_state* state_uncond, void* workspace,
                              size_t workspace_bytes, acid_stream_t stream);

/* One guided step.  Both states must be at the same step.  log_cond /
 * log_uncond: host, one entry each, or NULL; ms of the conditional entry is
 * that branch's time, ms of the unconditional entry covers that branch and
 * the guided Euler update.  Synchronises once per non-warmup branch step,
 * as acid_denoise_step does.  guidance_scale must be finite. */
acid_status acid_guided_step(const acid_model* m, const acid_loop_cfg* cfg_cond,
                             const acid_loop_cfg* cfg_uncond, double guidance_scale,
                             acid_loop_state* state_cond, acid_loop_state* state_uncond,
                             void* latent, acid_step_log* log_cond, acid_step_log* log_uncond,
                             void* workspace, size_t workspace_bytes, acid_stream_t stream);

/* acid_guided_begin followed by n_steps calls of acid_guided_step.
 *   log_cond, log_uncond   host [n_steps] each, or NULL. */
acid_status acid_denoise_loop_guided(const acid_model* m, const acid_loop_cfg* cfg_cond,
                                     const acid_loop_cfg* cfg_uncond, double guidance_scale,
                                     void* latent, const void* text_cond, const void* text_uncond,
                                     acid_step_log* log_cond, acid_step_log* log_uncond,
                                     void* workspace, size_t workspace_bytes, acid_stream_t stream);

/* The same guided generation as acid_denoise_loop_guided, launched as one
 * CUDA graph (as acid_denoise_loop_graph): per step, both branches' signals
 * and Algorithm 1 decisions are taken on the device, each selecting its own
 * compute or reuse body.  Arithmetic and decisions are those of the
 * host-driven guided loop; log entries have ms = NaN.  n_steps <= 1024. */
acid_status acid_denoise_loop_guided_graph(const acid_model* m, const acid_loop_cfg* cfg_cond,
                                           const acid_loop_cfg* cfg_uncond, double guidance_scale,
                                           void* latent, const void* text_cond, const void* text_uncond,
                                           acid_step_log* log_cond, acid_step_log* log_uncond,
                                           void* workspace, size_t workspace_bytes, acid_stream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* ACID_H_ */
