// HBM-bound kernels of the step: drift reduction (+ fused cache apply),
// adaLN LayerNorm, GEMVs for the timestep and modulation vectors, RoPE
// tables, patchify / unpatchify + Euler update.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace acid {

namespace {

constexpr int kThreads = 256;
constexpr int kDriftMaxBlocks = 152 * 4;  // one wave of 4 CTAs per SM on GB300

int num_sms_elem() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
  }
  return n;
}

__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

template <typename T> struct Vec;  // 16-byte vector of T
template <> struct Vec<__nv_bfloat16> {
  static constexpr int N = 8;
  static __device__ __forceinline__ void ld(const __nv_bfloat16* p, float* v) { load8(p, v); }
  static __device__ __forceinline__ void st(__nv_bfloat16* p, const float* v) { store8(p, v); }
};
template <> struct Vec<float> {
  static constexpr int N = 4;
  static __device__ __forceinline__ void ld(const float* p, float* v) {
    float4 a = *reinterpret_cast<const float4*>(p);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  }
  static __device__ __forceinline__ void st(float* p, const float* v) {
    *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
  }
};

// One pass over prev/cur: per-thread fp32 sums of |cur - prev| and |prev|,
// fp64 across the CTA, one partial per CTA.  kApply also writes
// out = cur + resid in the same pass.  Loads are raw 16-byte vectors, U of
// them in flight per tensor and thread, unpacked after all have been issued.
template <typename T>
__device__ __forceinline__ void unpack16(const uint4& u, float* v);
template <>
__device__ __forceinline__ void unpack16<__nv_bfloat16>(const uint4& u, float* v) {
  v[0] = bf16_lo(u.x); v[1] = bf16_hi(u.x); v[2] = bf16_lo(u.y); v[3] = bf16_hi(u.y);
  v[4] = bf16_lo(u.z); v[5] = bf16_hi(u.z); v[6] = bf16_lo(u.w); v[7] = bf16_hi(u.w);
}
template <>
__device__ __forceinline__ void unpack16<float>(const uint4& u, float* v) {
  v[0] = __uint_as_float(u.x); v[1] = __uint_as_float(u.y); v[2] = __uint_as_float(u.z); v[3] = __uint_as_float(u.w);
}

template <typename T, bool kApply>
__global__ void __launch_bounds__(kThreads, 4) drift_partials_kernel(const T* __restrict__ prev,
                                                                     const T* __restrict__ cur,
                                                                     const T* __restrict__ resid, T* out,
                                                                     int64_t n, double2* __restrict__ partials) {
  constexpr int V = Vec<T>::N;
  constexpr int U = kApply ? 2 : 4;  // 16-byte vectors in flight per thread and tensor
  const int64_t nvec = n / V;
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const uint4* p4 = reinterpret_cast<const uint4*>(prev);
  const uint4* c4 = reinterpret_cast<const uint4*>(cur);
  const uint4* r4 = reinterpret_cast<const uint4*>(resid);
  float num0 = 0.f, num1 = 0.f, den0 = 0.f, den1 = 0.f;
  for (int64_t base = tid; base < nvec; base += U * stride) {
    uint4 pr[U], cr[U], rr[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t i = base + u * stride;
      if (i < nvec && ACID_IN_BOUNDS(kSiteDrift, i * V + V - 1, n)) {
        pr[u] = __ldcs(p4 + i);
        cr[u] = __ldcs(c4 + i);
        if (kApply) rr[u] = __ldcs(r4 + i);
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t i = base + u * stride;
      if (i < nvec) {
        float p[V], c[V];
        unpack16<T>(pr[u], p);
        unpack16<T>(cr[u], c);
#pragma unroll
        for (int j = 0; j < V; j += 2) {
          num0 += fabsf(c[j] - p[j]);
          num1 += fabsf(c[j + 1] - p[j + 1]);
          den0 += fabsf(p[j]);
          den1 += fabsf(p[j + 1]);
        }
        if (kApply) {
          float r[V];
          unpack16<T>(rr[u], r);
#pragma unroll
          for (int j = 0; j < V; ++j) r[j] += c[j];
          Vec<T>::st(out + i * V, r);
        }
      }
    }
  }
  float num = num0 + num1, den = den0 + den1;
  for (int64_t i = nvec * V + tid; i < n; i += stride) {  // ragged tail
    const float pv = io<T>::ld(prev + i), cv = io<T>::ld(cur + i);
    num += fabsf(cv - pv);
    den += fabsf(pv);
    if (kApply) io<T>::st(out + i, cv + io<T>::ld(resid + i));
  }
  __shared__ double sn[kThreads / 32], sd[kThreads / 32];
  double dn = warp_sum_d((double)num), dd = warp_sum_d((double)den);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) { sn[warp] = dn; sd[warp] = dd; }
  __syncthreads();
  if (warp == 0) {
    dn = lane < kThreads / 32 ? sn[lane] : 0.0;
    dd = lane < kThreads / 32 ? sd[lane] : 0.0;
    dn = warp_sum_d(dn);
    dd = warp_sum_d(dd);
    if (lane == 0) partials[blockIdx.x] = make_double2(dn, dd);
  }
}

// {rel, num, den} of the drift from its two sums (zero denominator: 0 when
// the numerator is 0, else +inf).
__device__ __forceinline__ void write_drift_result(double num, double den, double* result) {
  double rel;
  if (den == 0.0) rel = (num == 0.0) ? 0.0 : INFINITY;
  else rel = num / den;
  result[0] = rel;
  result[1] = num;
  result[2] = den;
}

// Fixed-order reduction of the CTA partials; result = {rel, num, den}.
__global__ void __launch_bounds__(kThreads) drift_final_kernel(const double2* __restrict__ partials, int nparts,
                                                               double* __restrict__ result) {
  double n = 0.0, d = 0.0;
  for (int i = threadIdx.x; i < nparts; i += kThreads) {
    n += partials[i].x;
    d += partials[i].y;
  }
  __shared__ double sn[kThreads], sd[kThreads];
  sn[threadIdx.x] = n;
  sd[threadIdx.x] = d;
  __syncthreads();
  for (int s = kThreads / 2; s > 0; s >>= 1) {
    if (threadIdx.x < s) {
      sn[threadIdx.x] += sn[threadIdx.x + s];
      sd[threadIdx.x] += sd[threadIdx.x + s];
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) write_drift_result(sn[0], sd[0], result);
}

template <typename T>
__global__ void __launch_bounds__(kThreads) add_vec_kernel(const T* __restrict__ a, const T* __restrict__ b, T* out,
                                                           int64_t n) {
  constexpr int V = Vec<T>::N;
  const int64_t nvec = n / V;
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = tid; i < nvec; i += stride) {
    if (!ACID_IN_BOUNDS(kSiteAdd, i * V + V - 1, n)) continue;
    float x[V], r[V];
    Vec<T>::ld(a + i * V, x);
    Vec<T>::ld(b + i * V, r);
#pragma unroll
    for (int j = 0; j < V; ++j) x[j] += r[j];
    Vec<T>::st(out + i * V, x);
  }
  for (int64_t i = nvec * V + tid; i < n; i += stride) io<T>::st(out + i, io<T>::ld(a + i) + io<T>::ld(b + i));
}

template <typename TA, typename TB, typename TO>
__global__ void add_mixed_kernel(const TA* __restrict__ a, const TB* __restrict__ b, TO* out, int64_t n, float bs) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
    io<TO>::st(out + i, io<TA>::ld(a + i) + bs * io<TB>::ld(b + i));
}

// The same on eight consecutive values per thread (16-byte aligned operands);
// READ_B false: out = a (b_scale 0, b not read).
template <typename TA, typename TB, typename TO, bool READ_B>
__global__ void add_mixed8_kernel(const TA* __restrict__ a, const TB* __restrict__ b, TO* out, int64_t n, float bs) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  for (int64_t i = tid; i < n / 8; i += stride) {
    if (!ACID_IN_BOUNDS(kSiteAdd, 8 * i + 7, n)) continue;
    float x[8];
    load8(a + 8 * i, x);
    if constexpr (READ_B) {
      float y[8];
      load8(b + 8 * i, y);
#pragma unroll
      for (int j = 0; j < 8; ++j) x[j] = x[j] + bs * y[j];
    }
    store8(out + 8 * i, x);
  }
  for (int64_t i = n / 8 * 8 + tid; i < n; i += stride)
    io<TO>::st(out + i, READ_B ? io<TA>::ld(a + i) + bs * io<TB>::ld(b + i) : io<TA>::ld(a + i));
}

// ---------------------------------------------------------------- LayerNorm
// One warp per row; row kept in registers (d <= 256 * kMaxV).
constexpr int kLnMaxV = 12;

// NV: 8-element vectors per lane (d <= 256 * NV); sized to the row so that
// short rows keep few registers and many rows in flight.  The row stays in
// registers as loaded (bf16 packed, four registers per 8 values) and is
// unpacked in each of the three passes.
template <typename Tin, typename Tout, int NV>
__global__ void __launch_bounds__(kThreads) ln_mod_kernel(const Tin* __restrict__ x, Tout* __restrict__ y,
                                                          int64_t rows, int d, const float* __restrict__ shv,
                                                          const float* __restrict__ scv,
                                                          const float* __restrict__ sht,
                                                          const float* __restrict__ sct, int64_t split, float eps) {
  constexpr int kW = sizeof(Tin) == 2 ? 1 : 2;  // uint4 words per 8 values
  const int64_t row = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const Tin* xr = x + row * d;
  uint4 raw[NV][kW];
  auto unpack = [&](int i, float* f) {
    if constexpr (kW == 1) {
      const uint32_t w[4] = {raw[i][0].x, raw[i][0].y, raw[i][0].z, raw[i][0].w};
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        f[2 * j] = bf16_lo(w[j]);
        f[2 * j + 1] = bf16_hi(w[j]);
      }
    } else {
      const float4 p0 = *reinterpret_cast<const float4*>(&raw[i][0]), p1 = *reinterpret_cast<const float4*>(&raw[i][1]);
      f[0] = p0.x; f[1] = p0.y; f[2] = p0.z; f[3] = p0.w;
      f[4] = p1.x; f[5] = p1.y; f[6] = p1.z; f[7] = p1.w;
    }
  };
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    const int c = (i * 32 + lane) * 8;
    if (c < d && ACID_IN_BOUNDS(kSiteLayerNorm, row * d + c + 7, rows * d)) {
      const uint4* src = reinterpret_cast<const uint4*>(xr + c);
#pragma unroll
      for (int k = 0; k < kW; ++k) raw[i][k] = src[k];
    }
  }
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    const int c = (i * 32 + lane) * 8;
    if (c < d) {
      float f[8];
      unpack(i, f);
#pragma unroll
      for (int j = 0; j < 8; ++j) s += f[j];
    }
  }
  const float mean = warp_sum_f(s) / d;
  float q = 0.f;
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    const int c = (i * 32 + lane) * 8;
    if (c < d) {
      float f[8];
      unpack(i, f);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float t = f[j] - mean;
        q += t * t;
      }
    }
  }
  const float rstd = rsqrtf(warp_sum_f(q) / d + eps);
  const bool text = row < split;
  const float* sh = text ? sht : shv;
  const float* sc = text ? sct : scv;
  Tout* yr = y + row * d;
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    const int c = (i * 32 + lane) * 8;
    if (c < d) {
      float f[8], o[8];
      unpack(i, f);
      if (sc != nullptr) {
        float a[8], b[8];
        load8(sc + c, a);
        load8(sh + c, b);
#pragma unroll
        for (int j = 0; j < 8; ++j) o[j] = fmaf((f[j] - mean) * rstd, 1.0f + a[j], b[j]);
      } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) o[j] = (f[j] - mean) * rstd;
      }
      if (ACID_IN_BOUNDS(kSiteLayerNorm, row * d + c + 7, rows * d)) store8(yr + c, o);
    }
  }
}

// ------------------------------------------- TEMNI drift from two H_in rows
// The sums |TEMNI_t - TEMNI_{t-1}| and |TEMNI_{t-1}| of the TeaCache signal,
// with TEMNI = LN(H_in) (1 + scale) + shift at each step's own (shift,
// scale).  Both TEMNI rows are formed in registers from the fp32 patch
// embeddings H_in_t (xc) and H_in_{t-1} (xp), so the kernel reads 8 bytes per
// element and writes nothing but one fp64 partial pair per CTA (reduced by
// drift_final_kernel, or with a done counter by the CTA that finishes last).
// One warp per row pair (rows counted from the end: gw, gw + total warps, ...
// from the last row down), reductions by warp
// shuffles only.  Lane 0 of each warp streams the warp's row pairs into its
// own two-stage shared-memory ring with 1D bulk copies (completion counted on
// the stage's mbarrier), so the bytes in flight come from shared memory, not
// registers; the stage is refilled as soon as every lane has read it.  The
// four modulation vectors (shift and 1 + scale of both steps) are staged once
// per CTA in shared memory.  Row statistics: mean and variance from sums of
// (x - K) and (x - K)^2 with K the row's first element, which keeps the
// fp32 cancellation small (K lies within a few standard deviations of the
// mean).  HOLD: rows of up to 1536 values stay in registers after one read of
// the stage (16 per lane), else the stage is read again for the final pass.
// Step 0 gives zero sums.
constexpr int kTemniStages = 2;
constexpr int kTemniMaxWarps = 8;

__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(dst)),
               "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}

// The same with an L2 cache policy for the source lines.
__device__ __forceinline__ void bulk_load_hint(void* dst, const void* src, uint32_t bytes, uint64_t* bar,
                                               uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
          smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

template <int NV4, bool HOLD>
__global__ void __launch_bounds__(32 * kTemniMaxWarps, 1) temni_drift_kernel(const float* __restrict__ xc,
                                                                            const float* __restrict__ xp,
                                                                            const int* step_dev, int step_host,
                                                                            int64_t rows, int d,
                                                                            const float* __restrict__ shc,
                                                                            const float* __restrict__ scc,
                                                                            const float* __restrict__ shp,
                                                                            const float* __restrict__ scp, float eps,
                                                                            double2* __restrict__ partials,
                                                                            unsigned int* done, double* result) {
  extern __shared__ __align__(128) uint8_t tsm[];
  const int nwarps = blockDim.x >> 5;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // four d-long vectors: shift_c, 1 + scale_c, shift_p, 1 + scale_p (separate
  // arrays, so that a warp's 16-byte reads of one vector are contiguous)
  float4* mod = reinterpret_cast<float4*>(tsm);
  float* ring = reinterpret_cast<float*>(tsm + (size_t)16 * d);                       // [warp][stage][2][d]
  uint64_t* full = reinterpret_cast<uint64_t*>(ring + (size_t)nwarps * kTemniStages * 2 * d);  // [warp][stage]
  __shared__ double rd[2][kTemniMaxWarps];
  const int step = step_dev ? *step_dev : step_host;
  float* wr = ring + (size_t)warp * kTemniStages * 2 * d;
  uint64_t* wf = full + warp * kTemniStages;
  const int64_t gw = (int64_t)blockIdx.x * nwarps + warp, nw = (int64_t)gridDim.x * nwarps;
  const int64_t n_my = (step > 0 && gw < rows) ? (rows - 1 - gw) / nw + 1 : 0;
  const uint32_t row_bytes = (uint32_t)d * sizeof(float);
  // Rows from the last one down: the patch embedding that writes h_cur just
  // before this kernel leaves its last rows in L2 (dirty), so they are read
  // first.  The previous step's rows are not read again in this step: they
  // are loaded evict-first, so that they, and not those dirty h_cur lines,
  // give way to new lines, and no write-back of h_cur falls into this kernel.
  const uint64_t prev_policy = l2_policy_evict_first();
  auto issue = [&](int64_t k) {
    const int st = (int)(k % kTemniStages);
    int64_t row = rows - 1 - (gw + k * nw);
    if (!ACID_IN_BOUNDS(kSiteTemni, row, rows)) row = 0;  // (debug builds) read row 0 instead
    mbar_expect_tx(&wf[st], 2 * row_bytes);
    bulk_load(wr + (size_t)st * 2 * d, xc + row * d, row_bytes, &wf[st]);
    bulk_load_hint(wr + (size_t)st * 2 * d + d, xp + row * d, row_bytes, &wf[st], prev_policy);
  };
  // each warp's first copies are issued before the modulation vectors are
  // staged, so their latency overlaps the staging
  if (lane == 0) {
    for (int i = 0; i < kTemniStages; ++i) mbar_init(&wf[i], 1);
    mbar_fence_init();
    for (int64_t k = 0; k < n_my && k < kTemniStages; ++k) issue(k);
  }
  for (int i = threadIdx.x; i < d / 4; i += blockDim.x) {
    const float4 a = reinterpret_cast<const float4*>(shc)[i], b = reinterpret_cast<const float4*>(scc)[i];
    const float4 c = reinterpret_cast<const float4*>(shp)[i], e = reinterpret_cast<const float4*>(scp)[i];
    const int q = d / 4;
    mod[i] = a;
    mod[q + i] = make_float4(1.f + b.x, 1.f + b.y, 1.f + b.z, 1.f + b.w);
    mod[2 * q + i] = c;
    mod[3 * q + i] = make_float4(1.f + e.x, 1.f + e.y, 1.f + e.z, 1.f + e.w);
  }
  __syncthreads();  // modulation vectors staged, barriers initialised
  const float inv_d = 1.0f / d;
  float num = 0.f, den = 0.f;
  int64_t k = 0;
  for (; k < n_my; ++k) {
    const int st = (int)(k % kTemniStages);
    const bool ok = __all_sync(0xffffffffu, mbar_wait(&wf[st], (uint32_t)((k / kTemniStages) & 1)));
    if (!ok) break;
    const float4* rc = reinterpret_cast<const float4*>(wr + (size_t)st * 2 * d);
    const float4* rp = rc + d / 4;
    // lane's vectors: i * 32 + lane, i < NV4 (4 columns each)
    float4 cv[HOLD ? NV4 : 1], pv[HOLD ? NV4 : 1];
    const float kc = wr[(size_t)st * 2 * d], kp = wr[(size_t)st * 2 * d + d];  // shifts: the rows' first elements
    float s1c = 0.f, s2c = 0.f, s1p = 0.f, s2p = 0.f;
#pragma unroll
    for (int i = 0; i < NV4; ++i) {
      const int v = i * 32 + lane;
      if (v < d / 4) {
        const float4 c = rc[v], p = rp[v];
        if constexpr (HOLD) {
          cv[i] = c;
          pv[i] = p;
        }
        const float c0 = c.x - kc, c1 = c.y - kc, c2 = c.z - kc, c3 = c.w - kc;
        const float p0 = p.x - kp, p1 = p.y - kp, p2 = p.z - kp, p3 = p.w - kp;
        s1c += (c0 + c1) + (c2 + c3);
        s2c = fmaf(c0, c0, fmaf(c1, c1, fmaf(c2, c2, fmaf(c3, c3, s2c))));
        s1p += (p0 + p1) + (p2 + p3);
        s2p = fmaf(p0, p0, fmaf(p1, p1, fmaf(p2, p2, fmaf(p3, p3, s2p))));
      }
    }
    if (HOLD) {
      __syncwarp();
      if (lane == 0 && k + kTemniStages < n_my) issue(k + kTemniStages);  // every lane holds its values
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      s1c += __shfl_xor_sync(0xffffffffu, s1c, o);
      s2c += __shfl_xor_sync(0xffffffffu, s2c, o);
      s1p += __shfl_xor_sync(0xffffffffu, s1p, o);
      s2p += __shfl_xor_sync(0xffffffffu, s2p, o);
    }
    const float dc = s1c * inv_d, dp = s1p * inv_d;  // mean - K
    const float mc = kc + dc, mp = kp + dp;
    const float rsc = rsqrtf(fmaxf(s2c * inv_d - dc * dc, 0.f) + eps);
    const float rsp = rsqrtf(fmaxf(s2p * inv_d - dp * dp, 0.f) + eps);
#pragma unroll
    for (int i = 0; i < NV4; ++i) {
      const int v = i * 32 + lane;
      if (v < d / 4) {
        float4 c, p;
        if constexpr (HOLD) {
          c = cv[i];
          p = pv[i];
        } else {
          c = rc[v];
          p = rp[v];
        }
        const int q = d / 4;
        const float4 bcv = mod[v], acv = mod[q + v], bpv = mod[2 * q + v], apv = mod[3 * q + v];
        const float cc[4] = {c.x, c.y, c.z, c.w}, pp[4] = {p.x, p.y, p.z, p.w};
        const float ac[4] = {acv.x, acv.y, acv.z, acv.w}, bc[4] = {bcv.x, bcv.y, bcv.z, bcv.w};
        const float ap[4] = {apv.x, apv.y, apv.z, apv.w}, bp[4] = {bpv.x, bpv.y, bpv.z, bpv.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float uc = fmaf((cc[j] - mc) * rsc, ac[j], bc[j]);
          const float up = fmaf((pp[j] - mp) * rsp, ap[j], bp[j]);
          num += fabsf(uc - up);
          den += fabsf(up);
        }
      }
    }
    if (!HOLD) {
      __syncwarp();
      if (lane == 0 && k + kTemniStages < n_my) issue(k + kTemniStages);  // every lane is done with the stage
    }
  }
  // after a wait ran out: the copies already issued land before the CTA exits
  if (k < n_my && lane == 0)
    for (int64_t j = k; j < n_my && j < k + kTemniStages; ++j)
      mbar_wait(&wf[j % kTemniStages], (uint32_t)((j / kTemniStages) & 1));
  double dn = warp_sum_d((double)num), dd = warp_sum_d((double)den);
  if (lane == 0) {
    rd[0][warp] = dn;
    rd[1][warp] = dd;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    dn = 0.0;
    dd = 0.0;
    for (int w = 0; w < nwarps; ++w) {
      dn += rd[0][w];
      dd += rd[1][w];
    }
    partials[blockIdx.x] = make_double2(dn, dd);
  }
  // With a done counter (zero on entry), the CTA that finishes last sums the
  // partials in a fixed order and writes the result, then sets the counter
  // back to zero: no second launch.
  if (done != nullptr) {
    __shared__ bool last;
    if (threadIdx.x == 0) {
      __threadfence();  // this CTA's partial is visible before it is counted
      last = atomicAdd(done, 1u) == gridDim.x - 1;
    }
    __syncthreads();
    if (last && warp == 0) {
      __threadfence();
      double n = 0.0, e = 0.0;
      for (int i = lane; i < (int)gridDim.x; i += 32) {
        const double2 p = __ldcg(&partials[i]);
        n += p.x;
        e += p.y;
      }
      n = warp_sum_d(n);
      e = warp_sum_d(e);
      if (lane == 0) {
        write_drift_result(n, e, result);
        *done = 0u;
      }
    }
  }
}

// ---------------------------------------------------------------- GEMV
template <typename TW>
__global__ void __launch_bounds__(kThreads) gemv_kernel(const TW* __restrict__ W, const float* __restrict__ b,
                                                        const float* __restrict__ x, float* __restrict__ y,
                                                        int n_out, int k, int silu_in) {
  extern __shared__ float xs[];
  for (int i = threadIdx.x; i < k; i += blockDim.x) xs[i] = silu_in ? silu(x[i]) : x[i];
  __syncthreads();
  const int row = blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= n_out) return;
  const TW* wr = W + (int64_t)row * k;
  float acc = 0.f;
  for (int c = lane * 8; c < k; c += 256) {
    if (!ACID_IN_BOUNDS(kSiteGemv, (int64_t)row * k + c + 7, (int64_t)n_out * k)) continue;
    float w[8];
    load8(wr + c, w);
#pragma unroll
    for (int j = 0; j < 8; ++j) acc = fmaf(w[j], xs[c + j], acc);
  }
  acc = warp_sum_f(acc);
  if (lane == 0) y[row] = acc + (b ? b[row] : 0.f);
}

__device__ __forceinline__ void sinusoid_at(float* out, double t, int half, int j) {
  const double f = exp(-log(10000.0) * (double)j / (double)half);
  out[j] = (float)cos(t * f);
  out[half + j] = (float)sin(t * f);
}

__global__ void sinusoid_kernel(float* out, double t, int half) {
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j < half) sinusoid_at(out, t, half, j);
}

// t = 1000 sigma[step] with the step index read from device memory
__global__ void sinusoid_sig_kernel(float* out, const double* sig, const int* step, int half) {
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j < half) sinusoid_at(out, 1000.0 * sig[*step], half, j);
}

__global__ void rope_table_kernel(float2* tbl, int F, int H, int W, int pt, int ph, int pw, double theta) {
  // pt / ph / pw: rotation pairs per axis (t, h, w)
  const int64_t total = (int64_t)F * pt + (int64_t)H * ph + (int64_t)W * pw;
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= total) return;
  int64_t r = i;
  int pos, j, pairs;
  if (r < (int64_t)F * pt) {
    pos = (int)(r / pt); j = (int)(r % pt); pairs = pt;
  } else if ((r -= (int64_t)F * pt) < (int64_t)H * ph) {
    pos = (int)(r / ph); j = (int)(r % ph); pairs = ph;
  } else {
    r -= (int64_t)H * ph;
    pos = (int)(r / pw); j = (int)(r % pw); pairs = pw;
  }
  const double dim = 2.0 * pairs;
  const double ang = (double)pos * pow(theta, -2.0 * j / dim);
  tbl[i] = make_float2((float)cos(ang), (float)sin(ang));
}

// ---------------------------------------------------------------- patches
template <typename TO>
__global__ void patchify_kernel(const float* __restrict__ lat, TO* __restrict__ tok, int C, int F, int H, int W,
                                int pt, int ph, int pw) {
  const int Hp = H / ph, Wp = W / pw;
  const int P = C * pt * ph * pw;
  const int64_t total = (int64_t)(F / pt) * Hp * Wp * P;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += stride) {
    const int64_t n = i / P;
    int p = (int)(i % P);
    const int f = (int)(n / ((int64_t)Hp * Wp)), h = (int)((n / Wp) % Hp), w = (int)(n % Wp);
    const int dw = p % pw; p /= pw;
    const int dh = p % ph; p /= ph;
    const int dt = p % pt; p /= pt;
    const int c = p;
    const int64_t src = (((int64_t)c * F + (f * pt + dt)) * H + (h * ph + dh)) * W + (w * pw + dw);
    if (ACID_IN_BOUNDS(kSitePatchify, src, (int64_t)C * F * H * W)) io<TO>::st(tok + i, lat[src]);
  }
}

// The same gather into bf16 tokens of width 2P that carry each fp32 value as
// the sum of two bf16 parts: hi = bf16(x) in column p, lo = bf16(x - hi) in
// column P + p.  x - hi is exact in fp32 and lo rounds it to 8 bits, so
// hi + lo equals x to within 2^-17 |x|; a bf16 GEMM against the weights
// repeated along K ([W | W]) then forms the fp32-input patch embedding on
// tensor cores.
__global__ void patchify_split_kernel(const float* __restrict__ lat, __nv_bfloat16* __restrict__ tok, int C, int F,
                                      int H, int W, int pt, int ph, int pw) {
  const int Hp = H / ph, Wp = W / pw;
  const int P = C * pt * ph * pw;
  const int64_t total = (int64_t)(F / pt) * Hp * Wp * P;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += stride) {
    const int64_t n = i / P;
    int p = (int)(i % P);
    const int p0 = p;
    const int f = (int)(n / ((int64_t)Hp * Wp)), h = (int)((n / Wp) % Hp), w = (int)(n % Wp);
    const int dw = p % pw; p /= pw;
    const int dh = p % ph; p /= ph;
    const int dt = p % pt; p /= pt;
    const int c = p;
    const int64_t src = (((int64_t)c * F + (f * pt + dt)) * H + (h * ph + dh)) * W + (w * pw + dw);
    if (!ACID_IN_BOUNDS(kSitePatchify, src, (int64_t)C * F * H * W) ||
        !ACID_IN_BOUNDS(kSitePatchify, n * 2 * P + P + p0, total * 2))
      continue;
    const float x = lat[src];
    const __nv_bfloat16 hi = __float2bfloat16_rn(x);
    tok[n * 2 * P + p0] = hi;
    tok[n * 2 * P + P + p0] = __float2bfloat16_rn(x - __bfloat162float(hi));
  }
}

__global__ void unpatchify_euler_kernel(const float* __restrict__ vtok, float* __restrict__ vout, float* lat, int C,
                                        int F, int H, int W, int pt, int ph, int pw, float dsig) {
  const int Hp = H / ph, Wp = W / pw;
  const int P = C * pt * ph * pw;
  const int64_t total = (int64_t)C * F * H * W;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += stride) {
    const int w = (int)(i % W);
    const int h = (int)((i / W) % H);
    const int f = (int)((i / ((int64_t)W * H)) % F);
    const int c = (int)(i / ((int64_t)W * H * F));
    const int64_t n = ((int64_t)(f / pt) * Hp + h / ph) * Wp + w / pw;
    const int p = ((c * pt + f % pt) * ph + h % ph) * pw + w % pw;
    if (!ACID_IN_BOUNDS(kSiteUnpatchify, n * P + p, (int64_t)(F / pt) * Hp * Wp * P)) continue;
    const float v = vtok[n * P + p];
    if (vout) vout[i] = v;
    if (lat) lat[i] = fmaf(dsig, v, lat[i]);
  }
}

__global__ void euler_kernel(float* lat, const float* __restrict__ v, int64_t n, float dsig) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) lat[i] = fmaf(dsig, v[i], lat[i]);
}

// Classifier-free guidance and the Euler step: x += dsig * (v_u + g (v_c - v_u)).
__global__ void guided_euler_kernel(float* lat, const float* __restrict__ vc, const float* __restrict__ vu, int64_t n,
                                    float g, float dsig) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    const float u = vu[i];
    lat[i] = fmaf(dsig, fmaf(g, vc[i] - u, u), lat[i]);
  }
}

// The same with dsigma read from device memory (graph-launched loops).
__global__ void guided_euler_sig_kernel(float* lat, const float* __restrict__ vc, const float* __restrict__ vu,
                                        int64_t n, float g, const double* sig, const int* step) {
  const int i0 = *step;
  const float dsig = (float)(sig[i0 + 1] - sig[i0]);
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    const float u = vu[i];
    lat[i] = fmaf(dsig, fmaf(g, vc[i] - u, u), lat[i]);
  }
}

// dsigma = sigma[step + 1] - sigma[step] with the step index read from device memory
__global__ void euler_sig_kernel(float* lat, const float* __restrict__ v, int64_t n, const double* sig,
                                 const int* step) {
  const int i0 = *step;
  const float dsig = (float)(sig[i0 + 1] - sig[i0]);
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) lat[i] = fmaf(dsig, v[i], lat[i]);
}

int grid_for(int64_t work, int per_block = kThreads, int cap = 152 * 16) {
  int64_t g = (work + per_block - 1) / per_block;
  if (g < 1) g = 1;
  if (g > cap) g = cap;
  return (int)g;
}

}  // namespace

ACID_BOUNDS_READER(take_bounds_elementwise)

// =========================================================================
// host launchers
// =========================================================================

size_t drift_workspace_bytes(int64_t) { return sizeof(double2) * kDriftMaxBlocks + 64; }

acid_status drift_launch(int dtype, const void* prev, const void* cur, const void* resid, void* out, int64_t n,
                         double* d_result, void* workspace, size_t ws_bytes, cudaStream_t s) {
  ACID_REQUIRE(ws_bytes >= sizeof(double2) * kDriftMaxBlocks, ACID_ERR_WORKSPACE, "drift: workspace too small");
  double2* parts = static_cast<double2*>(workspace);
  const int V = dtype == ACID_BF16 ? 8 : 4;
  const int64_t nvec = n / V;
  int grid = (int)std::min<int64_t>(kDriftMaxBlocks, std::max<int64_t>(1, (nvec + kThreads - 1) / kThreads));
  const double esz = dtype == ACID_BF16 ? 2.0 : 4.0;
  ProfScope prof(PROF_DRIFT, (double)n * esz * (resid ? 4.0 : 2.0), s);  // algorithmic bytes
  if (dtype == ACID_BF16) {
    using T = __nv_bfloat16;
    if (resid)
      drift_partials_kernel<T, true><<<grid, kThreads, 0, s>>>((const T*)prev, (const T*)cur, (const T*)resid,
                                                              (T*)out, n, parts);
    else
      drift_partials_kernel<T, false><<<grid, kThreads, 0, s>>>((const T*)prev, (const T*)cur, nullptr, nullptr, n,
                                                               parts);
  } else {
    if (resid)
      drift_partials_kernel<float, true><<<grid, kThreads, 0, s>>>((const float*)prev, (const float*)cur,
                                                                  (const float*)resid, (float*)out, n, parts);
    else
      drift_partials_kernel<float, false><<<grid, kThreads, 0, s>>>((const float*)prev, (const float*)cur, nullptr,
                                                                   nullptr, n, parts);
  }
  ACID_CHECK_LAUNCH();
  drift_final_kernel<<<1, kThreads, 0, s>>>(parts, grid, d_result);
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

acid_status add_same(int dtype, const void* a, const void* b, void* out, int64_t n, cudaStream_t s) {
  const int V = dtype == ACID_BF16 ? 8 : 4;
  const int grid = grid_for(n / V + 1, kThreads, 152 * 8);
  if (dtype == ACID_BF16)
    add_vec_kernel<__nv_bfloat16><<<grid, kThreads, 0, s>>>((const __nv_bfloat16*)a, (const __nv_bfloat16*)b,
                                                            (__nv_bfloat16*)out, n);
  else
    add_vec_kernel<float><<<grid, kThreads, 0, s>>>((const float*)a, (const float*)b, (float*)out, n);
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

acid_status add_mixed(int ad, const void* a, int bd, const void* b, int od, void* out, int64_t n, float bs,
                      cudaStream_t s) {
  using H = __nv_bfloat16;
  const bool vec = aligned(a, 16) && aligned(b, 16) && aligned(out, 16);
  const int grid = vec ? grid_for(n / 8 + 1, kThreads, 152 * 8) : grid_for(n);
#define ACID_ADD(TA, TB, TO)                                                                                   \
  (!vec ? add_mixed_kernel<TA, TB, TO><<<grid, kThreads, 0, s>>>((const TA*)a, (const TB*)b, (TO*)out, n, bs)  \
   : bs == 0.0f                                                                                                \
       ? add_mixed8_kernel<TA, TB, TO, false><<<grid, kThreads, 0, s>>>((const TA*)a, (const TB*)b, (TO*)out, n, \
                                                                       bs)                                   \
       : add_mixed8_kernel<TA, TB, TO, true><<<grid, kThreads, 0, s>>>((const TA*)a, (const TB*)b, (TO*)out, n, bs))
  const int key = ad * 4 + bd * 2 + od;  // ACID_BF16 = 0, ACID_FP32 = 1
  switch (key) {
    case 0: ACID_ADD(H, H, H); break;
    case 1: ACID_ADD(H, H, float); break;
    case 2: ACID_ADD(H, float, H); break;
    case 3: ACID_ADD(H, float, float); break;
    case 4: ACID_ADD(float, H, H); break;
    case 5: ACID_ADD(float, H, float); break;
    case 6: ACID_ADD(float, float, H); break;
    default: ACID_ADD(float, float, float); break;
  }
#undef ACID_ADD
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

template <int NV>
acid_status launch_ln_mod(int in_dtype, int out_dtype, const void* x, void* y, int64_t rows, int d, const float* shv,
                          const float* scv, const float* sht, const float* sct, int64_t split, float eps, int blocks,
                          cudaStream_t s) {
  using H = __nv_bfloat16;
  if (in_dtype == ACID_BF16 && out_dtype == ACID_BF16)
    ln_mod_kernel<H, H, NV><<<blocks, kThreads, 0, s>>>((const H*)x, (H*)y, rows, d, shv, scv, sht, sct, split, eps);
  else if (in_dtype == ACID_BF16)
    ln_mod_kernel<H, float, NV><<<blocks, kThreads, 0, s>>>((const H*)x, (float*)y, rows, d, shv, scv, sht, sct, split,
                                                          eps);
  else if (out_dtype == ACID_BF16)
    ln_mod_kernel<float, H, NV><<<blocks, kThreads, 0, s>>>((const float*)x, (H*)y, rows, d, shv, scv, sht, sct, split,
                                                          eps);
  else
    ln_mod_kernel<float, float, NV><<<blocks, kThreads, 0, s>>>((const float*)x, (float*)y, rows, d, shv, scv, sht, sct,
                                                              split, eps);
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

acid_status ln_mod(int in_dtype, const void* x, int out_dtype, void* y, int64_t rows, int d, const float* shv,
                   const float* scv, const float* sht, const float* sct, int64_t split, float eps, cudaStream_t s) {
  ACID_REQUIRE(d % 8 == 0 && d <= 256 * kLnMaxV, ACID_ERR_UNSUPPORTED, "ln_mod: d must be a multiple of 8, <= 3072");
  if (rows == 0) return ACID_OK;
  if (sht == nullptr) { sht = shv; sct = scv; }
  const int64_t blocks = (rows * 32 + kThreads - 1) / kThreads;
  if (d <= 256 * 4) return launch_ln_mod<4>(in_dtype, out_dtype, x, y, rows, d, shv, scv, sht, sct, split, eps, blocks, s);
  if (d <= 256 * 6) return launch_ln_mod<6>(in_dtype, out_dtype, x, y, rows, d, shv, scv, sht, sct, split, eps, blocks, s);
  if (d <= 256 * 8) return launch_ln_mod<8>(in_dtype, out_dtype, x, y, rows, d, shv, scv, sht, sct, split, eps, blocks, s);
  return launch_ln_mod<kLnMaxV>(in_dtype, out_dtype, x, y, rows, d, shv, scv, sht, sct, split, eps, blocks, s);
}

template <int NV4, bool HOLD>
acid_status launch_temni_drift(const float* h_cur, const float* h_prev, const float* mod_cur, const float* mod_prev,
                               const int* step_dev, int step_host, int64_t rows, int d, float eps, double2* parts,
                               unsigned int* done, double* result, cudaStream_t s, int* grid_out) {
  constexpr int kSmemMax = 226 * 1024;  // dynamic shared memory, below the 227 KB limit less the static part
  static bool attr_done = false;
  if (!attr_done) {
    ACID_CUDA(cudaFuncSetAttribute(temni_drift_kernel<NV4, HOLD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   kSmemMax));
    attr_done = true;
  }
  // warps per CTA: as many two-stage rings (8 d bytes per stage) as fit
  // beside the staged modulation vectors (16 d bytes), at most eight
  const size_t ring_per_warp = (size_t)kTemniStages * 8 * d + kTemniStages * sizeof(uint64_t);
  const int warps = (int)std::max<size_t>(1, std::min<size_t>(kTemniMaxWarps, (kSmemMax - 16 * (size_t)d) /
                                                                                   ring_per_warp));
  const size_t smem = 16 * (size_t)d + warps * ring_per_warp;
  const int grid = (int)std::min<int64_t>(std::min<int64_t>(kDriftMaxBlocks, (int64_t)num_sms_elem()),
                                          std::max<int64_t>(1, (rows + warps - 1) / warps));
  temni_drift_kernel<NV4, HOLD><<<grid, 32 * warps, smem, s>>>(h_cur, h_prev, step_dev, step_host, rows, d, mod_cur,
                                                               mod_cur + d, mod_prev, mod_prev + d, eps, parts,
                                                               done, result);
  ACID_CHECK_LAUNCH();
  *grid_out = grid;
  return ACID_OK;
}

acid_status temni_drift(const float* h_cur, const float* h_prev, const float* mod_cur, const float* mod_prev,
                        const int* step_dev, int step_host, int64_t rows, int d, float eps, double* d_result,
                        void* workspace, size_t ws_bytes, cudaStream_t s, unsigned int* done) {
  ACID_REQUIRE(d % 8 == 0 && d <= 3072, ACID_ERR_UNSUPPORTED, "temni_drift: d must be a multiple of 8, <= 3072");
  ACID_REQUIRE(ws_bytes >= sizeof(double2) * kDriftMaxBlocks, ACID_ERR_WORKSPACE, "temni_drift: workspace too small");
  ACID_REQUIRE(aligned(h_cur, 16) && aligned(h_prev, 16) && aligned(mod_cur, 16) && aligned(mod_prev, 16),
               ACID_ERR_UNSUPPORTED, "temni_drift: inputs must be 16-byte aligned");
  double2* parts = static_cast<double2*>(workspace);
  ProfScope prof(PROF_DRIFT, (double)rows * d * 8.0, s);  // read both steps' H_in (fp32)
  int grid = 1;
  if (d <= 512)
    ACID_TRY((launch_temni_drift<4, true>(h_cur, h_prev, mod_cur, mod_prev, step_dev, step_host, rows, d, eps, parts, done,
                                         d_result, s, &grid)));
  else if (d <= 1536)
    ACID_TRY((launch_temni_drift<12, true>(h_cur, h_prev, mod_cur, mod_prev, step_dev, step_host, rows, d, eps, parts,
                                          done, d_result, s, &grid)));
  else
    ACID_TRY((launch_temni_drift<24, false>(h_cur, h_prev, mod_cur, mod_prev, step_dev, step_host, rows, d, eps, parts,
                                           done, d_result, s, &grid)));
  if (done == nullptr) {
    drift_final_kernel<<<1, kThreads, 0, s>>>(parts, grid, d_result);
    ACID_CHECK_LAUNCH();
  }
  return ACID_OK;
}

acid_status gemv(int w_dtype, const void* W, const float* b, const float* x, float* y, int n_out, int k,
                 bool silu_input, cudaStream_t s) {
  ACID_REQUIRE(k % 8 == 0 && k <= 16384, ACID_ERR_UNSUPPORTED, "gemv: k must be a multiple of 8, <= 16384");
  const int blocks = (n_out + kThreads / 32 - 1) / (kThreads / 32);
  const size_t smem = sizeof(float) * k;
  if (w_dtype == ACID_BF16)
    gemv_kernel<__nv_bfloat16><<<blocks, kThreads, smem, s>>>((const __nv_bfloat16*)W, b, x, y, n_out, k, silu_input);
  else
    gemv_kernel<float><<<blocks, kThreads, smem, s>>>((const float*)W, b, x, y, n_out, k, silu_input);
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

acid_status timestep_sinusoid(float* out, double t, int dim, cudaStream_t s) {
  const int half = dim / 2;
  sinusoid_kernel<<<(half + 127) / 128, 128, 0, s>>>(out, t, half);
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

RopeTable rope_layout(int grid_f, int grid_h, int grid_w, int head_dim) {
  RopeTable t;
  const int dh = 2 * (head_dim / 6);
  const int dt = head_dim - 2 * dh;
  t.grid_f = grid_f; t.grid_h = grid_h; t.grid_w = grid_w;
  t.pairs_t = dt / 2; t.pairs_h = dh / 2; t.pairs_w = dh / 2;
  if (grid_h > 0 && grid_w > 0) {
    t.inv_hw = 1.0f / (float)(grid_h * grid_w);
    t.inv_w = 1.0f / (float)grid_w;
  }
  return t;
}

acid_status rope_build(RopeTable& t, float2* storage, float theta, cudaStream_t s) {
  t.table = storage;
  const int64_t total = t.elems();
  if (total == 0) return ACID_OK;
  rope_table_kernel<<<(int)((total + 127) / 128), 128, 0, s>>>(storage, t.grid_f, t.grid_h, t.grid_w, t.pairs_t,
                                                              t.pairs_h, t.pairs_w, (double)theta);
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

acid_status patchify(const float* latent, int out_dtype, void* tokens, int C, int F, int H, int W, int pt, int ph,
                     int pw, cudaStream_t s) {
  const int64_t total = (int64_t)C * F * H * W;
  const int grid = grid_for(total);
  if (out_dtype == ACID_BF16)
    patchify_kernel<__nv_bfloat16><<<grid, kThreads, 0, s>>>(latent, (__nv_bfloat16*)tokens, C, F, H, W, pt, ph, pw);
  else
    patchify_kernel<float><<<grid, kThreads, 0, s>>>(latent, (float*)tokens, C, F, H, W, pt, ph, pw);
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

acid_status patchify_split(const float* latent, void* tokens, int C, int F, int H, int W, int pt, int ph, int pw,
                           cudaStream_t s) {
  const int64_t total = (int64_t)C * F * H * W;
  patchify_split_kernel<<<grid_for(total), kThreads, 0, s>>>(latent, (__nv_bfloat16*)tokens, C, F, H, W, pt, ph, pw);
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

acid_status unpatchify_euler(const float* vtok, float* v_out, float* latent, int C, int F, int H, int W, int pt,
                             int ph, int pw, float dsigma, cudaStream_t s) {
  const int64_t total = (int64_t)C * F * H * W;
  unpatchify_euler_kernel<<<grid_for(total), kThreads, 0, s>>>(vtok, v_out, latent, C, F, H, W, pt, ph, pw, dsigma);
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

acid_status euler_update(float* latent, const float* v, int64_t n, float dsigma, cudaStream_t s) {
  euler_kernel<<<grid_for(n), kThreads, 0, s>>>(latent, v, n, dsigma);
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

acid_status guided_euler_update(float* latent, const float* v_cond, const float* v_uncond, int64_t n, float scale,
                               float dsigma, cudaStream_t s) {
  guided_euler_kernel<<<grid_for(n), kThreads, 0, s>>>(latent, v_cond, v_uncond, n, scale, dsigma);
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

acid_status guided_euler_update_sig(float* latent, const float* v_cond, const float* v_uncond, int64_t n, float scale,
                                   const double* sig, const int* step, cudaStream_t s) {
  guided_euler_sig_kernel<<<grid_for(n), kThreads, 0, s>>>(latent, v_cond, v_uncond, n, scale, sig, step);
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

acid_status euler_update_sig(float* latent, const float* v, int64_t n, const double* sig, const int* step,
                             cudaStream_t s) {
  euler_sig_kernel<<<grid_for(n), kThreads, 0, s>>>(latent, v, n, sig, step);
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

acid_status timestep_sinusoid_sig(float* out, const double* sig, const int* step, int dim, cudaStream_t s) {
  const int half = dim / 2;
  sinusoid_sig_kernel<<<(half + 127) / 128, 128, 0, s>>>(out, sig, step, half);
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

}  // namespace acid
