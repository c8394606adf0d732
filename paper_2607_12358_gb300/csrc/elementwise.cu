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
      if (i < nvec) {
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
  if (threadIdx.x == 0) {
    const double num = sn[0], den = sd[0];
    double rel;
    if (den == 0.0) rel = (num == 0.0) ? 0.0 : INFINITY;
    else rel = num / den;
    result[0] = rel;
    result[1] = num;
    result[2] = den;
  }
}

template <typename T>
__global__ void __launch_bounds__(kThreads) add_vec_kernel(const T* __restrict__ a, const T* __restrict__ b, T* out,
                                                           int64_t n) {
  constexpr int V = Vec<T>::N;
  const int64_t nvec = n / V;
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = tid; i < nvec; i += stride) {
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
    if (c < d) {
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
      store8(yr + c, o);
    }
  }
}

// ------------------------------------------------- fused TEMNI + drift
// TEMNI_cur = LN(x) (1 + scale) + shift (fp32) and, in the same pass, the
// sums |TEMNI_cur - TEMNI_prev| and |TEMNI_prev| for the relative-L1 drift.
// The two TEMNI buffers alternate with the step's parity: cur = tem[step & 1],
// prev = tem[(step + 1) & 1]; `step` is read from device memory when
// step_dev is given (graph-launched loops), else step_host is used.  At step
// 0 there is no previous TEMNI and the sums are zero.  One warp per row
// (grid-strided), fp64 CTA partials reduced by drift_final_kernel.
// NV: 8-element vectors per lane (d <= 256 * NV), so that the row held in
// registers is sized to d.  For rows up to 1536 wide the previous TEMNI row
// is loaded together with x: a row then costs one DRAM round trip, not two.
// The arithmetic and its order do not depend on NV.
template <int NV>
__global__ void __launch_bounds__(kThreads, 2) ln_mod_drift_kernel(const float* __restrict__ x, float* tem0,
                                                                   float* tem1, const int* step_dev, int step_host,
                                                                   int64_t rows, int d,
                                                                   const float* __restrict__ shift,
                                                                   const float* __restrict__ scale, float eps,
                                                                   double2* __restrict__ partials) {
  constexpr bool kPrevEarly = NV <= 6;
  const int step = step_dev ? *step_dev : step_host;
  float* cur = (step & 1) ? tem1 : tem0;
  const float* prev = (step & 1) ? tem0 : tem1;
  const bool has_prev = step > 0;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t gw = (int64_t)blockIdx.x * (kThreads / 32) + warp;
  const int64_t nw = (int64_t)gridDim.x * (kThreads / 32);
  float num = 0.f, den = 0.f;
  for (int64_t row = gw; row < rows; row += nw) {
    const float* xr = x + row * d;
    const float* pr = prev + row * d;
    float v[NV][8];
    float pe[kPrevEarly ? NV : 1][8];
#pragma unroll
    for (int i = 0; i < NV; ++i) {
      const int c = (i * 32 + lane) * 8;
      if (c < d) {
        load8(xr + c, v[i]);
        if constexpr (kPrevEarly) {
          if (has_prev) load8(pr + c, pe[i]);
        }
      }
    }
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < NV; ++i) {
      const int c = (i * 32 + lane) * 8;
      if (c < d) {
#pragma unroll
        for (int j = 0; j < 8; ++j) s += v[i][j];
      }
    }
    const float mean = warp_sum_f(s) / d;
    float q = 0.f;
#pragma unroll
    for (int i = 0; i < NV; ++i) {
      const int c = (i * 32 + lane) * 8;
      if (c < d) {
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const float t = v[i][j] - mean;
          q += t * t;
        }
      }
    }
    const float rstd = rsqrtf(warp_sum_f(q) / d + eps);
#pragma unroll
    for (int i = 0; i < NV; ++i) {
      const int c = (i * 32 + lane) * 8;
      if (c < d) {
        float a[8], b[8];
        load8(scale + c, a);
        load8(shift + c, b);
        float* o = v[i];  // the output replaces the input in place
#pragma unroll
        for (int j = 0; j < 8; ++j) o[j] = fmaf((o[j] - mean) * rstd, 1.0f + a[j], b[j]);
        store8(cur + row * d + c, o);
        if (has_prev) {
          float pl[kPrevEarly ? 1 : 8];
          const float* p = pl;
          if constexpr (kPrevEarly) {
            p = pe[i];
          } else {
            load8(pr + c, pl);
          }
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            num += fabsf(o[j] - p[j]);
            den += fabsf(p[j]);
          }
        }
      }
    }
  }
  __shared__ double sn[kThreads / 32], sd[kThreads / 32];
  double dn = warp_sum_d((double)num), dd = warp_sum_d((double)den);
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
    io<TO>::st(tok + i, lat[src]);
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
  const int grid = grid_for(n);
  using H = __nv_bfloat16;
#define ACID_ADD(TA, TB, TO) \
  add_mixed_kernel<TA, TB, TO><<<grid, kThreads, 0, s>>>((const TA*)a, (const TB*)b, (TO*)out, n, bs)
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

acid_status ln_mod_drift(const float* x, float* tem0, float* tem1, const int* step_dev, int step_host, int64_t rows,
                         int d, const float* shift, const float* scale, float eps, double* d_result, void* workspace,
                         size_t ws_bytes, cudaStream_t s) {
  ACID_REQUIRE(d % 8 == 0 && d <= 256 * kLnMaxV, ACID_ERR_UNSUPPORTED, "ln_mod_drift: d must be a multiple of 8, <= 3072");
  ACID_REQUIRE(ws_bytes >= sizeof(double2) * kDriftMaxBlocks, ACID_ERR_WORKSPACE, "ln_mod_drift: workspace too small");
  double2* parts = static_cast<double2*>(workspace);
  const int64_t want = (rows * 32 + kThreads - 1) / kThreads;
  const int grid = (int)std::min<int64_t>(kDriftMaxBlocks, std::max<int64_t>(1, want));
  ProfScope prof(PROF_DRIFT, (double)rows * d * 12.0, s);  // read x and prev, write cur (fp32)
  if (d <= 256 * 4)
    ln_mod_drift_kernel<4><<<grid, kThreads, 0, s>>>(x, tem0, tem1, step_dev, step_host, rows, d, shift, scale, eps, parts);
  else if (d <= 256 * 6)
    ln_mod_drift_kernel<6><<<grid, kThreads, 0, s>>>(x, tem0, tem1, step_dev, step_host, rows, d, shift, scale, eps, parts);
  else if (d <= 256 * 8)
    ln_mod_drift_kernel<8><<<grid, kThreads, 0, s>>>(x, tem0, tem1, step_dev, step_host, rows, d, shift, scale, eps, parts);
  else
    ln_mod_drift_kernel<kLnMaxV><<<grid, kThreads, 0, s>>>(x, tem0, tem1, step_dev, step_host, rows, d, shift, scale,
                                                           eps, parts);
  ACID_CHECK_LAUNCH();
  drift_final_kernel<<<1, kThreads, 0, s>>>(parts, grid, d_result);
  ACID_CHECK_LAUNCH();
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
