// Linear layers of the DiT block.
//
// bf16: persistent tcgen05 GEMMs.  A CTA (or, for N or K above 2048, a pair
// of CTAs on two SMs with tcgen05.mma.cta_group::2) computes 128 x BN (pair:
// 256 x 256) output tiles with the fp32 accumulator in tensor memory (TMEM),
// double-buffered.  Warp 0 streams the A and B tiles with TMA (128-byte
// swizzle) through a STAGES-deep mbarrier ring; warp 1 issues tcgen05.mma
// from one thread; warps 2-9 read the accumulator back with tcgen05.ld (one
// thread per output row) and apply the fused epilogue (bias, GELU-tanh, 3D
// RoPE of q/k, gated or plain residual) before storing.  Long-K pair GEMMs
// inside a block can finish their last round as split-K units (see
// splitk_plan).
//
// fp32: a register-tiled SIMT GEMM with the same epilogue (the fp32 mode's
// 1e-4 tolerance rules out tf32 tensor cores).
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace acid {

namespace {

// Epilogue parameters as passed to the kernels.
struct EpiDev {
  int kind;
  const float* bias;
  const float* gate_v;
  const float* gate_t;
  int64_t gate_split;
  const void* res;
  int64_t ldr;
  int res_fp32;
  int64_t row_base;
  RopeTable rope;
  int64_t rope_first_video;
  int d, head_dim;
};

EpiDev to_dev(const Epilogue& e) {
  EpiDev d;
  d.kind = e.kind;
  d.bias = e.bias;
  d.gate_v = e.gate_video;
  d.gate_t = e.gate_text ? e.gate_text : e.gate_video;
  d.gate_split = e.gate_split;
  d.res = e.residual;
  d.ldr = e.ldr;
  d.res_fp32 = e.res_fp32 ? 1 : 0;
  d.row_base = e.row_base;
  d.rope = e.rope;
  d.rope_first_video = e.rope_first_video;
  d.d = e.d;
  d.head_dim = e.head_dim;
  return d;
}

// Video position -> (frame, row, column) of the latent grid in 32-bit
// arithmetic.  Positions are below 2^24 (checked on the host), so the float
// quotient n * (1/d) is within one of floor(n / d) and one correction step
// makes it exact.
struct RopePos {
  int f, h, w;
};
__device__ __forceinline__ int div_small(int n, int d, float inv_d) {
  int q = (int)((float)n * inv_d);
  const int r = n - q * d;
  q += (r >= d) - (r < 0);
  return q;
}
__device__ __forceinline__ RopePos rope_pos(const RopeTable& t, int pos) {
  const int hw = t.grid_h * t.grid_w;
  RopePos p;
  p.f = div_small(pos, hw, t.inv_hw);
  const int rem = pos - p.f * hw;
  p.h = div_small(rem, t.grid_w, t.inv_w);
  p.w = rem - p.h * t.grid_w;
  return p;
}

// Table entry (cos, sin) of the RoPE angle of pair `jj` (within the head) at a
// decomposed position.
__device__ __forceinline__ const float2& rope_cs_ptr(const RopeTable& t, const RopePos& p, int jj) {
  if (jj < t.pairs_t) return t.table[p.f * t.pairs_t + jj];
  jj -= t.pairs_t;
  const int off_h = t.grid_f * t.pairs_t;
  if (jj < t.pairs_h) return t.table[off_h + p.h * t.pairs_h + jj];
  jj -= t.pairs_h;
  const int off_w = off_h + t.grid_h * t.pairs_h;
  return t.table[off_w + p.w * t.pairs_w + jj];
}
__device__ __forceinline__ float2 rope_cs(const RopeTable& t, const RopePos& p, int jj) { return rope_cs_ptr(t, p, jj); }
// (debug builds) the table entry's index lies inside the table
__device__ __forceinline__ bool rope_in_bounds(const RopeTable& t, const float2& e) {
  const int64_t n = (int64_t)t.grid_f * t.pairs_t + (int64_t)t.grid_h * t.pairs_h + (int64_t)t.grid_w * t.pairs_w;
  return ACID_IN_BOUNDS(kSiteGemmRope, &e - t.table, n);
}

// Applies the epilogue to the adjacent outputs (grow, col) and (grow, col+1).
// r0/r1: residual values (read by the caller) for the residual kinds.
template <bool kFastGelu>
__device__ __forceinline__ void epi_pair(const EpiDev& e, int64_t grow, int col, float& a, float& b, float r0,
                                         float r1) {
  if (e.bias) {
    a += e.bias[col];
    b += e.bias[col + 1];
  }
  switch (e.kind) {
    case EPI_GELU:
      a = gelu_tanh<kFastGelu>(a);
      b = gelu_tanh<kFastGelu>(b);
      break;
    case EPI_ROPE_QKV:
      if (col < 2 * e.d && grow >= e.rope_first_video) {
        const float2 cs = rope_cs(e.rope, rope_pos(e.rope, (int)(grow - e.rope_first_video)), (col % e.head_dim) >> 1);
        const float x0 = a, x1 = b;
        a = x0 * cs.x - x1 * cs.y;
        b = x0 * cs.y + x1 * cs.x;
      }
      break;
    case EPI_GATED_RES: {
      const float* g = grow < e.gate_split ? e.gate_t : e.gate_v;
      a = fmaf(g[col], a, r0);
      b = fmaf(g[col + 1], b, r1);
      break;
    }
    case EPI_RES:
      a += r0;
      b += r1;
      break;
    default:
      break;
  }
}

__host__ __device__ __forceinline__ bool epi_reads_res(int kind) { return kind == EPI_GATED_RES || kind == EPI_RES; }

// ===========================================================================
// tcgen05 GEMM (bf16 in, fp32 accumulate), persistent
//
// One CTA per SM walks output tiles (N fastest, so the CTAs running together
// share A row blocks in L2 and the weight tiles stay L2-resident).  The TMEM
// accumulator is double-buffered (2 x BN columns): the MMA warp fills buffer
// b for tile i+1 while eight epilogue warps drain buffer b^1 of tile i.
// ===========================================================================
constexpr int BM = 128, BK = 64;
constexpr int kEpiWarps = 8;
constexpr int kGemmThreads = 64 + 32 * kEpiWarps;

template <int BN>
struct TcCfg {
  static constexpr int STAGES = BN == 256 ? 4 : (BN == 128 ? 6 : 8);
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int EPI_STAGE_FLOATS = 32 * 32;  // one 32x32 chunk per epilogue warp (swizzled units)
  static constexpr int EPI_BYTES = kEpiWarps * EPI_STAGE_FLOATS * 4;
  static constexpr int SMEM = STAGES * STAGE_BYTES + EPI_BYTES + 1024 + 256;
  static constexpr uint32_t TMEM_COLS = 2 * BN;
};

struct GemmDims {
  int64_t M;
  int N, K;
  void* out;
  int64_t ldo;
  int out_fp32;
  // split-K launches of the pair kernel only: work unit = (tile, split);
  // split s covers k-blocks [s kb_split, (s + 1) kb_split) and stores its
  // raw fp32 accumulator at rows s m_pad + row of the partial buffer
  int splits = 1, kb_split = 0;
  int64_t m_pad = 0;
};

// Epilogue of 32-row x 32-column accumulator chunks held by a warp (thread =
// row after tcgen05.ld).  Each chunk is transposed through shared memory so
// that every global access of the warp covers whole row segments: lane l
// handles columns 4(l%8) .. 4(l%8)+3 of rows 4p + l/8, p = 0..7.  Residual
// values of the next chunk are loaded while the current one is processed, so
// each lane keeps up to 16 loads in flight.
// R32: the residual is fp32 (else bf16); fixed per kernel so that a bf16
// residual keeps two registers per row
template <bool R32>
struct ResChunk {
  uint32_t w[8][R32 ? 4 : 2];  // residual of this lane's 4 columns on its 8 rows (bf16 pairs or fp32)
  float bias[4], gv[4], gt[4];  // per-column bias and gates (video / text stream)
};

// Loads what the epilogue of the chunk at columns [col, col+4) needs from
// global memory: the residual (for the residual kinds) and the per-column
// bias and gates, through the read-only path for the vectors.  Called one
// chunk ahead so that the loads overlap the previous chunk's work.
template <int KIND, bool R32>
__device__ __forceinline__ void load_chunk_inputs(const GemmDims& g, const EpiDev& e, int64_t row0, int col,
                                                  ResChunk<R32>& rc) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    rc.bias[k] = e.bias ? __ldg(e.bias + col + k) : 0.f;
    rc.gv[k] = KIND == EPI_GATED_RES ? __ldg(e.gate_v + col + k) : 0.f;
    rc.gt[k] = KIND == EPI_GATED_RES ? __ldg(e.gate_t + col + k) : 0.f;
  }
  if constexpr (KIND == EPI_GATED_RES || KIND == EPI_RES) {
#pragma unroll
    for (int p = 0; p < 8; ++p) {
      const int64_t row = row0 + 4 * p + (lane >> 3);
      if (row >= g.M || !ACID_IN_BOUNDS(kSiteGemmResidual, row * e.ldr + col + 3, (g.M - 1) * e.ldr + g.N)) {
        // computed but not stored by the epilogue
#pragma unroll
        for (int q = 0; q < (R32 ? 4 : 2); ++q) rc.w[p][q] = 0u;
        continue;
      }
      if constexpr (R32) {
        const uint4 t = *reinterpret_cast<const uint4*>(static_cast<const float*>(e.res) + row * e.ldr + col);
        rc.w[p][0] = t.x; rc.w[p][1] = t.y; rc.w[p][2] = t.z; rc.w[p][3] = t.w;
      } else {
        const uint2 t = *reinterpret_cast<const uint2*>(static_cast<const __nv_bfloat16*>(e.res) + row * e.ldr + col);
        rc.w[p][0] = t.x; rc.w[p][1] = t.y;
      }
    }
  }
}

template <bool R32>
__device__ __forceinline__ float res_value(const ResChunk<R32>& rc, int p, int k) {
  if constexpr (R32) {
    return __uint_as_float(rc.w[p][k]);
  } else {
    const uint32_t w = rc.w[p][k >> 1];
    return (k & 1) ? bf16_hi(w) : bf16_lo(w);
  }
}

// GELU (tanh form) of a packed pair, with the arithmetic of gelu_tanh<true>
// done two lanes at a time: u = sqrt(2/pi) (x + 0.044715 x^3), out = h + h tanh(u)
// with h = x / 2.
__device__ __forceinline__ uint64_t gelu_x2(uint64_t x) {
  const uint64_t c3 = f2_pack(0.044715f, 0.044715f), k0 = f2_pack(0.7978845608028654f, 0.7978845608028654f);
  const uint64_t half = f2_pack(0.5f, 0.5f);
  const uint64_t u = f2_mul(k0, f2_fma(f2_mul(c3, x), f2_mul(x, x), x));
  float u0, u1;
  f2_unpack(u, u0, u1);
  const uint64_t t = f2_pack(tanh_fast(u0), tanh_fast(u1));
  const uint64_t h = f2_mul(half, x);
  return f2_fma(h, t, h);
}

// The stage of one epilogue warp: 32 rows x 32 fp32 columns, row-major, the
// eight 16-byte units of row r stored in the order u ^ (r & 7), so that both
// the row-wise writes (lane = row) and the transposed reads (8 lanes per row)
// touch every bank once per 128 bytes.
__device__ __forceinline__ float4* stage_unit(float* stage, int row, int unit) {
  return reinterpret_cast<float4*>(stage) + row * 8 + (unit ^ (row & 7));
}

// Output box of one chunk in the stage, as the tensor store reads it: 32 rows
// x 32 columns, row-major.  fp32: 128-byte rows with the 128-byte swizzle
// (16-byte unit u of row r at u ^ (r & 7)), the stage's own layout, so each
// lane overwrites in place the 16 bytes it has just read.  bf16: 64-byte rows
// with the 64-byte swizzle (unit u at u ^ ((r >> 1) & 3)); box row r lies in
// stage row r / 2, which the warp has read by the time row group r / 4 is
// written (row groups are written behind a __syncwarp).
__device__ __forceinline__ void box_store_f32(float* stage, int rr, int lane, const float* v) {
  *stage_unit(stage, rr, lane & 7) = make_float4(v[0], v[1], v[2], v[3]);
}
__device__ __forceinline__ void box_store_bf16(float* stage, int rr, int lane, const float* v) {
  const int u = (lane & 7) >> 1;
  uint8_t* p = reinterpret_cast<uint8_t*>(stage) + rr * 64 + ((u ^ ((rr >> 1) & 3)) << 4) + (lane & 1) * 8;
  *reinterpret_cast<uint2*>(p) = make_uint2(pack_bf16(v[0], v[1]), pack_bf16(v[2], v[3]));
}

// Output stores of the epilogue: kinds without a residual write each chunk's
// results back into the stage as the output box and hand it to one tensor
// store (the TMA engine then writes the 2-4 KB box; rows past M and columns
// past N are clipped by the tensor map).  The residual kinds keep a residual
// prefetch of two chunks in registers and store directly from registers
// (coalesced 8-16-byte stores per lane), which leaves them without spills at
// the 168-register limit of ten warps.
template <int KIND>
constexpr bool kTmaStore = !(KIND == EPI_GATED_RES || KIND == EPI_RES);

// Epilogue of one 32-row x 32-column chunk held by a warp (thread = row, as
// tcgen05.ld delivers it).  The chunk is transposed through the stage so that
// each lane handles four columns of eight rows, then stored as above.  With
// tensor stores the caller waits for the previous store to have read the
// stage before calling again.
template <int KIND, bool R32, bool O32>
__device__ __forceinline__ void epilogue_chunk(const GemmDims& g, const EpiDev& e, const CUtensorMap* tmO,
                                               float* stage, int64_t row0, int col0, const uint32_t* r,
                                               const ResChunk<R32>& rc) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int u = 0; u < 8; ++u)
    *stage_unit(stage, lane, u) = make_float4(__uint_as_float(r[4 * u]), __uint_as_float(r[4 * u + 1]),
                                              __uint_as_float(r[4 * u + 2]), __uint_as_float(r[4 * u + 3]));
  __syncwarp();
  const int c = 4 * (lane & 7);
  const int col = col0 + c;
  // RoPE: the (cos, sin) of this lane's two pairs on its eight rows, all
  // loaded through the read-only path before the row groups are processed
  float2 rcs[KIND == EPI_ROPE_QKV ? 8 : 1][2];
  if constexpr (KIND == EPI_ROPE_QKV) {
    const int j0 = (col & (e.head_dim - 1)) >> 1;
#pragma unroll
    for (int p = 0; p < 8; ++p) {
      const int64_t grow = row0 + 4 * p + (lane >> 3) + e.row_base;
      rcs[p][0] = rcs[p][1] = make_float2(1.f, 0.f);
      if (col < 2 * e.d && grow >= e.rope_first_video && row0 + 4 * p + (lane >> 3) < g.M) {
        const RopePos pp = rope_pos(e.rope, (int)(grow - e.rope_first_video));
#pragma unroll
        for (int q = 0; q < 2; ++q)
          if (rope_in_bounds(e.rope, rope_cs_ptr(e.rope, pp, j0 + q))) rcs[p][q] = __ldg(&rope_cs_ptr(e.rope, pp, j0 + q));
      }
    }
  }
  const uint64_t b01 = f2_pack(rc.bias[0], rc.bias[1]), b23 = f2_pack(rc.bias[2], rc.bias[3]);
  // rows past M are computed like the others (from whatever the stage and
  // residual registers hold); the tensor store clips them
#pragma unroll
  for (int p = 0; p < 8; ++p) {
    const int rr = 4 * p + (lane >> 3);
    const int64_t grow = row0 + rr + e.row_base;
    const float4 sv = *stage_unit(stage, rr, lane & 7);
    uint64_t v01 = f2_add(f2_pack(sv.x, sv.y), b01), v23 = f2_add(f2_pack(sv.z, sv.w), b23);
    switch (KIND) {
      case EPI_GELU:
        v01 = gelu_x2(v01);
        v23 = gelu_x2(v23);
        break;
      case EPI_ROPE_QKV: {
        // (cos, sin) = (1, 0) on rows and columns that are not rotated; the
        // four columns lie in one head (head_dim is a power of two)
        float v[4];
        f2_unpack(v01, v[0], v[1]);
        f2_unpack(v23, v[2], v[3]);
#pragma unroll
        for (int k = 0; k < 4; k += 2) {
          const float2 cs = rcs[p][k >> 1];
          const float x0 = v[k], x1 = v[k + 1];
          v[k] = x0 * cs.x - x1 * cs.y;
          v[k + 1] = x0 * cs.y + x1 * cs.x;
        }
        v01 = f2_pack(v[0], v[1]);
        v23 = f2_pack(v[2], v[3]);
        break;
      }
      case EPI_GATED_RES: {
        const bool text = grow < e.gate_split;
        const uint64_t g01 = text ? f2_pack(rc.gt[0], rc.gt[1]) : f2_pack(rc.gv[0], rc.gv[1]);
        const uint64_t g23 = text ? f2_pack(rc.gt[2], rc.gt[3]) : f2_pack(rc.gv[2], rc.gv[3]);
        v01 = f2_fma(g01, v01, f2_pack(res_value(rc, p, 0), res_value(rc, p, 1)));
        v23 = f2_fma(g23, v23, f2_pack(res_value(rc, p, 2), res_value(rc, p, 3)));
        break;
      }
      case EPI_RES:
        v01 = f2_add(v01, f2_pack(res_value(rc, p, 0), res_value(rc, p, 1)));
        v23 = f2_add(v23, f2_pack(res_value(rc, p, 2), res_value(rc, p, 3)));
        break;
      default:
        break;
    }
    float v[4];
    f2_unpack(v01, v[0], v[1]);
    f2_unpack(v23, v[2], v[3]);
    if constexpr (kTmaStore<KIND>) {
      if constexpr (O32) {
        box_store_f32(stage, rr, lane, v);  // in place: this lane's own 16 bytes
      } else {
        __syncwarp();  // the stage row this box row overwrites has been read by every lane
        box_store_bf16(stage, rr, lane, v);
      }
    } else {
      const int64_t row = row0 + rr;
      if (row >= g.M || !ACID_IN_BOUNDS(kSiteGemmStore, row * g.ldo + col + 3, (g.M - 1) * g.ldo + g.N)) continue;
      if constexpr (O32)
        *reinterpret_cast<float4*>(static_cast<float*>(g.out) + row * g.ldo + col) = make_float4(v[0], v[1], v[2], v[3]);
      else
        *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(g.out) + row * g.ldo + col) =
            make_uint2(pack_bf16(v[0], v[1]), pack_bf16(v[2], v[3]));
    }
  }
  if constexpr (kTmaStore<KIND>) {
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      tma_store_2d(tmO, stage, col0, (int)row0);
      bulk_commit_group();
    }
  } else {
    __syncwarp();  // every lane has read the stage before the next chunk overwrites it
  }
}

// Bias of a chunk's 32 columns, the same for every lane (broadcast loads
// through the read-only path; 16-byte loads where the vector is aligned).
__device__ __forceinline__ void load_bias32(const EpiDev& e, int col0, float* bias) {
  if (e.bias == nullptr) {
#pragma unroll
    for (int k = 0; k < 32; ++k) bias[k] = 0.f;
  } else if ((reinterpret_cast<uintptr_t>(e.bias + col0) & 15) == 0) {
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float4 t = __ldg(reinterpret_cast<const float4*>(e.bias + col0) + k);
      bias[4 * k] = t.x; bias[4 * k + 1] = t.y; bias[4 * k + 2] = t.z; bias[4 * k + 3] = t.w;
    }
  } else {
#pragma unroll
    for (int k = 0; k < 32; ++k) bias[k] = __ldg(e.bias + col0 + k);
  }
}

// Epilogue of one 32-row x 32-column chunk of a kind without a residual, in
// the layout tcgen05.ld delivers (thread = row, 32 consecutive columns): the
// bias and the kind's arithmetic in registers, then the output box written
// once into the warp's stage in the tensor store's swizzled layout (fp32:
// 128-byte rows, 16-byte unit u of row r at u ^ (r & 7); bf16: 64-byte rows,
// unit u at u ^ ((r >> 1) & 3); both place the 32 rows' units of a given u in
// distinct bank groups) and handed to one TMA store, which clips rows past M.
// Shared-memory traffic is one write and one TMA read of the box.  The caller
// makes sure the store that last read this stage has finished reading.
template <int KIND, bool O32>
__device__ __forceinline__ void epilogue_rows(const GemmDims& g, const EpiDev& e, const CUtensorMap* tmO,
                                              uint8_t* stage, int64_t row0, int64_t store_row0, int col0,
                                              const uint32_t* r, const float* bias) {
  const int lane = threadIdx.x & 31;
  uint64_t v[16];
#pragma unroll
  for (int k = 0; k < 16; ++k)
    v[k] = f2_add(f2_pack(__uint_as_float(r[2 * k]), __uint_as_float(r[2 * k + 1])),
                  f2_pack(bias[2 * k], bias[2 * k + 1]));
  if constexpr (KIND == EPI_GELU) {
#pragma unroll
    for (int k = 0; k < 16; ++k) v[k] = gelu_x2(v[k]);
  } else if constexpr (KIND == EPI_ROPE_QKV) {
    // the chunk's 16 pairs lie in one head (head_dim is a power of two >= 32)
    const int64_t row = row0 + lane, grow = row + e.row_base;
    if (col0 < 2 * e.d && grow >= e.rope_first_video && row < g.M) {
      const RopePos pp = rope_pos(e.rope, (int)(grow - e.rope_first_video));
      const int j0 = (col0 & (e.head_dim - 1)) >> 1;
#pragma unroll
      for (int k = 0; k < 16; ++k) {
        const float2& ce = rope_cs_ptr(e.rope, pp, j0 + k);
        const float2 cs = rope_in_bounds(e.rope, ce) ? __ldg(&ce) : make_float2(1.f, 0.f);
        float x0, x1;
        f2_unpack(v[k], x0, x1);
        v[k] = f2_pack(x0 * cs.x - x1 * cs.y, x0 * cs.y + x1 * cs.x);
      }
    }
  }
  if constexpr (O32) {
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      float a0, a1, a2, a3;
      f2_unpack(v[2 * u], a0, a1);
      f2_unpack(v[2 * u + 1], a2, a3);
      *reinterpret_cast<float4*>(stage + lane * 128 + ((u ^ (lane & 7)) << 4)) = make_float4(a0, a1, a2, a3);
    }
  } else {
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      uint32_t w[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        float a0, a1;
        f2_unpack(v[4 * u + q], a0, a1);
        w[q] = pack_bf16(a0, a1);
      }
      *reinterpret_cast<uint4*>(stage + lane * 64 + ((u ^ ((lane >> 1) & 3)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
    }
  }
  fence_proxy_async_smem();
  __syncwarp();
  if (lane == 0) {
    tma_store_2d(tmO, stage, col0, (int)store_row0);
    bulk_commit_group();
  }
}

// One chunk of a kind without a residual: accumulator and bias loads, the
// stage (bf16 output: two 2 KB stages per warp used in turn, so a chunk waits
// only for the store before last; fp32 output: one 4 KB stage), epilogue_rows.
template <int KIND, bool O32>
__device__ __forceinline__ void tma_kind_chunk(const GemmDims& g, const EpiDev& e, const CUtensorMap* tmO,
                                               uint8_t* stage, uint32_t taddr, int64_t row0, int64_t store_row0,
                                               int col0, bool ok, int& nstore) {
  const int lane = threadIdx.x & 31;
  uint32_t r[32];
  float bias[32];
  tmem_ld32(taddr, r);
  const bool live = ok && row0 < g.M && col0 < g.N;
  if (live) load_bias32(e, col0, bias);
  tmem_wait_ld();
  if (!live) return;
  uint8_t* st = stage;
  if constexpr (O32) {
    if (lane == 0) bulk_wait_group_read<0>();
  } else {
    st += (nstore & 1) * 2048;
    if (lane == 0) bulk_wait_group_read<1>();
  }
  __syncwarp();
  epilogue_rows<KIND, O32>(g, e, tmO, st, row0, store_row0, col0, r, bias);
  ++nstore;
}

template <int BN, int KIND, bool R32, bool O32>
__global__ void __launch_bounds__(kGemmThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmO, GemmDims g, EpiDev e) {
  using C = TcCfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::STAGES * C::STAGE_BYTES + C::EPI_BYTES);
  uint64_t* empty = full + C::STAGES;
  uint64_t* acc_full = empty + C::STAGES;  // [2]
  uint64_t* acc_empty = acc_full + 2;      // [2]
  uint64_t* drain = acc_empty + 2;         // failure path: the MMAs issued so far have completed
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int num_kb = (g.K + BK - 1) / BK;
  const int num_n = (g.N + BN - 1) / BN;
  const int num_tiles = (int)((g.M + BM - 1) / BM) * num_n;

  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 32 * kEpiWarps);
    }
    mbar_init(drain, 1);
    mbar_fence_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {  // TMA producer: one continuous stage ring across tiles
      int it = 0;
      bool ok = true;
      for (int tile = blockIdx.x; ok && tile < num_tiles; tile += gridDim.x) {
        const int m_tile = tile / num_n, n_tile = tile % num_n;
        for (int kb = 0; kb < num_kb; ++kb, ++it) {
          const int s = it % C::STAGES, round = it / C::STAGES;
          if (round > 0 && !mbar_wait(&empty[s], (round - 1) & 1)) { ok = false; break; }
          mbar_expect_tx(&full[s], C::STAGE_BYTES);
          tma_load_2d(sA + s * C::A_BYTES, &tmA, &full[s], kb * BK, m_tile * BM);
          tma_load_2d(sB + s * C::B_BYTES, &tmB, &full[s], kb * BK, n_tile * BN);
        }
      }
      // After a wait ran out: the loads of the last STAGES issues may still be
      // in flight; wait (bounded) until they have landed, so that no TMA
      // writes into this CTA's shared memory after it exits.  Earlier issues
      // were consumed by the MMA thread before their stage was refilled.
      if (!ok)
        for (int j = std::max(0, it - C::STAGES); j < it; ++j) mbar_wait(&full[j % C::STAGES], (j / C::STAGES) & 1);
    }
  } else if (warp == 1) {
    if (lane == 0) {  // MMA issuer
      constexpr uint32_t idesc = idesc_bf16_f32(BM, BN, false, false);
      int it = 0, local = 0;
      bool ok = true;
      for (int tile = blockIdx.x; ok && tile < num_tiles; tile += gridDim.x, ++local) {
        const int b = local & 1, use = local >> 1;
        if (use > 0 && !mbar_wait(&acc_empty[b], (use - 1) & 1)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d = tmem + b * BN;
        for (int kb = 0; kb < num_kb; ++kb, ++it) {
          const int s = it % C::STAGES, round = it / C::STAGES;
          if (!mbar_wait(&full[s], round & 1)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + s * C::A_BYTES);
          const uint32_t b0 = smem_u32(sB + s * C::B_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            const uint64_t ad = smem_desc_sw128(a0 + k * 32, 16, 1024);
            const uint64_t bd = smem_desc_sw128(b0 + k * 32, 16, 1024);
            mma_bf16_ss(d, ad, bd, idesc, (kb | k) != 0);
          }
          mma_commit(&empty[s]);
        }
        if (ok) mma_commit(&acc_full[b]);
      }
      // After a wait ran out: let the MMAs already issued finish (bounded)
      // before the accumulator's tensor memory is freed below.
      if (!ok) {
        mma_commit(drain);
        mbar_wait(drain, 0);
      }
    }
  } else {  // epilogue: warps 2..9; lane quarter = warp % 4, column half = (warp - 2) / 4
    const int q = warp & 3, half = (warp - 2) >> 2;
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    float* stage = reinterpret_cast<float*>(smem + C::STAGES * C::STAGE_BYTES) + (warp - 2) * C::EPI_STAGE_FLOATS;
    int local = 0;
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x, ++local) {
      const int b = local & 1, use = local >> 1;
      const int m_tile = tile / num_n, n_tile = tile % num_n;
      const bool ok = mbar_wait(&acc_full[b], use & 1);
      tc_fence_after();
      const int64_t row0 = (int64_t)m_tile * BM + q * 32;
      // this warp's chunks: columns [half * BN/2, (half + 1) * BN/2) of the tile, 32 at a time;
      // the global inputs of chunk i+1 (residual, bias, gates) are loaded while chunk i is processed
      constexpr int NC = BN / 64;
      const int cbeg = half * (BN / 2);
      const int lcol = 4 * (lane & 7);
      auto process = [&](int i, const ResChunk<R32>& cur, ResChunk<R32>& nxt) {
        const int c = cbeg + 32 * i;
        uint32_t r[32];
        tmem_ld32(tmem + lane_base + b * BN + c, r);
        tmem_wait_ld();
        const int col0 = n_tile * BN + c;
        if (i + 1 < NC && row0 < g.M && col0 + 32 < g.N) load_chunk_inputs<KIND, R32>(g, e, row0, col0 + 32 + lcol, nxt);
        if (ok && row0 < g.M && col0 < g.N) {
          if constexpr (kTmaStore<KIND>) {
            if (lane == 0) bulk_wait_group_read<0>();  // the previous box has left the stage
            __syncwarp();
          }
          epilogue_chunk<KIND, R32, O32>(g, e, &tmO, stage, row0, col0, r, cur);
        }
      };
      ResChunk<R32> rc0, rc1;
      if (row0 < g.M && n_tile * BN + cbeg < g.N) load_chunk_inputs<KIND, R32>(g, e, row0, n_tile * BN + cbeg + lcol, rc0);
#pragma unroll 1
      for (int i = 0; i < NC; i += 2) {
        process(i, rc0, rc1);
        if (i + 1 < NC) process(i + 1, rc1, rc0);
      }
      tc_fence_before();
      mbar_arrive(&acc_empty[b]);
      if (!ok) break;
    }
    if (lane == 0) bulk_wait_group<0>();  // tensor stores complete before the CTA exits
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// ===========================================================================
// tcgen05 GEMM on SM pairs (cta_group::2), persistent
//
// A cluster of two CTAs on two SMs computes 256 x 256 output tiles: each CTA
// stages its own 128 rows of A and its own 128 rows of B (half of the tile's
// output columns) per 64-wide k-step, and one thread of CTA rank 0 issues
// M256 N256 K16 MMAs that read both CTAs' shared memory and write each CTA's
// 128 x 256 fp32 accumulator into that CTA's TMEM.  Per SM and k-step this
// moves 32 KB into shared memory for 128 x 256 x 64 MACs, against 48 KB for
// the single-SM 128 x 256 tile: the single-SM kernel is bound by that
// L2-to-SM delivery.
//   warp 0   TMA producer in both CTAs; both CTAs' loads count on rank 0's
//            full[s] barrier (rank 0 expects the bytes of both);
//   warp 1   rank 0: MMA issuer; each k-step is committed to empty[s] of both
//            CTAs, each tile to acc_full[b] of both CTAs;
//   warps 2-9 epilogue of this CTA's 128 accumulator rows (as in
//            gemm_tc_kernel); one lane per warp then arrives on rank 0's
//            acc_empty[b], which counts the epilogue warps of both CTAs.
// ===========================================================================
struct Tc2Cfg {
  static constexpr int BN = 256;  // output columns per pair tile
  static constexpr int STAGES = 6;
  static constexpr int A_BYTES = BM * BK * 2;        // this CTA's 128 rows of A
  static constexpr int B_BYTES = (BN / 2) * BK * 2;  // this CTA's 128 rows of B
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int EPI_STAGE_FLOATS = 32 * 32;
  static constexpr int EPI_BYTES = kEpiWarps * EPI_STAGE_FLOATS * 4;
  static constexpr int SMEM = STAGES * STAGE_BYTES + EPI_BYTES + 1024 + 256;
  static constexpr uint32_t TMEM_COLS = 2 * BN;  // double-buffered 128 x 256 accumulator
};
static_assert(Tc2Cfg::SMEM <= 232448, "pair GEMM shared memory");

template <int KIND, bool R32, bool O32, bool SPLIT = false>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kGemmThreads, 1)
    gemm_tc2_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const __grid_constant__ CUtensorMap tmO, GemmDims g, EpiDev e) {
  using C = Tc2Cfg;
  constexpr int BN = C::BN;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::STAGES * C::STAGE_BYTES + C::EPI_BYTES);
  uint64_t* empty = full + C::STAGES;
  uint64_t* acc_full = empty + C::STAGES;  // [2]
  uint64_t* acc_empty = acc_full + 2;      // [2] (rank 0's counts both CTAs' epilogue warps)
  uint64_t* drain = acc_empty + 2;         // failure path: the MMAs issued so far have completed
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const int pair = (int)blockIdx.x >> 1, npairs = (int)gridDim.x >> 1;
  const int num_kb = SPLIT ? g.kb_split : (g.K + BK - 1) / BK;
  const int num_n = (g.N + BN - 1) / BN;
  const int num_tiles = (int)((g.M + 2 * BM - 1) / (2 * BM)) * num_n;
  const int num_units = SPLIT ? num_tiles * g.splits : num_tiles;  // (tile, split) pairs

  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 2 * kEpiWarps);
    }
    mbar_init(drain, 1);
    mbar_fence_init();
  }
  if (warp == 1) tmem_alloc_pair(tmem_slot, C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // both CTAs' barriers exist before any cross-CTA arrival
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {  // TMA producer (both CTAs): one continuous stage ring across tiles
      const uint32_t full0 = mapa_shared(smem_u32(full), 0);  // rank 0's full[0]
      int it = 0;
      bool ok = true;
      for (int unit = pair; ok && unit < num_units; unit += npairs) {
        const int tile = SPLIT ? unit / g.splits : unit;
        const int kb0 = SPLIT ? (unit % g.splits) * num_kb : 0;
        const int m_tile = tile / num_n, n_tile = tile % num_n;
        for (int kb = 0; kb < num_kb; ++kb, ++it) {
          const int s = it % C::STAGES, round = it / C::STAGES;
          if (round > 0 && !mbar_wait(&empty[s], (round - 1) & 1)) { ok = false; break; }
          if (rank == 0) mbar_expect_tx(&full[s], 2 * C::STAGE_BYTES);
          tma_load_2d_pair(sA + s * C::A_BYTES, &tmA, full0 + 8 * s, (kb0 + kb) * BK, m_tile * 2 * BM + (int)rank * BM);
          tma_load_2d_pair(sB + s * C::B_BYTES, &tmB, full0 + 8 * s, (kb0 + kb) * BK,
                           n_tile * BN + (int)rank * (BN / 2));
        }
      }
      // After a wait ran out: rank 0 waits (bounded) for the last STAGES
      // stages it expected to land.  Rank 1's loads count on rank 0's
      // barriers, which rank 1 cannot poll; it idles about 2^16 clocks, far
      // above the latency of a 32 KB load, before both CTAs meet at the exit.
      if (!ok) {
        if (rank == 0) {
          for (int j = std::max(0, it - C::STAGES); j < it; ++j) mbar_wait(&full[j % C::STAGES], (j / C::STAGES) & 1);
        } else {
          const long long t0 = clock64();
          while (clock64() - t0 < (1LL << 16)) {
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {  // MMA issuer (rank 0 only)
      constexpr uint32_t idesc = idesc_bf16_f32(2 * BM, BN, false, false);
      const uint32_t empty_l = smem_u32(empty), empty_r = mapa_shared(empty_l, 1);
      const uint32_t accf_l = smem_u32(acc_full), accf_r = mapa_shared(accf_l, 1);
      int it = 0, local = 0;
      bool ok = true;
      for (int unit = pair; ok && unit < num_units; unit += npairs, ++local) {
        const int b = local & 1, use = local >> 1;
        if (use > 0 && !mbar_wait_cluster(&acc_empty[b], (use - 1) & 1)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d = tmem + b * BN;
        for (int kb = 0; kb < num_kb; ++kb, ++it) {
          const int s = it % C::STAGES, round = it / C::STAGES;
          if (!mbar_wait(&full[s], round & 1)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + s * C::A_BYTES);
          const uint32_t b0 = smem_u32(sB + s * C::B_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            const uint64_t ad = smem_desc_sw128(a0 + k * 32, 16, 1024);
            const uint64_t bd = smem_desc_sw128(b0 + k * 32, 16, 1024);
            mma_bf16_ss_pair(d, ad, bd, idesc, (kb | k) != 0);
          }
          mma_commit_pair(empty_l + 8 * s);
          mma_commit_pair(empty_r + 8 * s);
        }
        if (ok) {
          mma_commit_pair(accf_l + 8 * b);
          mma_commit_pair(accf_r + 8 * b);
        }
      }
      if (!ok) {
        mma_commit_pair(smem_u32(drain));
        mbar_wait(drain, 0);
      }
    }
  } else {  // epilogue: warps 2..9 of each CTA, this CTA's 128 rows of the pair tile
    const int q = warp & 3, half = (warp - 2) >> 2;
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    float* stage = reinterpret_cast<float*>(smem + C::STAGES * C::STAGE_BYTES) + (warp - 2) * C::EPI_STAGE_FLOATS;
    const uint32_t acc_empty0 = mapa_shared(smem_u32(acc_empty), 0);
    int local = 0, nstore = 0;
    for (int unit = pair; unit < num_units; unit += npairs, ++local) {
      const int tile = SPLIT ? unit / g.splits : unit;
      const int b = local & 1, use = local >> 1;
      const int m_tile = tile / num_n, n_tile = tile % num_n;
      const bool ok = mbar_wait(&acc_full[b], use & 1);
      tc_fence_after();
      const int64_t row0 = (int64_t)m_tile * 2 * BM + (int64_t)rank * BM + q * 32;
      if constexpr (kTmaStore<KIND>) {
        constexpr int NC = BN / 64;
        const int cbeg = half * (BN / 2);
        const int64_t store_row0 = SPLIT ? row0 + (int64_t)(unit % g.splits) * g.m_pad : row0;
#pragma unroll 1
        for (int i = 0; i < NC; ++i)
          tma_kind_chunk<KIND, O32>(g, e, &tmO, reinterpret_cast<uint8_t*>(stage),
                                    tmem + lane_base + b * BN + cbeg + 32 * i, row0, store_row0,
                                    n_tile * BN + cbeg + 32 * i, ok, nstore);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(acc_empty0 + 8 * b);
        if (!ok) break;
        continue;
      }
      constexpr int NC = BN / 64;
      const int cbeg = half * (BN / 2);
      const int lcol = 4 * (lane & 7);
      auto process = [&](int i, const ResChunk<R32>& cur, ResChunk<R32>& nxt) {
        const int c = cbeg + 32 * i;
        uint32_t r[32];
        tmem_ld32(tmem + lane_base + b * BN + c, r);
        tmem_wait_ld();
        const int col0 = n_tile * BN + c;
        if (i + 1 < NC && row0 < g.M && col0 + 32 < g.N) load_chunk_inputs<KIND, R32>(g, e, row0, col0 + 32 + lcol, nxt);
        if (ok && row0 < g.M && col0 < g.N) {
          if constexpr (kTmaStore<KIND>) {
            if (lane == 0) bulk_wait_group_read<0>();  // the previous box has left the stage
            __syncwarp();
          }
          epilogue_chunk<KIND, R32, O32>(g, e, &tmO, stage, row0, col0, r, cur);
        }
      };
      ResChunk<R32> rc0, rc1;
      if (row0 < g.M && n_tile * BN + cbeg < g.N) load_chunk_inputs<KIND, R32>(g, e, row0, n_tile * BN + cbeg + lcol, rc0);
#pragma unroll 1
      for (int i = 0; i < NC; i += 2) {
        process(i, rc0, rc1);
        if (i + 1 < NC) process(i + 1, rc1, rc0);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(acc_empty0 + 8 * b);
      if (!ok) break;
    }
    if (lane == 0) bulk_wait_group<0>();  // tensor stores complete before the CTA exits
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // no CTA leaves while its peer may still signal its barriers
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, C::TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------
// TMA descriptor encoding through the driver entry point (no -lcuda needed)
// ---------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

}  // namespace

// Row-major matrix [rows, cols] of 2-byte (bf16) or 4-byte (fp32) elements
// with row stride ld (elements), boxes of box_rows x box_cols, the given
// swizzle, zero fill out of bounds (loads) and clipping (stores).
acid_status make_tmap_2d(CUtensorMap* map, CUtensorMapDataType type, int esize, const void* base, int64_t rows,
                         int64_t cols, int64_t ld, int box_cols, int box_rows, CUtensorMapSwizzle swizzle) {
  auto fn = encode_fn();
  ACID_REQUIRE(fn != nullptr, ACID_ERR_CUDA, "cuTensorMapEncodeTiled entry point unavailable");
  ACID_REQUIRE(aligned(base, 16) && (ld * esize) % 16 == 0, ACID_ERR_UNSUPPORTED,
               "TMA operand must be 16-byte aligned with a row stride that is a multiple of 16 bytes");
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)(ld * esize)};
  cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1u, 1u};
  CUresult r = fn(map, type, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  ACID_REQUIRE(r == CUDA_SUCCESS, ACID_ERR_CUDA, "cuTensorMapEncodeTiled failed (code " + std::to_string((int)r) + ")");
  return ACID_OK;
}

acid_status make_tmap_bf16_box(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int64_t ld,
                               int box_cols, int box_rows, CUtensorMapSwizzle swizzle) {
  return make_tmap_2d(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, rows, cols, ld, box_cols, box_rows, swizzle);
}

// Boxes of box_rows x 64 columns with 128-byte swizzle (the MMA operand layout).
acid_status make_tmap_bf16(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int64_t ld, int box_rows) {
  return make_tmap_bf16_box(map, base, rows, cols, ld, 64, box_rows, CU_TENSOR_MAP_SWIZZLE_128B);
}

namespace {

// The GEMM output as the epilogue's tensor stores see it: 32 x 32 boxes, the
// swizzle of the box layout in epilogue_chunk (128-byte rows for fp32,
// 64-byte rows for bf16).
acid_status make_tmap_out(CUtensorMap* map, void* out, int64_t M, int N, int64_t ldo, bool fp32) {
  return fp32 ? make_tmap_2d(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, out, M, N, ldo, 32, 32, CU_TENSOR_MAP_SWIZZLE_128B)
              : make_tmap_2d(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, out, M, N, ldo, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B);
}

int num_sms() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
  }
  return n;
}

template <int BN, int KIND, bool R32, bool O32>
acid_status launch_tc_kind1(const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap& to, const GemmDims& g,
                           const Epilogue& epi, int grid, cudaStream_t s) {
  using C = TcCfg<BN>;
  static bool attr_done = false;
  if (!attr_done) {
    ACID_CUDA(cudaFuncSetAttribute(gemm_tc_kernel<BN, KIND, R32, O32>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM));
    attr_done = true;
  }
  gemm_tc_kernel<BN, KIND, R32, O32><<<grid, kGemmThreads, C::SMEM, s>>>(ta, tb, to, g, to_dev(epi));
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

// dispatch on the output dtype (a template parameter: it selects the box layout)
template <int BN, int KIND, bool R32 = false>
acid_status launch_tc_kind(const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap& to, const GemmDims& g,
                           const Epilogue& epi, int grid, cudaStream_t s) {
  return g.out_fp32 ? launch_tc_kind1<BN, KIND, R32, true>(ta, tb, to, g, epi, grid, s)
                    : launch_tc_kind1<BN, KIND, R32, false>(ta, tb, to, g, epi, grid, s);
}

template <int BN>
acid_status launch_tc(const void* A, int64_t lda, int64_t M, int K, const void* W, int N, void* out, int64_t ldo,
                      const Epilogue& epi, cudaStream_t s) {
  CUtensorMap ta, tb, to;
  ACID_TRY(make_tmap_bf16(&ta, A, M, K, lda, BM));
  ACID_TRY(make_tmap_bf16(&tb, W, N, K, K, BN));
  ACID_TRY(make_tmap_out(&to, out, M, N, ldo, epi.out_fp32));
  GemmDims g{M, N, K, out, ldo, epi.out_fp32 ? 1 : 0};
  const int64_t tiles = ((M + BM - 1) / BM) * ((N + BN - 1) / BN);
  const int grid = (int)std::min<int64_t>(tiles, num_sms());
  ProfScope prof(PROF_LINEAR, 2.0 * (double)M * N * K, s);
  switch (epi.kind) {
    case EPI_GELU: return launch_tc_kind<BN, EPI_GELU>(ta, tb, to, g, epi, grid, s);
    case EPI_ROPE_QKV: return launch_tc_kind<BN, EPI_ROPE_QKV>(ta, tb, to, g, epi, grid, s);
    case EPI_GATED_RES:
      return epi.res_fp32 ? launch_tc_kind<BN, EPI_GATED_RES, true>(ta, tb, to, g, epi, grid, s)
                          : launch_tc_kind<BN, EPI_GATED_RES, false>(ta, tb, to, g, epi, grid, s);
    case EPI_RES:
      return epi.res_fp32 ? launch_tc_kind<BN, EPI_RES, true>(ta, tb, to, g, epi, grid, s)
                          : launch_tc_kind<BN, EPI_RES, false>(ta, tb, to, g, epi, grid, s);
    default: return launch_tc_kind<BN, EPI_BIAS>(ta, tb, to, g, epi, grid, s);
  }
}

// CTA pairs that can be resident at once for the pair kernel (clusters are
// placed within a GPC, so this can be below half the SM count).
template <int KIND, bool R32, bool O32>
int max_pairs() {
  static int n = -1;
  if (n < 0) {
    // the dynamic shared memory limit must be raised before the query
    if (cudaFuncSetAttribute(gemm_tc2_kernel<KIND, R32, O32>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             Tc2Cfg::SMEM) != cudaSuccess)
      return 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2 * 76, 1, 1);
    cfg.blockDim = dim3(kGemmThreads, 1, 1);
    cfg.dynamicSmemBytes = Tc2Cfg::SMEM;
    int c = 0;
    n = (cudaOccupancyMaxActiveClusters(&c, gemm_tc2_kernel<KIND, R32, O32>, &cfg) == cudaSuccess && c > 0) ? c : 0;
  }
  return n;
}

template <int KIND, bool R32, bool O32>
acid_status launch_tc2_kind1(const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap& to, const GemmDims& g,
                            const Epilogue& epi, int64_t tiles, cudaStream_t s) {
  static bool attr_done = false;
  if (!attr_done) {
    ACID_CUDA(cudaFuncSetAttribute(gemm_tc2_kernel<KIND, R32, O32>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   Tc2Cfg::SMEM));
    attr_done = true;
  }
  const int pairs = max_pairs<KIND, R32, O32>();
  ACID_REQUIRE(pairs > 0, ACID_ERR_CUDA, "linear: no resident CTA pair for the pair GEMM");
  const int grid = 2 * (int)std::min<int64_t>(tiles, pairs);
  gemm_tc2_kernel<KIND, R32, O32><<<grid, kGemmThreads, Tc2Cfg::SMEM, s>>>(ta, tb, to, g, to_dev(epi));
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

template <int KIND, bool R32 = false>
acid_status launch_tc2_kind(const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap& to, const GemmDims& g,
                            const Epilogue& epi, int64_t tiles, cudaStream_t s) {
  return g.out_fp32 ? launch_tc2_kind1<KIND, R32, true>(ta, tb, to, g, epi, tiles, s)
                    : launch_tc2_kind1<KIND, R32, false>(ta, tb, to, g, epi, tiles, s);
}

acid_status launch_tc2(const void* A, int64_t lda, int64_t M, int K, const void* W, int N, void* out, int64_t ldo,
                       const Epilogue& epi, cudaStream_t s) {
  CUtensorMap ta, tb, to;
  ACID_TRY(make_tmap_bf16(&ta, A, M, K, lda, BM));
  ACID_TRY(make_tmap_bf16(&tb, W, N, K, K, Tc2Cfg::BN / 2));
  ACID_TRY(make_tmap_out(&to, out, M, N, ldo, epi.out_fp32));
  GemmDims g{M, N, K, out, ldo, epi.out_fp32 ? 1 : 0};
  const int64_t tiles = ((M + 2 * BM - 1) / (2 * BM)) * ((N + Tc2Cfg::BN - 1) / Tc2Cfg::BN);
  ProfScope prof(PROF_LINEAR, 2.0 * (double)M * N * K, s);
  switch (epi.kind) {
    case EPI_GELU: return launch_tc2_kind<EPI_GELU>(ta, tb, to, g, epi, tiles, s);
    case EPI_ROPE_QKV: return launch_tc2_kind<EPI_ROPE_QKV>(ta, tb, to, g, epi, tiles, s);
    case EPI_GATED_RES:
      return epi.res_fp32 ? launch_tc2_kind<EPI_GATED_RES, true>(ta, tb, to, g, epi, tiles, s)
                          : launch_tc2_kind<EPI_GATED_RES, false>(ta, tb, to, g, epi, tiles, s);
    case EPI_RES:
      return epi.res_fp32 ? launch_tc2_kind<EPI_RES, true>(ta, tb, to, g, epi, tiles, s)
                          : launch_tc2_kind<EPI_RES, false>(ta, tb, to, g, epi, tiles, s);
    default: return launch_tc2_kind<EPI_BIAS>(ta, tb, to, g, epi, tiles, s);
  }
}

// ---------------------------------------------------------------------------
// Split-K last round of the pair GEMM.  With K long, a persistent launch
// whose last round keeps only a few CTA pairs busy spends a whole tile's
// mainloop on it.  The rows that fill whole rounds then run as usual, and
// the remaining rows run as (tile, k-split) units, one per pair, each storing
// its raw fp32 accumulator into scratch; splitk_fixup_kernel adds a row's
// partials in split order and applies the epilogue.
struct SplitKPlan {
  int64_t rows_main = 0;  // rows of the ordinary launch (whole 256-row tiles)
  int splits = 0, kb_split = 0;
  int64_t m_pad = 0;      // tail rows rounded up to 256 (per-split stride of the scratch)
};

bool splitk_plan(int64_t M, int N, int K, size_t ws_bytes, int pairs, SplitKPlan* p) {
  constexpr int64_t bm = 2 * BM;
  const int64_t n_tiles = (N + Tc2Cfg::BN - 1) / Tc2Cfg::BN, m_tiles = (M + bm - 1) / bm;
  const int64_t tiles = m_tiles * n_tiles, num_kb = (K + BK - 1) / BK;
  if (pairs <= 0 || num_kb < 64) return false;  // short mainloops: the last round is cheap
  const int64_t full = tiles / pairs, last = tiles - full * pairs;
  if (full < 1 || last == 0 || 2 * last >= pairs) return false;
  const int64_t rows_main = (full * pairs / n_tiles) * bm;
  if (rows_main <= 0 || rows_main >= M) return false;
  const int64_t tail = M - rows_main, tail_tiles = ((tail + bm - 1) / bm) * n_tiles;
  const int64_t splits = std::min<int64_t>({pairs / tail_tiles, num_kb / 16, 16});
  if (splits < 3) return false;
  p->rows_main = rows_main;
  p->splits = (int)splits;
  p->kb_split = (int)((num_kb + splits - 1) / splits);
  p->m_pad = ((tail + bm - 1) / bm) * bm;
  return (size_t)splits * p->m_pad * N * sizeof(float) <= ws_bytes;
}

template <int KIND, bool R32, bool O32>
__global__ void __launch_bounds__(256) splitk_fixup_kernel(const float* __restrict__ part, int splits, int64_t m_pad,
                                                           int64_t M, int N, void* out, int64_t ldo, EpiDev e) {
  const int64_t npair = N / 2, total = M * npair;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += stride) {
    const int64_t row = i / npair;
    const int col = (int)(i - row * npair) * 2;
    float a = 0.f, b = 0.f;
    for (int sp = 0; sp < splits; ++sp) {
      const float2 v = *reinterpret_cast<const float2*>(part + ((int64_t)sp * m_pad + row) * N + col);
      a += v.x;
      b += v.y;
    }
    float r0 = 0.f, r1 = 0.f;
    if constexpr (KIND == EPI_GATED_RES || KIND == EPI_RES) {
      if constexpr (R32) {
        const float2 rv = *reinterpret_cast<const float2*>(static_cast<const float*>(e.res) + row * e.ldr + col);
        r0 = rv.x;
        r1 = rv.y;
      } else {
        const uint32_t rv = *reinterpret_cast<const uint32_t*>(static_cast<const __nv_bfloat16*>(e.res) + row * e.ldr + col);
        r0 = bf16_lo(rv);
        r1 = bf16_hi(rv);
      }
    }
    epi_pair<true>(e, row + e.row_base, col, a, b, r0, r1);
    if (!ACID_IN_BOUNDS(kSiteGemmStore, row * ldo + col + 1, (M - 1) * ldo + N)) continue;
    if constexpr (O32)
      *reinterpret_cast<float2*>(static_cast<float*>(out) + row * ldo + col) = make_float2(a, b);
    else
      *reinterpret_cast<uint32_t*>(static_cast<__nv_bfloat16*>(out) + row * ldo + col) = pack_bf16(a, b);
  }
}

template <int KIND, bool R32, bool O32>
acid_status launch_splitk_fixup(const SplitKPlan& sp, const float* part, int64_t M, int N, void* out, int64_t ldo,
                                const Epilogue& epi, cudaStream_t s) {
  const int64_t total = M * (N / 2);
  const int grid = (int)std::min<int64_t>((total + 255) / 256, (int64_t)num_sms() * 8);
  splitk_fixup_kernel<KIND, R32, O32><<<grid, 256, 0, s>>>(part, sp.splits, sp.m_pad, M, N, out, ldo, to_dev(epi));
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

template <int KIND, bool R32 = false>
acid_status launch_splitk_fixup_kind(const SplitKPlan& sp, const float* part, int64_t M, int N, void* out,
                                     int64_t ldo, const Epilogue& epi, cudaStream_t s) {
  return epi.out_fp32 ? launch_splitk_fixup<KIND, R32, true>(sp, part, M, N, out, ldo, epi, s)
                      : launch_splitk_fixup<KIND, R32, false>(sp, part, M, N, out, ldo, epi, s);
}

// The split-K units of the tail rows [M rows of A], then the fixup into out.
acid_status launch_tc2_splitk(const void* A, int64_t lda, int64_t M, int K, const void* W, int N, void* out,
                              int64_t ldo, const Epilogue& epi, const SplitKPlan& sp, cudaStream_t s) {
  using Kern = decltype(&gemm_tc2_kernel<EPI_BIAS, false, true, true>);
  const Kern kern = gemm_tc2_kernel<EPI_BIAS, false, true, true>;
  static bool attr_done = false;
  if (!attr_done) {
    ACID_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Tc2Cfg::SMEM));
    attr_done = true;
  }
  float* part = static_cast<float*>(epi.splitk_ws);
  CUtensorMap ta, tb, to;
  ACID_TRY(make_tmap_bf16(&ta, A, M, K, lda, BM));
  ACID_TRY(make_tmap_bf16(&tb, W, N, K, K, Tc2Cfg::BN / 2));
  ACID_TRY(make_tmap_out(&to, part, (int64_t)sp.splits * sp.m_pad, N, N, true));
  GemmDims g{M, N, K, part, N, 1};
  g.splits = sp.splits;
  g.kb_split = sp.kb_split;
  g.m_pad = sp.m_pad;
  Epilogue raw;  // the accumulator as it is: no bias, fp32
  raw.out_fp32 = true;
  const int64_t units = ((M + 2 * BM - 1) / (2 * BM)) * ((N + Tc2Cfg::BN - 1) / Tc2Cfg::BN) * sp.splits;
  const int pairs = max_pairs<EPI_BIAS, false, true>();
  ACID_REQUIRE(pairs > 0, ACID_ERR_CUDA, "linear: no resident CTA pair for the pair GEMM");
  {
    ProfScope prof(PROF_LINEAR, 2.0 * (double)M * N * K, s);
    kern<<<2 * (int)std::min<int64_t>(units, pairs), kGemmThreads, Tc2Cfg::SMEM, s>>>(ta, tb, to, g, to_dev(raw));
    ACID_CHECK_LAUNCH();
  }
  switch (epi.kind) {
    case EPI_GELU: return launch_splitk_fixup_kind<EPI_GELU>(sp, part, M, N, out, ldo, epi, s);
    case EPI_ROPE_QKV: return launch_splitk_fixup_kind<EPI_ROPE_QKV>(sp, part, M, N, out, ldo, epi, s);
    case EPI_GATED_RES:
      return epi.res_fp32 ? launch_splitk_fixup_kind<EPI_GATED_RES, true>(sp, part, M, N, out, ldo, epi, s)
                          : launch_splitk_fixup_kind<EPI_GATED_RES, false>(sp, part, M, N, out, ldo, epi, s);
    case EPI_RES:
      return epi.res_fp32 ? launch_splitk_fixup_kind<EPI_RES, true>(sp, part, M, N, out, ldo, epi, s)
                          : launch_splitk_fixup_kind<EPI_RES, false>(sp, part, M, N, out, ldo, epi, s);
    default: return launch_splitk_fixup_kind<EPI_BIAS>(sp, part, M, N, out, ldo, epi, s);
  }
}

// ===========================================================================
// fp32 SIMT GEMM: 64x64 tile, 16-deep K slices, 4x4 outputs per thread
// ===========================================================================
constexpr int SB = 64, SK = 16;

template <typename TW>
__global__ void __launch_bounds__(256) gemm_f32_kernel(const float* __restrict__ A, int64_t lda, int64_t M, int K,
                                                       const TW* __restrict__ W, int N, float* out, int64_t ldo,
                                                       EpiDev e) {
  __shared__ float As[SK][SB + 4];
  __shared__ float Ws[SK][SB + 4];
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int64_t m0 = (int64_t)blockIdx.y * SB;
  const int n0 = blockIdx.x * SB;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += SK) {
    for (int i = threadIdx.x; i < SB * SK; i += 256) {
      const int r = i / SK, kk = i % SK;
      const int64_t gm = m0 + r;
      const int gk = k0 + kk, gn = n0 + r;
      As[kk][r] = (gm < M && gk < K) ? A[gm * lda + gk] : 0.f;
      Ws[kk][r] = (gn < N && gk < K) ? io<TW>::ld(W + (int64_t)gn * K + gk) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < SK; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        a[i] = As[kk][ty * 4 + i];
        b[i] = Ws[kk][tx * 4 + i];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  const float* res = static_cast<const float*>(e.res);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t row = m0 + ty * 4 + i;
    if (row >= M) continue;
    const int64_t grow = row + e.row_base;
#pragma unroll
    for (int j = 0; j < 4; j += 2) {
      const int col = n0 + tx * 4 + j;
      if (col >= N) continue;  // N is even
      float r0 = 0.f, r1 = 0.f;
      if (epi_reads_res(e.kind)) {
        r0 = res[row * e.ldr + col];
        r1 = res[row * e.ldr + col + 1];
      }
      float a = acc[i][j], b = acc[i][j + 1];
      epi_pair<false>(e, grow, col, a, b, r0, r1);
      if (!ACID_IN_BOUNDS(kSiteGemmF32, row * ldo + col + 1, (M - 1) * ldo + N)) continue;
      out[row * ldo + col] = a;
      out[row * ldo + col + 1] = b;
    }
  }
}

}  // namespace

acid_status linear_forward_f32(const void* A, int64_t lda, int64_t M, int K, int w_dtype, const void* W, int N,
                               void* out, int64_t ldo, const Epilogue& epi, cudaStream_t s) {
  ACID_REQUIRE(M >= 0 && K > 0 && N > 0, ACID_ERR_INVALID_ARG, "linear: bad shape");
  if (M == 0) return ACID_OK;  // no rows: nothing is read, pointers may be null
  ACID_REQUIRE(A && W && out, ACID_ERR_INVALID_ARG, "linear: null pointer");
  ACID_REQUIRE(N % 2 == 0, ACID_ERR_UNSUPPORTED, "linear fp32: N must be even");
  dim3 grid((N + SB - 1) / SB, (unsigned)((M + SB - 1) / SB));
  if (w_dtype == ACID_BF16)
    gemm_f32_kernel<__nv_bfloat16><<<grid, 256, 0, s>>>(static_cast<const float*>(A), lda, M, K,
                                                        static_cast<const __nv_bfloat16*>(W), N,
                                                        static_cast<float*>(out), ldo, to_dev(epi));
  else
    gemm_f32_kernel<float><<<grid, 256, 0, s>>>(static_cast<const float*>(A), lda, M, K,
                                                static_cast<const float*>(W), N, static_cast<float*>(out), ldo,
                                                to_dev(epi));
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

acid_status linear_forward(int dtype, const void* A, int64_t lda, int64_t M, int K, const void* W, int N, void* out,
                           int64_t ldo, const Epilogue& epi, cudaStream_t s) {
  ACID_REQUIRE(M >= 0 && K > 0 && N > 0, ACID_ERR_INVALID_ARG, "linear: bad shape");
  if (M == 0) return ACID_OK;  // no rows: nothing is read, pointers may be null
  ACID_REQUIRE(A && W && out, ACID_ERR_INVALID_ARG, "linear: null pointer");
  ACID_REQUIRE(epi.kind != EPI_ROPE_QKV || (epi.rope.table != nullptr && epi.head_dim > 0 && epi.d > 0),
               ACID_ERR_INVALID_ARG, "linear: RoPE epilogue needs a table");
  ACID_REQUIRE(epi.kind != EPI_ROPE_QKV ||
                   (int64_t)epi.rope.grid_f * epi.rope.grid_h * epi.rope.grid_w < (int64_t(1) << 24),
               ACID_ERR_UNSUPPORTED, "linear: RoPE positions must be below 2^24");
  ACID_REQUIRE(!epi_reads_res(epi.kind) || epi.residual != nullptr, ACID_ERR_INVALID_ARG,
               "linear: residual epilogue needs a residual");
  if (dtype == ACID_FP32) return linear_forward_f32(A, lda, M, K, ACID_FP32, W, N, out, ldo, epi, s);
  ACID_REQUIRE(N % 32 == 0 && K % 8 == 0, ACID_ERR_UNSUPPORTED, "linear bf16: need N % 32 == 0 and K % 8 == 0");
  ACID_REQUIRE(ldo % 8 == 0 && aligned(out, 16) && (!epi.residual || (epi.ldr % 8 == 0 && aligned(epi.residual, 16))),
               ACID_ERR_UNSUPPORTED, "linear bf16: output/residual must be 16-byte aligned rows");
  ACID_REQUIRE(epi.kind != EPI_ROPE_QKV || (epi.head_dim & (epi.head_dim - 1)) == 0, ACID_ERR_UNSUPPORTED,
               "linear bf16: the RoPE epilogue needs a power-of-two head_dim");
  // The widest tile that the output spans: a 128-wide tile moves a third more
  // shared-memory bytes per FLOP than a 256-wide one, which costs more than
  // the zero-filled columns of a partial last tile (N = 1920: 7% extra MMA
  // work, against about 1.6x the throughput).
  // SM pairs where the tiles' mainloop is long enough to matter: measured at
  // M = 32760, pairs are 1-2% faster for N = 4608 / 8960 or K = 8960 and 2-3%
  // slower for the 1536 x 1536 gated-residual output projection, whose
  // residual traffic bounds it as much as its FLOPs do.
  // Kinds without a residual leave through the pair kernel's accumulator-
  // layout epilogue, which makes pairs faster from N = 1024 on (measured at
  // M = 32760: cross-attention query 1535 -> 1565 TFLOP/s, the K = 128 patch
  // embedding 40 -> 32 us); the residual kinds stay on single SMs up to 2048.
  const bool no_res = epi.kind == EPI_BIAS || epi.kind == EPI_GELU || epi.kind == EPI_ROPE_QKV;
  if (N > 128 && (N > 2048 || K > 2048 || (no_res && N >= 1024))) {
    SplitKPlan sp;
    if (epi.splitk_ws != nullptr && aligned(epi.splitk_ws, 128) &&
        splitk_plan(M, N, K, epi.splitk_bytes, max_pairs<EPI_BIAS, false, true>(), &sp)) {
      ACID_TRY(launch_tc2(A, lda, sp.rows_main, K, W, N, out, ldo, epi, s));
      const size_t osz = epi.out_fp32 ? 4 : 2, rsz = epi.res_fp32 ? 4 : 2;
      Epilogue et = epi;
      et.row_base += sp.rows_main;
      if (et.residual) et.residual = static_cast<const uint8_t*>(et.residual) + sp.rows_main * et.ldr * rsz;
      return launch_tc2_splitk(static_cast<const uint8_t*>(A) + sp.rows_main * lda * 2, lda, M - sp.rows_main, K, W,
                               N, static_cast<uint8_t*>(out) + sp.rows_main * ldo * osz, ldo, et, sp, s);
    }
    return launch_tc2(A, lda, M, K, W, N, out, ldo, epi, s);
  }
  if (N > 128) return launch_tc<256>(A, lda, M, K, W, N, out, ldo, epi, s);
  if (N > 64) return launch_tc<128>(A, lda, M, K, W, N, out, ldo, epi, s);
  return launch_tc<64>(A, lda, M, K, W, N, out, ldo, epi, s);
}

ACID_DEVICE_FLAG_READER(take_device_error_gemm)
ACID_BOUNDS_READER(take_bounds_gemm)

}  // namespace acid
