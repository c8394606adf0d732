// Attention over the full spatio-temporal token sequence (self, joint and
// cross attention of the DiT blocks).  RoPE is applied to q and k once per
// token by the QKV projection's epilogue, so this kernel reads pre-rotated
// operands.
//
// bf16 path: a flash-attention kernel on tcgen05 tensor cores.  A work item
// is two 128-row query tiles (a, b) of one head; its CTA streams 128-key K/V
// tiles that both query tiles share:
//   warp 0      TMA producer: Q_a, Q_b once, then K_j and V_j into 2-deep rings
//               (128-byte swizzle);
//   warp 1      MMA issuer, in the order S_a(0) S_b(0) | PV_a(j) S_a(j+1)
//               PV_b(j) S_b(j+1) | ... so that the tensor core works on one
//               query tile while the softmax of the other runs;
//               S_t = Q_t K_j^T lands in TMEM, P_t is written back over S_t
//               (bf16, two per column) and O_t += P_t V_j reads P_t from TMEM
//               and V_j from shared memory;
//   warps 2-5   softmax of tile a, warps 6-9 softmax of tile b: one thread
//               per query row keeps the running max and sum, and rescales O_t
//               in TMEM only when the running max grows by more than 2^8 (the
//               final division by the sum makes the result independent of
//               when rescaling happens).
// attn_tc_kernel runs one item per CTA (long key ranges: self and joint
// attention).  attn_persist_kernel runs items of a few key tiles (cross
// attention over a short text) on persistent CTAs: the next item's Q loads
// and first S MMAs overlap the current item's last softmax, and the output
// leaves through shared memory and TMA stores.
// fp32 path: one warp per query row, exact expf, for the fp32 mode.
#include <cudaTypedefs.h>
#include <math.h>

#include <type_traits>

#include "common.cuh"
#include "internal.h"

namespace acid {

acid_status make_tmap_bf16(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int64_t ld, int box_rows);
acid_status make_tmap_bf16_box(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int64_t ld,
                               int box_cols, int box_rows, CUtensorMapSwizzle swizzle);

namespace {

constexpr int kTileQ = 128;  // query rows per tile (two tiles per CTA)
constexpr int kBQ = 2 * kTileQ;
constexpr int kAttnThreads = 320;
constexpr float kRescaleLog2 = 8.0f;
constexpr int kAttnPartCtas = kAttnSplitCtas;  // CTAs of a split tail wave (partials workspace capacity)

struct AttnDev {
  int64_t nq, nk;
  int q_col, k_col, v_col;
  void* out;
  int64_t ldo;
  int o_col;
  float scale_log2;  // log2(e) / sqrt(head_dim)
  // work item = (query-tile pair, head), numbered head-major.  attn_tc_kernel:
  // CTA blockIdx.x handles item item_base + blockIdx.x / splits and the
  // split-th part of the key range; with splits > 1 it writes its
  // unnormalised output and (max, sum) per row to part_o / part_ml instead of
  // the final output.  attn_persist_kernel: CTA blockIdx.x handles items
  // item_base + blockIdx.x + k * gridDim.x below item_end.
  int nqp;
  int item_base, item_end;
  int splits;
  float* part_o;   // [CTA][256 rows][D]
  float* part_ml;  // [CTA][256 rows][2]
};

template <int D>
struct AttnCfg {
  // Keys per K/V tile.  Head dim 128: 128-key tiles, one CTA per SM (S and O
  // of both query tiles fill TMEM).  Head dim 64: 64-key tiles, so a CTA needs
  // 256 TMEM columns and about 64 KB of shared memory and two CTAs share an
  // SM, four query tiles in flight: at this head dim the exponentials, not
  // the MMAs, set the pace and need more warps to overlap.
  static constexpr int BKV = D <= 64 ? 64 : 128;
  static constexpr int CTAS_PER_SM = D <= 64 ? 2 : 1;
  static constexpr int CH = D / 64;                  // 64-column chunks per row
  static constexpr int CHUNK_Q = 128 * 128;          // 128 rows x 128 bytes
  static constexpr int CHUNK_KV = BKV * 128;         // BKV rows x 128 bytes
  static constexpr int T_BYTES = CH * CHUNK_Q;       // one 128-row tile of Q
  static constexpr int KV_BYTES = CH * CHUNK_KV;     // one K or V tile
  static constexpr int OFF_Q = 0;                    // Q_a, Q_b
  static constexpr int OFF_K = OFF_Q + 2 * T_BYTES;  // 2-deep rings
  static constexpr int OFF_V = OFF_K + 2 * KV_BYTES;
  static constexpr int OFF_BAR = OFF_V + 2 * KV_BYTES;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;
  // attn_persist_kernel adds the output staging: per softmax warp two
  // 32-row x 32-column bf16 boxes (64-byte swizzle) for TMA stores
  static constexpr int STAGE_BOX = 32 * 64;
  static constexpr int OFF_STAGE_P = OFF_V + 2 * KV_BYTES;
  static constexpr int OFF_BAR_P = OFF_STAGE_P + 8 * 2 * STAGE_BOX;
  static constexpr int SMEM_P = OFF_BAR_P + 256 + 1024;
  // TMEM columns: S_a [0,BKV), S_b [BKV,2BKV) (P_t over the first BKV/2
  // columns of S_t), O_a [2BKV, 2BKV+D), O_b [2BKV+D, 2BKV+2D)
  static constexpr uint32_t S_COL = 0, O_COL = 2 * BKV;
  static constexpr uint32_t TMEM_COLS = 2 * BKV + 2 * D;
  __host__ __device__ static constexpr uint32_t o_col(int t) { return O_COL + t * D; }
};

// Softmax of one key tile for this thread's query row (row r of tile t is
// TMEM lane r): waits for S_t, writes P_t = 2^(s * scale - m) over the S
// region as bf16 pairs, updates the running reference max m and sum l,
// rescales O_t when the reference moves, and hands P_t to the MMA warp.
// phase: this tile's step count in the CTA (barrier parity); first: the
// item's first key tile; valid: keys of a masked (partial last) tile.
template <int D, bool MASKED>
__device__ __forceinline__ bool softmax_tile(uint64_t* s_full, uint64_t* pv_done, uint64_t* p_full, int phase,
                                             bool first, int valid, uint32_t s_addr, uint32_t o_addr,
                                             float scale_log2, float& m_run, float& l_run) {
  using C = AttnCfg<D>;
  // The lanes of a warp wait on the same phase, so they give up together
  // (after the wait limit) and the warp-collective tcgen05.ld / st below stay
  // convergent; a vote here would rule out a phase that completes exactly at
  // the limit for some lanes only, but costs 2-3% in this loop.
  if (!mbar_wait(s_full, phase & 1)) return false;
  // consume pv_done phase - 1 (already complete: s_full(phase) is committed
  // after PV(phase - 1)) so that no later parity wait is two phases behind;
  // at an item's first tile the previous item's output pass consumed it
  if (!first && !mbar_wait(pv_done, (phase - 1) & 1)) return false;
  tc_fence_after();
  float s[C::BKV];
#pragma unroll
  for (int c = 0; c < C::BKV / 32; ++c) tmem_ld32(s_addr + c * 32, reinterpret_cast<uint32_t*>(s + c * 32));
  tmem_wait_ld();
  bool resc = false;
  float f = 1.0f;
  if constexpr (MASKED) {
#pragma unroll
    for (int i = 0; i < C::BKV; ++i)
      if (i >= valid) s[i] = -INFINITY;
  }
  // e = s * scale - m_run in place (packed pairs; the first tile uses 0 as
  // the reference), with the row max of e alongside in four independent
  // 3-input max chains on the ALU pipe.  s_full(phase) is committed after
  // PV(phase - 1), so O_t and the P_t region are free here.  Lazy rescaling:
  // the reference max moves only on the first tile or when the row max
  // exceeds it by more than 2^8; then e is shifted in place.
  const uint64_t sc2 = f2_pack(scale_log2, scale_log2);
  {
    const float mref = first ? 0.f : m_run;
    const uint64_t nm2 = f2_pack(-mref, -mref);
    float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
    for (int i = 0; i < C::BKV / 2; ++i) {
      f2_unpack(f2_fma(f2_pack(s[2 * i], s[2 * i + 1]), sc2, nm2), s[2 * i], s[2 * i + 1]);
      m4[i & 3] = fmax3(m4[i & 3], s[2 * i], s[2 * i + 1]);
    }
    const float me = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
    if (first || me > kRescaleLog2) {
      if (!first) {
        resc = true;
        f = ex2_approx(-me);
        l_run *= f;
      }
      m_run = mref + me;
      const uint64_t sh2 = f2_pack(-me, -me);
#pragma unroll
      for (int i = 0; i < C::BKV / 2; ++i) f2_unpack(f2_add(f2_pack(s[2 * i], s[2 * i + 1]), sh2), s[2 * i], s[2 * i + 1]);
    }
  }
  // P = 2^e as bf16 pairs over the first BKV/2 columns of S_t, with the row
  // sum as packed fp32 pairs
  uint64_t acc0 = f2_pack(0.f, 0.f), acc1 = acc0;
#pragma unroll
  for (int half = 0; half < C::BKV / 64; ++half) {
    uint32_t pk[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const float p0 = ex2_approx(s[half * 64 + 2 * i]), p1 = ex2_approx(s[half * 64 + 2 * i + 1]);
      if (i & 1)
        acc1 = f2_add(acc1, f2_pack(p0, p1));
      else
        acc0 = f2_add(acc0, f2_pack(p0, p1));
      pk[i] = pack_bf16(p0, p1);
    }
    tmem_st32(s_addr + half * 32, pk);
  }
  float a0, a1, b0, b1;
  f2_unpack(acc0, a0, a1);
  f2_unpack(acc1, b0, b1);
  const float ls = (a0 + a1) + (b0 + b1);
  l_run += ls;
  if (__any_sync(0xffffffffu, resc)) {
#pragma unroll 1
    for (int c = 0; c < D; c += 32) {
      uint32_t o[32];
      tmem_ld32(o_addr + c, o);
      tmem_wait_ld();
#pragma unroll
      for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * f);
      tmem_st32(o_addr + c, o);
    }
  }
  tmem_wait_st();
  tc_fence_before();
  mbar_arrive(p_full);
  return true;
}

// S_t = Q_t K^T for one key tile: D/16 MMAs (M128, N = BKV, K16) into TMEM
// column d; qdesc_t / kdesc_slot: shared-memory descriptors of Q_t and of the
// K ring slot (an operand at byte offset o is the descriptor plus o >> 4).
template <int D>
__device__ __forceinline__ void issue_s_mma(uint32_t d, uint64_t qdesc_t, uint64_t kdesc_slot) {
  using C = AttnCfg<D>;
  constexpr uint32_t idesc_s = idesc_bf16_f32(128, C::BKV, false, false);
#pragma unroll
  for (int kk = 0; kk < D / 16; ++kk) {
    const uint64_t off_a = (uint64_t)(((kk >> 2) * C::CHUNK_Q + (kk & 3) * 32) >> 4);
    const uint64_t off_b = (uint64_t)(((kk >> 2) * C::CHUNK_KV + (kk & 3) * 32) >> 4);
    mma_bf16_ss(d, qdesc_t + off_a, kdesc_slot + off_b, idesc_s, kk != 0);
  }
}

// O_t (+)= P_t V for one key tile: BKV/16 MMAs (M128, N = D, K16), P_t from
// TMEM at column p (bf16 pairs over the S region), V MN-major from the ring
// slot; accumulate is false on an item's first key tile.
template <int D>
__device__ __forceinline__ void issue_pv_mma(uint32_t d, uint32_t p, uint64_t vdesc_slot, bool accumulate) {
  using C = AttnCfg<D>;
  constexpr uint32_t idesc_o = idesc_bf16_f32(128, D, false, true);
#pragma unroll
  for (int kk = 0; kk < C::BKV / 16; ++kk)
    mma_bf16_ts(d, p + kk * 8, vdesc_slot + (uint64_t)((kk * 16 * 128) >> 4), idesc_o, accumulate || kk != 0);
}

// TMA loads of one K or V tile (D / 64 chunks of 64 columns) into a ring slot.
template <int D>
__device__ __forceinline__ void load_kv_tile(uint8_t* dst, const CUtensorMap* map, uint64_t* bar, int col, int row) {
  using C = AttnCfg<D>;
  mbar_expect_tx(bar, C::KV_BYTES);
  for (int c = 0; c < C::CH; ++c) tma_load_2d(dst + c * C::CHUNK_KV, map, bar, col + c * 64, row);
}

// Failure path (a wait ran out): the producer waits, bounded, until the loads
// it has issued have landed (the Q tiles, and the last K and V tiles of each
// two-slot ring), so that no copy writes into the shared memory of a CTA
// that has left; the MMA thread waits, bounded, for the MMAs it has issued
// before tensor memory is freed.  Never called on the normal path.
__device__ __noinline__ void drain_loads(uint64_t* q_full, uint64_t* k_full, uint64_t* v_full, int nk, int nv) {
  mbar_wait(q_full, 0);
  for (int j = nk > 2 ? nk - 2 : 0; j < nk; ++j) mbar_wait(&k_full[j & 1], (j >> 1) & 1);
  for (int j = nv > 2 ? nv - 2 : 0; j < nv; ++j) mbar_wait(&v_full[j & 1], (j >> 1) & 1);
}
__device__ __noinline__ void drain_mmas(uint64_t* drain) {
  mma_commit(drain);
  mbar_wait(drain, 0);
}

template <int D>
__global__ void __launch_bounds__(kAttnThreads, AttnCfg<D>::CTAS_PER_SM)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                   const __grid_constant__ CUtensorMap tmV, AttnDev a) {
  using C = AttnCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem + C::OFF_Q;
  uint8_t* sK = smem + C::OFF_K;
  uint8_t* sV = smem + C::OFF_V;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* q_full = bars + 0;
  uint64_t* k_full = bars + 1;    // [2]
  uint64_t* k_empty = bars + 3;   // [2]
  uint64_t* v_full = bars + 5;    // [2]
  uint64_t* v_empty = bars + 7;   // [2]
  uint64_t* s_full = bars + 9;    // [2] per query tile
  uint64_t* p_full = bars + 11;   // [2] per query tile
  uint64_t* pv_done = bars + 13;  // [2] per query tile
  uint64_t* drain = bars + 15;    // failure path: the MMAs issued so far have completed
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 16);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int item = a.item_base + (int)blockIdx.x / a.splits, split = (int)blockIdx.x % a.splits;
  const int qt = item % a.nqp, h = item / a.nqp;
  const int nkv_all = (int)((a.nk + C::BKV - 1) / C::BKV);
  const int jb = (int)((int64_t)split * nkv_all / a.splits);  // this CTA's key tiles [jb, jb + nkv)
  const int nkv = (int)((int64_t)(split + 1) * nkv_all / a.splits) - jb;

  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&k_full[i], 1);
      mbar_init(&k_empty[i], 1);
      mbar_init(&v_full[i], 1);
      mbar_init(&v_empty[i], 1);
      mbar_init(&s_full[i], 1);
      mbar_init(&p_full[i], 128);
      mbar_init(&pv_done[i], 1);
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
    if (lane == 0) {  // ---------------------------------------- TMA producer
      mbar_expect_tx(q_full, 2 * C::T_BYTES);
      for (int t = 0; t < 2; ++t)
        for (int c = 0; c < C::CH; ++c)
          tma_load_2d(sQ + t * C::T_BYTES + c * C::CHUNK_Q, &tmQ, q_full, a.q_col + h * D + c * 64,
                      qt * kBQ + t * kTileQ);
      int nk_issued = 0, nv_issued = 0;
      for (int j = 0; j < nkv; ++j) {
        const int st = j & 1, round = j >> 1;
        if (round > 0 && !mbar_wait(&k_empty[st], (round - 1) & 1)) break;
        load_kv_tile<D>(sK + st * C::KV_BYTES, &tmK, &k_full[st], a.k_col + h * D, (jb + j) * C::BKV);
        nk_issued = j + 1;
        if (round > 0 && !mbar_wait(&v_empty[st], (round - 1) & 1)) break;
        load_kv_tile<D>(sV + st * C::KV_BYTES, &tmV, &v_full[st], a.v_col + h * D, (jb + j) * C::BKV);
        nv_issued = j + 1;
      }
      if (nv_issued < nkv) drain_loads(q_full, k_full, v_full, nk_issued, nv_issued);
    }
  } else if (warp == 1) {
    if (lane == 0) {  // ---------------------------------------- MMA issuer
      // Shared-memory descriptors are built once; an operand at byte offset o
      // from a base is the base descriptor plus o >> 4 (the 14-bit address
      // field cannot overflow: shared memory ends below 256 KB).
      const uint64_t qdesc = smem_desc_sw128(smem_u32(sQ), 16, 1024);
      const uint64_t kdesc = smem_desc_sw128(smem_u32(sK), 16, 1024);
      const uint64_t vdesc = smem_desc_sw128(smem_u32(sV), C::CHUNK_KV, 1024);
      // S_t(j) = Q_t K_j^T into the S region of tile t
      auto issue_s = [&](int t, int j) {
        issue_s_mma<D>(tmem + C::S_COL + t * C::BKV, qdesc + (uint64_t)((t * C::T_BYTES) >> 4),
                       kdesc + (uint64_t)(((j & 1) * C::KV_BYTES) >> 4));
        mma_commit(&s_full[t]);
      };
      bool ok = mbar_wait(q_full, 0) && mbar_wait(&k_full[0], 0);
      if (ok) {
        tc_fence_after();
        issue_s(0, 0);
        issue_s(1, 0);
        mma_commit(&k_empty[0]);
      }
      for (int j = 0; ok && j < nkv; ++j) {
        const int st = j & 1;
        for (int t = 0; t < 2 && ok; ++t) {
          if (!mbar_wait(&p_full[t], j & 1)) { ok = false; break; }
          if (t == 0 && !mbar_wait(&v_full[st], (j >> 1) & 1)) { ok = false; break; }
          tc_fence_after();
          // O_t += P_t V_j
          issue_pv_mma<D>(tmem + C::o_col(t), tmem + C::S_COL + t * C::BKV,
                          vdesc + (uint64_t)((st * C::KV_BYTES) >> 4), j != 0);
          mma_commit(&pv_done[t]);
          if (t == 1) mma_commit(&v_empty[st]);
          if (j + 1 < nkv) {
            if (t == 0 && !mbar_wait(&k_full[st ^ 1], ((j + 1) >> 1) & 1)) { ok = false; break; }
            tc_fence_after();
            issue_s(t, j + 1);
            if (t == 1) mma_commit(&k_empty[st ^ 1]);
          }
        }
      }
      if (!ok) drain_mmas(drain);
    }
  } else {  // ---------------------------------------- softmax: warps 2-5 tile a, 6-9 tile b
    const int t = (warp - 2) >> 2;
    const int q = warp & 3;
    const int r = q * 32 + lane;  // row within the query tile == TMEM lane
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    const uint32_t s_addr = tmem + lane_base + C::S_COL + t * C::BKV;
    const uint32_t o_addr = tmem + lane_base + C::o_col(t);
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    // One key tile; the masked variant (keys past the end of the sequence)
    // is compiled separately and runs only on a partial last tile.
    auto step = [&](int j, auto masked) -> bool {
      return softmax_tile<D, decltype(masked)::value>(&s_full[t], &pv_done[t], &p_full[t], j, j == 0,
                                                      (int)(a.nk - (int64_t)(jb + j) * C::BKV), s_addr, o_addr,
                                                      a.scale_log2, m_run, l_run);
    };
    const bool partial_last = (int64_t)(jb + nkv) * C::BKV > a.nk;
    for (int j = 0; j < nkv; ++j) {
      const bool ok_j = (j == nkv - 1 && partial_last) ? step(j, std::true_type{}) : step(j, std::false_type{});
      if (!ok_j) {
        ok = false;
        break;
      }
    }
    // ---------------------------------------------------- epilogue: O_t / l
    if (ok) ok = mbar_wait(&pv_done[t], (nkv - 1) & 1);
    tc_fence_after();
    const int64_t row = (int64_t)qt * kBQ + t * kTileQ + r;
    const float inv = 1.0f / l_run;
#pragma unroll 1
    for (int c = 0; c < D; c += 32) {
      uint32_t o[32];
      tmem_ld32(o_addr + c, o);
      tmem_wait_ld();
      if (!ok || row >= a.nq) continue;
      if (a.splits > 1) {  // partial result of this key range: unnormalised O
        float* pp = a.part_o + ((int64_t)blockIdx.x * kBQ + t * kTileQ + r) * D + c;
#pragma unroll
        for (int i = 0; i < 32; i += 4)
          *reinterpret_cast<float4*>(pp + i) = make_float4(__uint_as_float(o[i]), __uint_as_float(o[i + 1]),
                                                           __uint_as_float(o[i + 2]), __uint_as_float(o[i + 3]));
        continue;
      }
      float v[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(o[i]) * inv;
      __nv_bfloat16* op = static_cast<__nv_bfloat16*>(a.out) + row * a.ldo + a.o_col + h * D + c;
#pragma unroll
      for (int i = 0; i < 32; i += 8) store8(op + i, v + i);
    }
    if (a.splits > 1 && ok && row < a.nq)
      *reinterpret_cast<float2*>(a.part_ml + ((int64_t)blockIdx.x * kBQ + t * kTileQ + r) * 2) =
          make_float2(m_run, l_run);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// Persistent variant for items of a few key tiles.  Each CTA walks the items
// item_base + blockIdx.x + k * gridDim.x; one counter g numbers its key-tile
// steps across items, and every per-step barrier phase and ring slot follows
// it.  Q_t of the next item is loaded once the current item's last S_t MMA
// has completed (q_empty), so the MMA warp issues the next item's first S
// right after the current item's last PV.  The output leaves through two
// staging boxes per softmax warp and TMA stores, which frees the softmax
// warps for the next item.
template <int D>
__global__ void __launch_bounds__(kAttnThreads, AttnCfg<D>::CTAS_PER_SM)
    attn_persist_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                        const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmO,
                        AttnDev a) {
  using C = AttnCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem + C::OFF_Q;
  uint8_t* sK = smem + C::OFF_K;
  uint8_t* sV = smem + C::OFF_V;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR_P);
  uint64_t* q_full = bars + 0;    // [2] per query tile
  uint64_t* q_empty = bars + 2;   // [2] per query tile
  uint64_t* k_full = bars + 4;    // [2]
  uint64_t* k_empty = bars + 6;   // [2]
  uint64_t* v_full = bars + 8;    // [2]
  uint64_t* v_empty = bars + 10;  // [2]
  uint64_t* s_full = bars + 12;   // [2] per query tile
  uint64_t* p_full = bars + 14;   // [2] per query tile
  uint64_t* pv_done = bars + 16;  // [2] per query tile
  uint64_t* drain = bars + 18;    // failure path: the MMAs issued so far have completed
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 19);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int item0 = a.item_base + (int)blockIdx.x, item_step = (int)gridDim.x;
  const int n_items = item0 < a.item_end ? (a.item_end - 1 - item0) / item_step + 1 : 0;
  const int nkv = (int)((a.nk + C::BKV - 1) / C::BKV);
  const int total = n_items * nkv;  // key-tile steps of this CTA

  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
    tma_prefetch_desc(&tmO);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&q_full[i], 1);
      mbar_init(&q_empty[i], 1);
      mbar_init(&k_full[i], 1);
      mbar_init(&k_empty[i], 1);
      mbar_init(&v_full[i], 1);
      mbar_init(&v_empty[i], 1);
      mbar_init(&s_full[i], 1);
      mbar_init(&p_full[i], 128);
      mbar_init(&pv_done[i], 1);
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
    if (lane == 0) {  // ---------------------------------------- TMA producer
      bool ok = true;
      int nk_issued = 0, nv_issued = 0;
      for (int k = 0, g = 0; ok && k < n_items; ++k) {
        const int item = item0 + k * item_step;
        const int qt = item % a.nqp, h = item / a.nqp;
        // Q_t of item k replaces Q_t of item k - 1 once that item's last S_t is done
        for (int t = 0; t < 2 && ok; ++t) {
          if (k > 0 && !mbar_wait(&q_empty[t], (k - 1) & 1)) { ok = false; break; }
          mbar_expect_tx(&q_full[t], C::T_BYTES);
          for (int c = 0; c < C::CH; ++c)
            tma_load_2d(sQ + t * C::T_BYTES + c * C::CHUNK_Q, &tmQ, &q_full[t], a.q_col + h * D + c * 64,
                        qt * kBQ + t * kTileQ);
        }
        for (int j = 0; ok && j < nkv; ++j, ++g) {
          const int st = g & 1, round = g >> 1;
          if (round > 0 && !mbar_wait(&k_empty[st], (round - 1) & 1)) { ok = false; break; }
          load_kv_tile<D>(sK + st * C::KV_BYTES, &tmK, &k_full[st], a.k_col + h * D, j * C::BKV);
          nk_issued = g + 1;
          if (round > 0 && !mbar_wait(&v_empty[st], (round - 1) & 1)) { ok = false; break; }
          load_kv_tile<D>(sV + st * C::KV_BYTES, &tmV, &v_full[st], a.v_col + h * D, j * C::BKV);
          nv_issued = g + 1;
        }
      }
      // after a wait ran out: the last K and V loads of each ring have landed
      // (Q loads of an item are waited on by the MMA thread before any use)
      if (!ok) {
        for (int j = nk_issued > 2 ? nk_issued - 2 : 0; j < nk_issued; ++j) mbar_wait(&k_full[j & 1], (j >> 1) & 1);
        for (int j = nv_issued > 2 ? nv_issued - 2 : 0; j < nv_issued; ++j) mbar_wait(&v_full[j & 1], (j >> 1) & 1);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {  // ---------------------------------------- MMA issuer
      const uint64_t qdesc = smem_desc_sw128(smem_u32(sQ), 16, 1024);
      const uint64_t kdesc = smem_desc_sw128(smem_u32(sK), 16, 1024);
      const uint64_t vdesc = smem_desc_sw128(smem_u32(sV), C::CHUNK_KV, 1024);
      // S_t = Q_t K^T of step g into the S region of tile t; after an item's
      // last key tile (last_tile) the producer may replace Q_t
      auto issue_s = [&](int t, int g, bool last_tile) {
        issue_s_mma<D>(tmem + C::S_COL + t * C::BKV, qdesc + (uint64_t)((t * C::T_BYTES) >> 4),
                       kdesc + (uint64_t)(((g & 1) * C::KV_BYTES) >> 4));
        mma_commit(&s_full[t]);
        if (last_tile) mma_commit(&q_empty[t]);
      };
      bool ok = total > 0 && mbar_wait(&k_full[0], 0);
      for (int t = 0; t < 2 && ok; ++t) {
        if (!mbar_wait(&q_full[t], 0)) { ok = false; break; }
        tc_fence_after();
        issue_s(t, 0, nkv == 1);
      }
      if (ok) mma_commit(&k_empty[0]);
      // step g (key tile j of item k): PV_a(g) S_a(g+1) PV_b(g) S_b(g+1); at an
      // item boundary S(g+1) reads the next item's Q
      for (int g = 0, j = 0, k = 0; ok && g < total; ++g) {
        const int st = g & 1, gn = g + 1;
        const bool boundary = j + 1 == nkv;  // step gn starts item k + 1
        const int jn = boundary ? 0 : j + 1;
        for (int t = 0; t < 2 && ok; ++t) {
          if (!mbar_wait(&p_full[t], g & 1)) { ok = false; break; }
          if (t == 0 && !mbar_wait(&v_full[st], (g >> 1) & 1)) { ok = false; break; }
          tc_fence_after();
          issue_pv_mma<D>(tmem + C::o_col(t), tmem + C::S_COL + t * C::BKV,
                          vdesc + (uint64_t)((st * C::KV_BYTES) >> 4), j != 0);
          mma_commit(&pv_done[t]);
          if (t == 1) mma_commit(&v_empty[st]);
          if (gn < total) {
            if (t == 0 && !mbar_wait(&k_full[st ^ 1], (gn >> 1) & 1)) { ok = false; break; }
            if (boundary && !mbar_wait(&q_full[t], (k + 1) & 1)) { ok = false; break; }
            tc_fence_after();
            issue_s(t, gn, jn == nkv - 1);
            if (t == 1) mma_commit(&k_empty[st ^ 1]);
          }
        }
        j = jn;
        k += boundary;
      }
      if (!ok) drain_mmas(drain);
    }
  } else {  // ---------------------------------------- softmax: warps 2-5 tile a, 6-9 tile b
    const int t = (warp - 2) >> 2;
    const int q = warp & 3;
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    const uint32_t s_addr = tmem + lane_base + C::S_COL + t * C::BKV;
    const uint32_t o_addr = tmem + lane_base + C::o_col(t);
    uint8_t* stage = smem + C::OFF_STAGE_P + (warp - 2) * 2 * C::STAGE_BOX;
    const int valid_last = (int)(a.nk - (int64_t)(nkv - 1) * C::BKV);  // keys of the last tile
    int n_st = 0;  // output boxes this warp has stored
    bool ok = true;
    for (int item = item0, g = 0; ok && item < a.item_end; item += item_step) {
      float m_run = -INFINITY, l_run = 0.f;
      for (int j = 0; j < nkv; ++j, ++g) {
        const bool ok_j = (j == nkv - 1 && valid_last < C::BKV)
                              ? softmax_tile<D, true>(&s_full[t], &pv_done[t], &p_full[t], g, j == 0, valid_last,
                                                      s_addr, o_addr, a.scale_log2, m_run, l_run)
                              : softmax_tile<D, false>(&s_full[t], &pv_done[t], &p_full[t], g, j == 0, C::BKV,
                                                       s_addr, o_addr, a.scale_log2, m_run, l_run);
        if (!ok_j) {
          ok = false;
          break;
        }
      }
      // ------------------------------------------------ output: O_t / l
      // (the next PV_t, which overwrites O_t, follows this warpgroup's next
      // p_full arrival, issued after these loads have completed)
      if (ok) ok = mbar_wait(&pv_done[t], (g - 1) & 1);
      ok = __all_sync(0xffffffffu, ok);  // the item loop continues for the whole warp or not at all
      tc_fence_after();
      const int qt = item % a.nqp, h = item / a.nqp;
      const int64_t row0 = (int64_t)qt * kBQ + t * kTileQ + q * 32;  // this warp's 32 rows
      const float inv = 1.0f / l_run;
#pragma unroll 1
      for (int c = 0; c < D; c += 32) {
        uint32_t o[32];
        tmem_ld32(o_addr + c, o);
        tmem_wait_ld();
        if (!ok || row0 >= a.nq) continue;  // warp-uniform
        // The warp's 32 x 32 box leaves through shared memory and one TMA
        // store (rows past nq are clipped by the tensor map).  Two boxes
        // alternate; the store issued two boxes ago must have read this one.
        uint8_t* box = stage + (n_st & 1) * C::STAGE_BOX;
        if (lane == 0 && n_st >= 2) bulk_wait_group_read<1>();
        __syncwarp();
        // row `lane`: 64 bytes as four 16-byte units, unit u stored at
        // u ^ ((lane >> 1) & 3) (the 64-byte swizzle: conflict-free writes)
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          uint4 w;
          w.x = pack_bf16(__uint_as_float(o[8 * u + 0]) * inv, __uint_as_float(o[8 * u + 1]) * inv);
          w.y = pack_bf16(__uint_as_float(o[8 * u + 2]) * inv, __uint_as_float(o[8 * u + 3]) * inv);
          w.z = pack_bf16(__uint_as_float(o[8 * u + 4]) * inv, __uint_as_float(o[8 * u + 5]) * inv);
          w.w = pack_bf16(__uint_as_float(o[8 * u + 6]) * inv, __uint_as_float(o[8 * u + 7]) * inv);
          *reinterpret_cast<uint4*>(box + lane * 64 + ((u ^ ((lane >> 1) & 3)) << 4)) = w;
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_store_2d(&tmO, box, a.o_col + h * D + c, (int)row0);
          bulk_commit_group();
        }
        ++n_st;
      }
    }
    if (lane == 0) bulk_wait_group<0>();  // output stores complete before the CTA ends
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// Merges the key-range parts of the split items: for every row,
// O = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s with M = max_s m_s.
// One warp per row (256 rows per item), D / 32 columns per lane.
template <int D>
__global__ void __launch_bounds__(256) attn_merge_kernel(AttnDev a, int item0, int tail, int splits) {
  const int wrow = (int)(blockIdx.x * 8 + (threadIdx.x >> 5));  // row over all tail items
  const int lane = threadIdx.x & 31;
  if (wrow >= tail * kBQ) return;
  const int it = wrow / kBQ, rr = wrow % kBQ;
  const int item = item0 + it;
  const int qt = item % a.nqp, h = item / a.nqp;
  const int64_t row = (int64_t)qt * kBQ + rr;
  if (row >= a.nq) return;
  float M = -INFINITY;
  for (int sp = 0; sp < splits; ++sp) M = fmaxf(M, a.part_ml[((int64_t)(it * splits + sp) * kBQ + rr) * 2]);
  float acc[D / 32] = {};
  float L = 0.f;
  for (int sp = 0; sp < splits; ++sp) {
    const int64_t slot = (int64_t)(it * splits + sp) * kBQ + rr;
    const float w = ex2_approx(a.part_ml[slot * 2] - M);
    L += w * a.part_ml[slot * 2 + 1];
#pragma unroll
    for (int i = 0; i < D / 32; ++i) acc[i] = fmaf(w, a.part_o[slot * D + i * 32 + lane], acc[i]);
  }
  const float inv = 1.0f / L;
  if (!ACID_IN_BOUNDS(kSiteAttnMerge, row * a.ldo + a.o_col + h * D + D - 1, a.nq * a.ldo)) return;
  __nv_bfloat16* op = static_cast<__nv_bfloat16*>(a.out) + row * a.ldo + a.o_col + h * D;
#pragma unroll
  for (int i = 0; i < D / 32; ++i) op[i * 32 + lane] = __float2bfloat16_rn(acc[i] * inv);
}

int num_sms_attn() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
  }
  return n;
}

// Items with at most this many key tiles run on persistent CTAs.
constexpr int kPersistMaxKeyTiles = 8;

template <int D>
acid_status launch_attn_tc(const AttnArgs& x, cudaStream_t s) {
  using C = AttnCfg<D>;
  static bool attr_done = false;
  if (!attr_done) {
    ACID_CUDA(cudaFuncSetAttribute(attn_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM));
    ACID_CUDA(cudaFuncSetAttribute(attn_persist_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_P));
    attr_done = true;
  }
  CUtensorMap tq, tk, tv;
  ACID_TRY(make_tmap_bf16(&tq, x.q, x.nq, x.ldq, x.ldq, kTileQ));
  ACID_TRY(make_tmap_bf16(&tk, x.k, x.nk, x.ldk, x.ldk, C::BKV));
  ACID_TRY(make_tmap_bf16(&tv, x.v, x.nk, x.ldv, x.ldv, C::BKV));
  AttnDev a;
  a.nq = x.nq;
  a.nk = x.nk;
  a.q_col = x.q_col;
  a.k_col = x.k_col;
  a.v_col = x.v_col;
  a.out = x.out;
  a.ldo = x.ldo;
  a.o_col = x.o_col;
  a.scale_log2 = (float)(1.4426950408889634 / sqrt((double)D));
  a.nqp = (int)((x.nq + kBQ - 1) / kBQ);
  a.item_base = 0;
  a.item_end = 0;
  a.splits = 1;
  a.part_o = nullptr;
  a.part_ml = nullptr;
  const int items = a.nqp * x.heads;
  const int nkv_all = (int)((x.nk + C::BKV - 1) / C::BKV);
  // Long key ranges: items fill whole waves of CTAS_PER_SM CTAs per SM; the
  // items of a last, partial wave are split along the key range so that they
  // fill one wave together, and their partial results are merged.  Short key
  // ranges: persistent CTAs take all items, and the few CTAs that take one
  // item more cost less than a split wave's start-up and merge (measured:
  // 109 against 121 us for 32760 x 512 keys).
  const int slots = num_sms_attn() * C::CTAS_PER_SM;
  const int full = (items / slots) * slots, tail = items - full;
  int splits = tail > 0 ? std::min(std::min(kAttnPartCtas, slots) / tail, nkv_all) : 1;
  const size_t part_need = (size_t)tail * splits * kBQ * (D + 2) * sizeof(float);
  const bool persist = nkv_all <= kPersistMaxKeyTiles;
  const bool split_tail =
      !persist && full > 0 && tail > 0 && splits >= 2 && x.part != nullptr && x.part_bytes >= part_need;
  ProfScope prof(PROF_ATTENTION, 4.0 * (double)x.nq * (double)x.nk * D * x.heads, s);
  const int main_items = split_tail ? full : items;
  if (persist) {
    // output: 32-row x 32-column boxes, one per softmax warp and column chunk
    CUtensorMap to;
    ACID_TRY(make_tmap_bf16_box(&to, x.out, x.nq, x.ldo, x.ldo, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B));
    a.item_end = main_items;
    attn_persist_kernel<D><<<std::min(main_items, slots), kAttnThreads, C::SMEM_P, s>>>(tq, tk, tv, to, a);
  } else {
    attn_tc_kernel<D><<<main_items, kAttnThreads, C::SMEM, s>>>(tq, tk, tv, a);
  }
  ACID_CHECK_LAUNCH();
  if (!split_tail) return ACID_OK;
  a.item_base = full;
  a.splits = splits;
  a.part_o = static_cast<float*>(x.part);
  a.part_ml = a.part_o + (size_t)tail * splits * kBQ * D;
  attn_tc_kernel<D><<<tail * splits, kAttnThreads, C::SMEM, s>>>(tq, tk, tv, a);
  ACID_CHECK_LAUNCH();
  attn_merge_kernel<D><<<tail * kBQ / 8, 256, 0, s>>>(a, full, tail, splits);
  ACID_CHECK_LAUNCH();
  return ACID_OK;
}

// ---------------------------------------------------------------- fp32 path
__global__ void __launch_bounds__(256) attn_f32_kernel(const float* __restrict__ q, int64_t ldq, int q_col,
                                                       const float* __restrict__ k, int64_t ldk, int k_col,
                                                       const float* __restrict__ v, int64_t ldv, int v_col, float* out,
                                                       int64_t ldo, int o_col, int64_t nq, int64_t nk, int D,
                                                       float scale) {
  const int64_t row = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int h = blockIdx.y;
  const int lane = threadIdx.x & 31;
  if (row >= nq) return;
  constexpr int kMaxPer = 4;  // D <= 128
  float qv[kMaxPer], o[kMaxPer];
  const int per = D / 32;
#pragma unroll
  for (int i = 0; i < kMaxPer; ++i) {
    qv[i] = i < per ? q[row * ldq + q_col + h * D + i * 32 + lane] : 0.f;
    o[i] = 0.f;
  }
  float m = -INFINITY, l = 0.f;
  for (int64_t j = 0; j < nk; ++j) {
    const float* kr = k + j * ldk + k_col + h * D;
    float sdot = 0.f;
#pragma unroll
    for (int i = 0; i < kMaxPer; ++i)
      if (i < per) sdot = fmaf(qv[i], kr[i * 32 + lane], sdot);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) sdot += __shfl_xor_sync(0xffffffffu, sdot, off);
    const float sc = sdot * scale;
    const float mn = fmaxf(m, sc);
    const float corr = expf(m - mn);
    const float p = expf(sc - mn);
    l = l * corr + p;
    const float* vr = v + j * ldv + v_col + h * D;
#pragma unroll
    for (int i = 0; i < kMaxPer; ++i)
      if (i < per) o[i] = fmaf(p, vr[i * 32 + lane], o[i] * corr);
    m = mn;
  }
  if (!ACID_IN_BOUNDS(kSiteAttnF32, row * ldo + o_col + h * D + D - 1, nq * ldo)) return;
#pragma unroll
  for (int i = 0; i < kMaxPer; ++i)
    if (i < per) out[row * ldo + o_col + h * D + i * 32 + lane] = o[i] / l;
}

}  // namespace

acid_status attention_forward(int dtype, const AttnArgs& x, cudaStream_t s) {
  ACID_REQUIRE(x.nk > 0 && x.nq >= 0 && x.heads > 0, ACID_ERR_INVALID_ARG, "attention: bad shape");
  if (x.nq == 0) return ACID_OK;  // no query rows: nothing is read, pointers may be null
  ACID_REQUIRE(x.q && x.k && x.v && x.out, ACID_ERR_INVALID_ARG, "attention: null pointer");
  if (dtype == ACID_FP32) {
    ACID_REQUIRE(x.head_dim % 32 == 0 && x.head_dim <= 128, ACID_ERR_UNSUPPORTED,
                 "attention fp32: head_dim must be 32, 64, 96 or 128");
    dim3 grid((unsigned)((x.nq + 7) / 8), (unsigned)x.heads);
    attn_f32_kernel<<<grid, 256, 0, s>>>((const float*)x.q, x.ldq, x.q_col, (const float*)x.k, x.ldk, x.k_col,
                                         (const float*)x.v, x.ldv, x.v_col, (float*)x.out, x.ldo, x.o_col, x.nq, x.nk,
                                         x.head_dim, (float)(1.0 / sqrt((double)x.head_dim)));
    ACID_CHECK_LAUNCH();
    return ACID_OK;
  }
  ACID_REQUIRE(x.head_dim == 64 || x.head_dim == 128, ACID_ERR_UNSUPPORTED, "attention bf16: head_dim must be 64 or 128");
  ACID_REQUIRE(x.q_col % 8 == 0 && x.k_col % 8 == 0 && x.v_col % 8 == 0 && x.o_col % 8 == 0 && x.ldo % 8 == 0,
               ACID_ERR_UNSUPPORTED, "attention bf16: column offsets must be multiples of 8");
  ACID_REQUIRE(aligned(x.out, 16), ACID_ERR_UNSUPPORTED, "attention bf16: output must be 16-byte aligned");
  if (x.head_dim == 128) return launch_attn_tc<128>(x, s);
  return launch_attn_tc<64>(x, s);
}

ACID_DEVICE_FLAG_READER(take_device_error_attention)
ACID_BOUNDS_READER(take_bounds_attention)

}  // namespace acid
