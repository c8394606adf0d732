// acid_dit_block_forward: one DiT block as a sequence of the library's
// kernels (adaLN LayerNorm, tcgen05 GEMMs with fused epilogues, flash
// attention), for the four block kinds of the workloads.
#include <string>

#include "block.h"
#include "common.cuh"
#include "internal.h"

namespace acid {

namespace {

size_t esize(int dtype) { return dtype == ACID_BF16 ? 2 : 4; }

template <typename T = uint8_t>
T* off(void* base, int64_t elems, int dtype) {
  return reinterpret_cast<T*>(static_cast<uint8_t*>(base) + elems * (int64_t)esize(dtype));
}
const void* coff(const void* base, int64_t elems, int dtype) {
  return static_cast<const uint8_t*>(base) + elems * (int64_t)esize(dtype);
}

acid_status lin(int dt, const void* A, int64_t lda, int64_t M, int K, const acid_linear& L, int N, void* out,
                int64_t ldo, Epilogue e, cudaStream_t s) {
  e.bias = L.b;
  return linear_forward(dt, A, lda, M, K, L.w, N, out, ldo, e, s);
}

}  // namespace

int64_t block_rows(const acid_block_desc& d) {
  const int64_t nv = (int64_t)d.grid_f * d.grid_h * d.grid_w;
  return d.kind == ACID_BLOCK_WAN ? nv : nv + d.n_text;
}

BlockWs block_ws_layout(const acid_block_desc& d, void* base) {
  Bump b{static_cast<uint8_t*>(base)};
  const int64_t rows = block_rows(d);
  const size_t es = esize(d.dtype);
  BlockWs w;
  w.mod = b.take<float>(12 * (size_t)d.d);
  w.mod_t = b.take<float>(6 * (size_t)d.d);
  RopeTable rt = rope_layout(d.grid_f, d.grid_h, d.grid_w, d.heads > 0 ? d.d / d.heads : 0);
  w.rope = b.take<float2>((size_t)rt.elems());
  w.u = b.take<uint8_t>(rows * d.d * es);
  w.qkv = b.take<uint8_t>(rows * 3 * (int64_t)d.d * es);
  const int64_t att_cols = d.kind == ACID_BLOCK_HV_SINGLE ? (int64_t)d.d + d.ffn : d.d;
  w.att = b.take<uint8_t>(rows * att_cols * es);
  w.hid = d.kind == ACID_BLOCK_HV_SINGLE ? nullptr : b.take<uint8_t>(rows * (int64_t)d.ffn * es);
  w.xm = d.kind == ACID_BLOCK_HV_SINGLE ? nullptr : b.take<float>(rows * (int64_t)d.d);
  if (d.dtype == ACID_BF16 && d.heads > 0) {
    w.attn_part_bytes = attn_part_bytes(d.d / d.heads);
    w.attn_part = b.take<uint8_t>(w.attn_part_bytes);
    w.splitk_bytes = kSplitKScratchBytes;
    w.splitk = b.take<uint8_t>(w.splitk_bytes);
  }
  w.kvc = (d.kind == ACID_BLOCK_WAN && d.n_text > 0) ? b.take<uint8_t>(d.n_text * 2 * (int64_t)d.d * es) : nullptr;
  w.bytes = b.off + 1024;
  return w;
}

acid_status validate_block_desc(const acid_block_desc& d) {
  ACID_REQUIRE(d.kind >= ACID_BLOCK_WAN && d.kind <= ACID_BLOCK_HV_SINGLE, ACID_ERR_INVALID_ARG, "block: unknown kind");
  ACID_REQUIRE(d.dtype == ACID_BF16 || d.dtype == ACID_FP32, ACID_ERR_INVALID_ARG, "block: unknown dtype");
  ACID_REQUIRE(d.d > 0 && d.heads > 0 && d.d % d.heads == 0 && d.ffn > 0, ACID_ERR_INVALID_ARG,
               "block: need d, heads, ffn > 0 and heads | d");
  ACID_REQUIRE(d.grid_f > 0 && d.grid_h > 0 && d.grid_w > 0 && d.n_text >= 0, ACID_ERR_INVALID_ARG,
               "block: bad token grid");
  ACID_REQUIRE(d.d % 64 == 0 && d.ffn % 64 == 0 && d.d <= 3072, ACID_ERR_UNSUPPORTED,
               "block: d and ffn must be multiples of 64, d <= 3072");
  const int hd = d.d / d.heads;
  if (d.dtype == ACID_BF16)
    ACID_REQUIRE(hd == 64 || hd == 128, ACID_ERR_UNSUPPORTED, "block bf16: head_dim must be 64 or 128");
  else
    ACID_REQUIRE(hd % 32 == 0 && hd <= 128, ACID_ERR_UNSUPPORTED, "block fp32: head_dim must be a multiple of 32, <= 128");
  ACID_REQUIRE(hd >= 12, ACID_ERR_UNSUPPORTED, "block: head_dim too small for 3D RoPE");
  return ACID_OK;
}

static acid_status need(const acid_linear& L, const char* name) {
  ACID_REQUIRE(L.w != nullptr, ACID_ERR_INVALID_ARG, std::string("block weights: missing ") + name);
  return ACID_OK;
}

acid_status validate_block_weights(const acid_block_desc& d, const acid_block_weights& w) {
  ACID_TRY(need(w.mod, "mod"));
  ACID_TRY(need(w.qkv, "qkv"));
  ACID_TRY(need(w.ff1, "ff1"));
  ACID_TRY(need(w.ff2, "ff2"));
  if (d.kind != ACID_BLOCK_HV_SINGLE) ACID_TRY(need(w.o, "o"));
  if (d.kind == ACID_BLOCK_WAN && d.n_text > 0) {
    ACID_TRY(need(w.cq, "cq"));
    ACID_TRY(need(w.ckv, "ckv"));
    ACID_TRY(need(w.co, "co"));
  }
  if (d.kind == ACID_BLOCK_HV_DUAL) {
    ACID_TRY(need(w.t_mod, "t_mod"));
    ACID_TRY(need(w.t_qkv, "t_qkv"));
    ACID_TRY(need(w.t_o, "t_o"));
    ACID_TRY(need(w.t_ff1, "t_ff1"));
    ACID_TRY(need(w.t_ff2, "t_ff2"));
  }
  return ACID_OK;
}

acid_status block_forward_impl(const acid_block_desc& D, void* x, const float* temb, const void* ctx,
                               const void* ctx_kv, const acid_block_weights& W, const BlockWs& ws,
                               const RopeTable* rope_in, cudaStream_t s) {
  const int dt = D.dtype;
  const int d = D.d, F = D.ffn, hd = d / D.heads;
  const int64_t L = D.kind == ACID_BLOCK_WAN ? 0 : D.n_text;  // joint text rows
  const int64_t rows = block_rows(D);
  const int64_t Nv = rows - L;
  const float eps = D.ln_eps;

  // rope tables for the video grid
  RopeTable rope;
  if (rope_in) {
    rope = *rope_in;
  } else {
    rope = rope_layout(D.grid_f, D.grid_h, D.grid_w, hd);
    ACID_TRY(rope_build(rope, ws.rope, D.rope_theta, s));
  }

  // modulation vectors
  const int nmod = D.kind == ACID_BLOCK_COG ? 12 * d : (D.kind == ACID_BLOCK_HV_SINGLE ? 3 * d : 6 * d);
  ACID_TRY(gemv(dt, W.mod.w, W.mod.b, temb, ws.mod, nmod, d, true, s));
  const float* mv = ws.mod;  // video stream (or only stream)
  const float* mt = mv;      // text stream
  if (D.kind == ACID_BLOCK_COG) mt = ws.mod + 6 * d;
  if (D.kind == ACID_BLOCK_HV_DUAL) {
    ACID_TRY(gemv(dt, W.t_mod.w, W.t_mod.b, temb, ws.mod_t, 6 * d, d, true, s));
    mt = ws.mod_t;
  }

  Epilogue ep_qkv;
  ep_qkv.kind = EPI_ROPE_QKV;
  ep_qkv.rope = rope;
  ep_qkv.rope_first_video = L;
  ep_qkv.d = d;
  ep_qkv.head_dim = hd;

  auto gated = [&](int part) {
    Epilogue e;
    e.kind = EPI_GATED_RES;
    e.gate_video = mv + part * d;
    e.gate_text = mt + part * d;
    e.gate_split = L;
    e.residual = x;
    e.ldr = d;
    return e;
  };

  AttnArgs self;
  self.q = self.k = self.v = ws.qkv;
  self.ldq = self.ldk = self.ldv = 3 * (int64_t)d;
  self.q_col = 0;
  self.k_col = d;
  self.v_col = 2 * d;
  self.nq = self.nk = rows;
  self.heads = D.heads;
  self.part = ws.attn_part;
  self.part_bytes = ws.attn_part_bytes;
  self.head_dim = hd;

  if (D.kind == ACID_BLOCK_HV_SINGLE) {
    const int64_t catw = (int64_t)d + F;
    ACID_TRY(ln_mod(dt, x, dt, ws.u, rows, d, mv, mv + d, nullptr, nullptr, 0, eps, s));
    ACID_TRY(lin(dt, ws.u, d, rows, d, W.qkv, 3 * d, ws.qkv, 3 * d, ep_qkv, s));
    Epilogue eg;
    eg.kind = EPI_GELU;
    ACID_TRY(lin(dt, ws.u, d, rows, d, W.ff1, F, off(ws.att, d, dt), catw, eg, s));
    self.out = ws.att;
    self.ldo = catw;
    ACID_TRY(attention_forward(dt, self, s));
    Epilogue e = gated(2);
    ACID_TRY(lin(dt, ws.att, catw, rows, (int)catw, W.ff2, d, x, d, e, s));
    return ACID_OK;
  }

  // The residual stream between the two branches is kept in fp32 (xm): the
  // attention branch writes x + g1 * (...) to xm, cross-attention adds into
  // xm, and the FFN branch writes the final x = xm + g2 * (...) in the block
  // dtype, so a bf16 block rounds its residual stream once.
  float* xm = ws.xm;
  auto gated_to_xm = [&](int64_t r0) {  // out: xm, residual: x (block dtype)
    Epilogue e = gated(2);
    e.row_base = r0;
    e.residual = off(x, r0 * d, dt);
    e.res_fp32 = dt == ACID_FP32;
    e.out_fp32 = true;
    return e;
  };
  auto gated_from_xm = [&](int64_t r0) {  // out: x (block dtype), residual: xm
    Epilogue e = gated(5);
    e.row_base = r0;
    e.residual = xm + r0 * d;
    e.res_fp32 = true;
    e.out_fp32 = dt == ACID_FP32;
    e.splitk_ws = ws.splitk;  // FFN2 (K = ffn): a long mainloop
    e.splitk_bytes = ws.splitk_bytes;
    return e;
  };

  // ---- attention branch: xm = x + g1 * O(Attn(RoPE(QKV(LNmod1 x))))
  ACID_TRY(ln_mod(dt, x, dt, ws.u, rows, d, mv, mv + d, mt, mt + d, L, eps, s));
  if (D.kind == ACID_BLOCK_HV_DUAL) {
    Epilogue et = ep_qkv;
    ACID_TRY(lin(dt, ws.u, d, L, d, W.t_qkv, 3 * d, ws.qkv, 3 * d, et, s));
    Epilogue ev = ep_qkv;
    ev.row_base = L;
    ACID_TRY(lin(dt, off(ws.u, L * d, dt), d, Nv, d, W.qkv, 3 * d, off(ws.qkv, L * 3 * d, dt), 3 * d, ev, s));
  } else {
    ACID_TRY(lin(dt, ws.u, d, rows, d, W.qkv, 3 * d, ws.qkv, 3 * d, ep_qkv, s));
  }
  self.out = ws.att;
  self.ldo = d;
  ACID_TRY(attention_forward(dt, self, s));
  if (D.kind == ACID_BLOCK_HV_DUAL) {
    ACID_TRY(lin(dt, ws.att, d, L, d, W.t_o, d, xm, d, gated_to_xm(0), s));
    ACID_TRY(lin(dt, off(ws.att, L * d, dt), d, Nv, d, W.o, d, xm + L * d, d, gated_to_xm(L), s));
  } else {
    ACID_TRY(lin(dt, ws.att, d, rows, d, W.o, d, xm, d, gated_to_xm(0), s));
  }

  // ---- cross-attention (WAN with text): xm += O_c(Attn(Q_c(LN xm), KV_c(ctx)))
  if (D.kind == ACID_BLOCK_WAN && D.n_text > 0) {
    ACID_TRY(ln_mod(ACID_FP32, xm, dt, ws.u, rows, d, nullptr, nullptr, nullptr, nullptr, 0, eps, s));
    Epilogue eb;
    ACID_TRY(lin(dt, ws.u, d, rows, d, W.cq, d, ws.att, d, eb, s));
    if (ctx_kv == nullptr) {
      ACID_TRY(lin(dt, ctx, d, D.n_text, d, W.ckv, 2 * d, ws.kvc, 2 * d, eb, s));
      ctx_kv = ws.kvc;
    }
    AttnArgs cross;
    cross.q = ws.att;
    cross.ldq = d;
    cross.k = cross.v = ctx_kv;
    cross.ldk = cross.ldv = 2 * (int64_t)d;
    cross.k_col = 0;
    cross.v_col = d;
    cross.out = ws.u;
    cross.ldo = d;
    cross.nq = rows;
    cross.nk = D.n_text;
    cross.heads = D.heads;
    cross.head_dim = hd;
    cross.part = ws.attn_part;
    cross.part_bytes = ws.attn_part_bytes;
    ACID_TRY(attention_forward(dt, cross, s));
    Epilogue er;
    er.kind = EPI_RES;
    er.residual = xm;
    er.ldr = d;
    er.res_fp32 = true;
    er.out_fp32 = true;
    ACID_TRY(lin(dt, ws.u, d, rows, d, W.co, d, xm, d, er, s));
  }

  // ---- FFN branch: x = xm + g2 * W2 GELU(W1 LNmod2 xm)
  ACID_TRY(ln_mod(ACID_FP32, xm, dt, ws.u, rows, d, mv + 3 * d, mv + 4 * d, mt + 3 * d, mt + 4 * d, L, eps, s));
  Epilogue eg;
  eg.kind = EPI_GELU;
  if (D.kind == ACID_BLOCK_HV_DUAL) {
    ACID_TRY(lin(dt, ws.u, d, L, d, W.t_ff1, F, ws.hid, F, eg, s));
    ACID_TRY(lin(dt, off(ws.u, L * d, dt), d, Nv, d, W.ff1, F, off(ws.hid, L * F, dt), F, eg, s));
    ACID_TRY(lin(dt, ws.hid, F, L, F, W.t_ff2, d, x, d, gated_from_xm(0), s));
    ACID_TRY(lin(dt, off(ws.hid, L * F, dt), F, Nv, F, W.ff2, d, off(x, L * d, dt), d, gated_from_xm(L), s));
  } else {
    ACID_TRY(lin(dt, ws.u, d, rows, d, W.ff1, F, ws.hid, F, eg, s));
    ACID_TRY(lin(dt, ws.hid, F, rows, F, W.ff2, d, x, d, gated_from_xm(0), s));
  }
  return ACID_OK;
}

}  // namespace acid

using namespace acid;

extern "C" acid_status acid_block_rows(const acid_block_desc* desc, int64_t* rows) {
  clear_error();
  ACID_REQUIRE(desc && rows, ACID_ERR_INVALID_ARG, "acid_block_rows: null argument");
  ACID_TRY(validate_block_desc(*desc));
  *rows = block_rows(*desc);
  return ACID_OK;
}

extern "C" acid_status acid_block_workspace_size(const acid_block_desc* desc, size_t* bytes) {
  clear_error();
  ACID_REQUIRE(desc && bytes, ACID_ERR_INVALID_ARG, "acid_block_workspace_size: null argument");
  ACID_TRY(validate_block_desc(*desc));
  *bytes = block_ws_layout(*desc, nullptr).bytes;
  return ACID_OK;
}

extern "C" acid_status acid_dit_block_forward(const acid_block_desc* desc, void* x, const acid_cond* cond,
                                              const acid_block_weights* w, void* workspace, size_t workspace_bytes,
                                              acid_stream_t stream) {
  clear_error();
  ACID_REQUIRE(desc && x && cond && w, ACID_ERR_INVALID_ARG, "acid_dit_block_forward: null argument");
  ACID_TRY(validate_block_desc(*desc));
  ACID_TRY(validate_block_weights(*desc, *w));
  ACID_REQUIRE(cond->temb != nullptr, ACID_ERR_INVALID_ARG, "acid_dit_block_forward: cond->temb is null");
  ACID_REQUIRE(!(desc->kind == ACID_BLOCK_WAN && desc->n_text > 0) || cond->ctx != nullptr || cond->ctx_kv != nullptr,
               ACID_ERR_INVALID_ARG, "acid_dit_block_forward: WAN cross-attention needs cond->ctx or cond->ctx_kv");
  ACID_REQUIRE(cond->ctx_kv == nullptr || aligned(cond->ctx_kv, 16), ACID_ERR_UNSUPPORTED,
               "acid_dit_block_forward: cond->ctx_kv must be 16-byte aligned");
  ACID_REQUIRE(aligned(x, 16), ACID_ERR_UNSUPPORTED, "acid_dit_block_forward: x must be 16-byte aligned");
  ACID_REQUIRE(workspace != nullptr && aligned(workspace, 1024), ACID_ERR_WORKSPACE,
               "acid_dit_block_forward: workspace must be non-null and 1024-byte aligned");
  BlockWs ws = block_ws_layout(*desc, workspace);
  ACID_REQUIRE(workspace_bytes >= ws.bytes, ACID_ERR_WORKSPACE,
               "acid_dit_block_forward: workspace too small (need " + std::to_string(ws.bytes) + " bytes)");
  return block_forward_impl(*desc, x, cond->temb, cond->ctx, cond->ctx_kv, *w, ws, nullptr, (cudaStream_t)stream);
}
