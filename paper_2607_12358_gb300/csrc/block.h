// Block-level internals shared by the block entry point and the step loop.
#pragma once

#include <stddef.h>
#include <stdint.h>

#include "acid.h"
#include "internal.h"

namespace acid {

// Bump allocator over a caller-provided workspace (base may be null to size it).
struct Bump {
  uint8_t* base = nullptr;
  size_t off = 0;
  template <typename T>
  T* take(size_t count) {
    off = (off + 1023) & ~size_t(1023);
    T* p = reinterpret_cast<T*>(base ? base + off : nullptr);
    off += count * sizeof(T);
    return p;
  }
};

struct BlockWs {
  float* mod = nullptr;    // [12d] modulation (video stream / only stream)
  float* mod_t = nullptr;  // [6d] HV_DUAL text-stream modulation
  float2* rope = nullptr;  // RoPE tables
  uint8_t* u = nullptr;    // [rows, d] LayerNorm output / scratch
  uint8_t* qkv = nullptr;  // [rows, 3d]
  uint8_t* att = nullptr;  // [rows, d] (HV_SINGLE: [rows, d + ffn])
  uint8_t* hid = nullptr;  // [rows, ffn]
  uint8_t* kvc = nullptr;  // [n_text, 2d] cross-attention keys / values
  float* xm = nullptr;     // [rows, d] fp32 residual stream between the two branches
  void* attn_part = nullptr;  // attention partial results of a split last wave
  size_t attn_part_bytes = 0;
  void* splitk = nullptr;     // partial accumulators of a split-K last GEMM round
  size_t splitk_bytes = 0;
  size_t bytes = 0;
};

int64_t block_rows(const acid_block_desc& d);
BlockWs block_ws_layout(const acid_block_desc& d, void* base);
acid_status validate_block_desc(const acid_block_desc& d);
acid_status validate_block_weights(const acid_block_desc& d, const acid_block_weights& w);
// ctx_kv: this block's cross-attention keys and values [n_text, 2d] computed
// ahead (the text is fixed for a generation), or null to project ctx here.
acid_status block_forward_impl(const acid_block_desc& D, void* x, const float* temb, const void* ctx,
                               const void* ctx_kv, const acid_block_weights& W, const BlockWs& ws,
                               const RopeTable* rope, cudaStream_t s);

}  // namespace acid
