// Shared between the tree-attention translation units.
#pragma once

#include "common.cuh"

namespace cure {

struct AttnArgs {
  const uint16_t* q;
  const uint16_t* tk;
  const uint16_t* tv;
  const uint16_t* kc;
  const uint16_t* vc;
  cure_kv_desc kv;
  const int32_t* cache_len;
  const int32_t* n_nodes;
  const uint64_t* anc;
  int batch, n_max, heads_q, G, W, chunk, splits, rows_pad, cap;
  float scale_log2;
  float* ws_o;
  float* ws_lse;
  uint16_t* out;
  int* err;
};

constexpr int kAttnD = 128;       // head dim
constexpr int kAttnRowsCta = 128; // query rows (node x group head) per CTA
constexpr int kAttnKeys = 64;     // keys per tile

// Main split-KV kernel on tcgen05 tensor cores: partial (O, lse) per row.
cudaError_t launch_tree_attn_tc(const AttnArgs& A, dim3 grid, cudaStream_t s);

}  // namespace cure
