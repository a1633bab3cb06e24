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
  int batch, n_max, heads_q, G, W, cap;
  int inplace;     // 1: no tree tensors; node j's K/V rows are cache slot L_b + j
  int units_max;   // piece counters in the workspace
  int unit_cost;   // fixed cost of a unit in the stream-K split, in 64-key tile times
  float scale_log2;
  int* cnt;        // [units_max] (launch tag << 9) | pieces arrived, per unit
  uint32_t tag;    // this launch's tag (set by the launcher)
  float* ws_o;     // [units_max + kAttnMaxCtas][32][256] float4 partial outputs
  float* ws_lse;   // [(units_max + kAttnMaxCtas) * 256] partial base-2 log-sum-exps
  uint16_t* out;
  int* err;
};

constexpr int kAttnD = 128;       // head dim
constexpr int kAttnRowsCta = 128; // query rows (node x group head) per CTA
constexpr int kAttnKeys = 64;     // keys per tile
constexpr int kAttnMaxBatch = 256;  // sequences per call (the CTA keeps per-sequence prefix sums)
constexpr int kAttnMaxCtas = 256;   // persistent CTAs (one per SM, at most this many)
// Fixed cost of a unit (its piece start-up, epilogue and split merge) in
// 64-key tile times, charged in the stream-K split so that CTAs starting
// more units get fewer tiles.
#ifndef CURE_ATTN_UNIT_COST
#define CURE_ATTN_UNIT_COST 3
#endif
constexpr int kAttnUnitCost = CURE_ATTN_UNIT_COST;
// Fewest tile positions (tiles plus unit costs) a CTA is given before the
// grid shrinks below one CTA per SM (0: always one per SM).
#ifndef CURE_ATTN_MIN_TILES
#define CURE_ATTN_MIN_TILES 8
#endif
constexpr int kAttnMinTiles = CURE_ATTN_MIN_TILES;

// The persistent tcgen05 kernel (writes `out`; merges split units itself).
cudaError_t launch_tree_attn_tc(const AttnArgs& A, dim3 grid, cudaStream_t s);

}  // namespace cure
