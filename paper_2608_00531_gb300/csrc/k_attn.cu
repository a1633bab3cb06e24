// Stage 4 host side: the workspace plan and the launch of the persistent
// tcgen05 tree-attention kernel (k_attn_tc.cu).
//
// Workspace layout (caller-owned, 256-byte aligned):
//   cnt     int32 [units_max], 256-byte rounded   (launch tag << 9) | pieces arrived,
//                                                 per unit (any initial contents)
//   ws_o    fp32  [units_max + kAttnMaxCtas][32][256] float4: per piece slot, column-major
//                 partial outputs (float4 column c of row r at [slot][c][r])
//   ws_lse  fp32  [(units_max + kAttnMaxCtas) * 256]        partial log-sum-exps
// A unit is (sequence, kv head, row group of 2 x floor(128 / G) tree nodes);
// a unit split across CTAs needs one slot per piece, and the pieces of all
// units number at most units + CTAs.
#include <algorithm>

#include "attn_common.cuh"

namespace cure {

bool plan_tree_attn(int batch, int n_max, int heads_q, const cure_kv_desc& kv, AttnPlan* plan) {
  if (kv.heads_kv <= 0 || heads_q % kv.heads_kv != 0) return false;
  const int G = heads_q / kv.heads_kv;
  if (G < 1 || G > kAttnRowsCta) return false;
  const int npb = kAttnRowsCta / G;
  const int rg_max = (n_max + 2 * npb - 1) / (2 * npb);
  AttnPlan p;
  p.units_max = batch * kv.heads_kv * rg_max;
  p.ws_cnt = ((size_t)p.units_max * sizeof(int) + 255) / 256 * 256;
  const size_t rows = (size_t)(p.units_max + kAttnMaxCtas) * 2 * kAttnRowsCta;
  p.ws_o = rows * kAttnD * sizeof(float);
  p.ws_lse = (rows * sizeof(float) + 255) / 256 * 256;
  *plan = p;
  return true;
}

cudaError_t launch_tree_attn(const AttnPlan& plan, const uint16_t* q, const uint16_t* tree_k,
                             const uint16_t* tree_v, const uint16_t* k_cache,
                             const uint16_t* v_cache, const cure_kv_desc& kv,
                             const int32_t* cache_len, const int32_t* n_nodes,
                             const uint64_t* anc, int batch, int n_max, int heads_q, float scale,
                             uint16_t* out, void* workspace, int* err, cudaStream_t s) {
  if (batch == 0) return cudaSuccess;
  AttnArgs A;
  A.q = q;
  A.tk = tree_k;
  A.tv = tree_v;
  A.inplace = tree_k == nullptr ? 1 : 0;
  A.kc = k_cache;
  A.vc = v_cache;
  A.kv = kv;
  A.cache_len = cache_len;
  A.n_nodes = n_nodes;
  A.anc = anc;
  A.batch = batch;
  A.n_max = n_max;
  A.heads_q = heads_q;
  A.G = heads_q / kv.heads_kv;
  A.W = (n_max + 63) / 64;
  A.cap = kv.layout == 0 ? kv.max_len : kv.max_len * kv.page_size;
  A.units_max = plan.units_max;
  A.unit_cost = kAttnUnitCost;
  A.scale_log2 = scale * 1.4426950408889634f;
  char* ws = reinterpret_cast<char*>(workspace);
  A.cnt = reinterpret_cast<int*>(ws);
  A.ws_o = reinterpret_cast<float*>(ws + plan.ws_cnt);
  A.ws_lse = reinterpret_cast<float*>(ws + plan.ws_cnt + plan.ws_o);
  A.out = out;
  A.err = err;
  // One CTA per SM, unless the shape's work (bounded above from the cache
  // capacity, since the lengths are on the device) gives a CTA fewer than
  // kAttnMinTiles tile positions: a unit cut into many pieces costs a merge of
  // that many partials, which the last piece does alone, so small problems
  // take fewer, longer pieces.
  const int64_t tiles_unit = (A.cap + kAttnKeys - 1) / kAttnKeys +
                             (A.inplace ? 0 : (n_max + kAttnKeys - 1) / kAttnKeys);
  const int64_t positions = (int64_t)plan.units_max * (tiles_unit + kAttnUnitCost);
  int ctas = std::min(num_sms(), kAttnMaxCtas);
  if (kAttnMinTiles > 0)
    ctas = (int)std::max<int64_t>(1, std::min<int64_t>(ctas, positions / kAttnMinTiles));
  return launch_tree_attn_tc(A, dim3(ctas, 1, 1), s);
}

}  // namespace cure
