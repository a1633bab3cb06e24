// Stage 4: tree-masked GQA attention (Sec. 3.2 / 3.4 / 3.5: the target
// verifies every path of the repair tree in one pass with Tree Attention).
//
// Decomposition.  For sequence b and kv head h the query rows are the
// (node j, group head g) pairs, r = j * G + g, so all G query heads that share
// a kv head read each K/V tile once.  Rows are cut into blocks of 128 (one CTA
// each); the cache keys 0..L_b-1 are cut into splits of `chunk` keys (split-KV
// flash decoding); the split that holds the last cache key also takes the
// tree keys, masked per row by the node's ancestor bits.  Each CTA writes a
// partial (normalised output, base-2 log-sum-exp) per row (k_attn_tc.cu); the
// reduce kernel here merges the splits and writes bf16.
#include <cuda_bf16.h>

#include <algorithm>

#include "attn_common.cuh"

namespace cure {
namespace {

constexpr int D = kAttnD;
constexpr int kRowsCta = kAttnRowsCta;
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// One warp per output row (b, j, query head); lane owns 4 of the 128 columns.
__global__ void __launch_bounds__(256) tree_attn_reduce_kernel(AttnArgs A) {
  const int64_t item = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  const int Hq = A.heads_q;
  if (item >= (int64_t)A.batch * A.n_max * Hq) return;
  const int hq = (int)(item % Hq);
  const int j = (int)((item / Hq) % A.n_max);
  const int b = (int)(item / ((int64_t)Hq * A.n_max));
  const int n = max(1, min(A.n_nodes[b], A.n_max));
  if (j >= n) return;
  const int L = max(0, min(A.cache_len[b], A.cap));
  const int nsplit = max(1, (L + A.chunk - 1) / A.chunk);
  const int Hkv = A.kv.heads_kv;
  const int h = hq / A.G, g = hq % A.G;
  const int r = j * A.G + g;
  const int64_t zb = (int64_t)(b * Hkv + h) * A.splits;
  float M = -INFINITY;
  for (int s = 0; s < nsplit; ++s) M = fmaxf(M, A.ws_lse[(zb + s) * A.rows_pad + r]);
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  float wsum = 0.f;
  for (int s = 0; s < nsplit; ++s) {
    const int64_t pr = (zb + s) * A.rows_pad + r;
    const float w = ex2(A.ws_lse[pr] - M);
    const float4 v = *reinterpret_cast<const float4*>(A.ws_o + pr * D + lane * 4);
    acc[0] += w * v.x;
    acc[1] += w * v.y;
    acc[2] += w * v.z;
    acc[3] += w * v.w;
    wsum += w;
  }
  const float inv = 1.f / wsum;
  uint2 packed;
  packed.x = pack_bf16(acc[0] * inv, acc[1] * inv);
  packed.y = pack_bf16(acc[2] * inv, acc[3] * inv);
  *reinterpret_cast<uint2*>(A.out + (((int64_t)b * A.n_max + j) * Hq + hq) * D + lane * 4) = packed;
}

}  // namespace

bool plan_tree_attn(int batch, int n_max, int heads_q, const cure_kv_desc& kv, AttnPlan* plan) {
  if (kv.heads_kv <= 0 || heads_q % kv.heads_kv != 0) return false;
  const int G = heads_q / kv.heads_kv;
  const int64_t cap = kv.layout == 0 ? (int64_t)kv.max_len : (int64_t)kv.max_len * kv.page_size;
  AttnPlan p;
  p.rows = n_max * G;
  p.row_blocks = (p.rows + kRowsCta - 1) / kRowsCta;
  const int rows_pad = p.row_blocks * kRowsCta;
  p.chunk = 1024;
  if (cap < p.chunk) p.chunk = (int)std::max<int64_t>(kAttnKeys, ((cap + kAttnKeys - 1) / kAttnKeys) * kAttnKeys);
  p.splits = (int)std::max<int64_t>(1, (cap + p.chunk - 1) / p.chunk);
  const int64_t prow = (int64_t)batch * kv.heads_kv * p.splits * rows_pad;
  p.ws_o = (size_t)(prow * D * sizeof(float));
  p.ws_lse = (size_t)(prow * sizeof(float));
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
  A.chunk = plan.chunk;
  A.splits = plan.splits;
  A.rows_pad = plan.row_blocks * kRowsCta;
  A.cap = kv.layout == 0 ? kv.max_len : kv.max_len * kv.page_size;
  A.scale_log2 = scale * kLog2e;
  A.ws_o = reinterpret_cast<float*>(workspace);
  A.ws_lse = reinterpret_cast<float*>(reinterpret_cast<char*>(workspace) + plan.ws_o);
  A.out = out;
  A.err = err;
  dim3 grid(plan.row_blocks, plan.splits, batch * kv.heads_kv);
  cudaError_t e = launch_tree_attn_tc(A, grid, s);
  if (e != cudaSuccess) return e;
  const int64_t items = (int64_t)batch * n_max * heads_q;
  tree_attn_reduce_kernel<<<(unsigned)((items + 7) / 8), 256, 0, s>>>(A);
  return cudaGetLastError();
}

}  // namespace cure
