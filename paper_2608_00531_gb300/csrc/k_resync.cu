// Stage 6: repair resynchronisation (Sec. 3.5, Alg. 1 last step).
//
// gather: one warp per (layer, K|V, sequence, depth) row; rows past the
// accepted length leave at once.  A row is heads_kv * head_dim bf16 values
// (1 KiB for 4 x 128), moved with 16-byte vector loads and stores.
// finalize: one thread per sequence writes the new lengths and the replay
// list; it runs after the gather so that cache_len_out may alias the input.
#include "common.cuh"

namespace cure {
namespace {

constexpr int kWarps = 8;

__global__ void __launch_bounds__(32 * kWarps)
resync_gather_kernel(int layers, LayerPtrs caches, cure_kv_desc kv, const uint4* __restrict__ tree_k,
                     const uint4* __restrict__ tree_v, int batch, int n_max, int block,
                     const int32_t* __restrict__ path_nodes, const int32_t* __restrict__ accept_len,
                     const int32_t* __restrict__ cache_len_in, int* err) {
  pdl_begin();
  const int lane = threadIdx.x & 31;
  const int T = block + 1;                      // depths 0..K
  const int64_t item = (int64_t)blockIdx.x * kWarps + (threadIdx.x >> 5);
  const int64_t per_layer = 2LL * batch * T;
  const int layer = (int)(item / per_layer);
  const int64_t rem = item % per_layer;
  const int which = (int)(rem / ((int64_t)batch * T));  // 0 = K, 1 = V
  const int b = (int)((rem / T) % batch);
  const int t = (int)(rem % T);
  if (layer >= layers) return;
  const int a = accept_len[b];
  if (t > a) return;
  const int node = path_nodes[(int64_t)b * (block + 2) + t];
  if (node < 0 || node >= n_max) {
    if (lane == 0) flag(err, CURE_DEVERR_NODES);
    return;
  }
  const int slot = cache_len_in[b] + t;
  const int row_vec = kv.heads_kv * kv.head_dim / 8;  // uint4 per row
  int64_t dst_row;
  if (kv.layout == 0) {
    if (slot < 0 || slot >= kv.max_len) {
      if (lane == 0) flag(err, CURE_DEVERR_SLOT);
      return;
    }
    dst_row = (int64_t)b * kv.max_len + slot;
  } else {
    const int pi = slot / kv.page_size;
    if (slot < 0 || pi >= kv.max_len) {
      if (lane == 0) flag(err, CURE_DEVERR_SLOT);
      return;
    }
    const int page = kv.block_table[(int64_t)b * kv.max_len + pi];
    if (page < 0 || page >= kv.num_pages) {
      if (lane == 0) flag(err, CURE_DEVERR_PAGE);
      return;
    }
    dst_row = (int64_t)page * kv.page_size + slot % kv.page_size;
  }
  const uint4* src = (which == 0 ? tree_k : tree_v) +
                     ((((int64_t)layer * batch + b) * n_max + node) * row_vec);
  uint4* dst = reinterpret_cast<uint4*>(which == 0 ? caches.k[layer] : caches.v[layer]) +
               dst_row * row_vec;
  for (int i = lane; i < row_vec; i += 32) dst[i] = __ldg(src + i);
}

__global__ void resync_finalize_kernel(int batch, int block, const int32_t* __restrict__ accept_len,
                                       const int32_t* __restrict__ diverge_depth,
                                       const int32_t* __restrict__ out_tokens,
                                       const int32_t* cache_len_in, int32_t* cache_len_out,
                                       int32_t* __restrict__ draft_valid_len,
                                       int32_t* __restrict__ replay_tokens,
                                       int32_t* __restrict__ n_replay) {
  pdl_begin();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= batch) return;
  const int P = block + 2;
  const int L = cache_len_in[b];
  const int a = accept_len[b];
  const int d = diverge_depth[b];
  int n = 0;
  if (d >= 0) {
    // path tokens at depths d..a are out_tokens[d-1 .. a-1]; then the next token
    for (int t = d; t <= a + 1; ++t) replay_tokens[(int64_t)b * P + n++] = out_tokens[(int64_t)b * P + t - 1];
    draft_valid_len[b] = L + d;
  } else {
    replay_tokens[(int64_t)b * P + n++] = out_tokens[(int64_t)b * P + a];
    draft_valid_len[b] = L + a + 1;
  }
  for (int t = n; t < P; ++t) replay_tokens[(int64_t)b * P + t] = -1;
  n_replay[b] = n;
  cache_len_out[b] = L + a + 1;
}

}  // namespace

cudaError_t launch_resync(int layers, const LayerPtrs& caches, const cure_kv_desc& kv,
                          const uint16_t* tree_k, const uint16_t* tree_v, int batch, int n_max,
                          int block, const int32_t* path_nodes, const int32_t* accept_len,
                          const int32_t* diverge_depth, const int32_t* out_tokens,
                          const int32_t* cache_len_in, int32_t* cache_len_out,
                          int32_t* draft_valid_len, int32_t* replay_tokens, int32_t* n_replay,
                          int* err, cudaStream_t s) {
  if (batch == 0) return cudaSuccess;
  if (layers > 0) {
    const int64_t items = (int64_t)layers * 2 * batch * (block + 1);
    const int64_t grid = (items + kWarps - 1) / kWarps;
    const cudaError_t e = launch_pdl(
        resync_gather_kernel, dim3((unsigned)grid), dim3(32 * kWarps), 0, s, layers, caches, kv,
        reinterpret_cast<const uint4*>(tree_k), reinterpret_cast<const uint4*>(tree_v), batch, n_max,
        block, path_nodes, accept_len, cache_len_in, err);
    if (e != cudaSuccess) return e;
  }
  return launch_pdl(resync_finalize_kernel, dim3((batch + 127) / 128), dim3(128), 0, s, batch, block,
                    accept_len, diverge_depth, out_tokens, cache_len_in, cache_len_out, draft_valid_len,
                    replay_tokens, n_replay);
}

}  // namespace cure
