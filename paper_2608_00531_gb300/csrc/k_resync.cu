// Stage 6: repair resynchronisation (Sec. 3.5, Alg. 1 last step).
//
// gather: one warp per (sequence, depth, K|V, group of kLayersPerWarp layers);
// warps past the accepted length leave at once.  With no tree tensors (the
// in-place layout, node j's rows at cache slot L + j) the path rows come from
// the cache itself, and a branch-0 node, whose slot L + j is already its
// depth's, copies nothing: only the rows past the divergence move.  The warp resolves the
// path row once (tree node, cache row through the block table) and copies
// the row of each layer of its group: heads_kv * head_dim bf16 values
// (1 KiB for 4 x 128) as 16-byte vectors, all the group's loads in flight
// before its stores.
// finalize: one thread per (sequence, replay slot) writes the replay list,
// and the slot-0 thread the new lengths.  It runs in the gather's grid, or,
// when cache_len_out aliases cache_len_in, as a kernel after the gather.
#include "common.cuh"

namespace cure {
namespace {

constexpr int kWarps = 8;
constexpr int kLayersPerWarp = 2;

// Writes slot t of sequence b's replay list, and for t = 0 its lengths.  With
// a divergence at depth d the path tokens at depths d..a (out_tokens[d-1 ..
// a-1]) and the next token are replayed, else only the next token.
__device__ __forceinline__ void finalize_slot(int b, int t, int P, const int32_t* __restrict__ accept_len,
                                              const int32_t* __restrict__ diverge_depth,
                                              const int32_t* __restrict__ out_tokens,
                                              const int32_t* cache_len_in, int32_t* cache_len_out,
                                              int32_t* __restrict__ draft_valid_len,
                                              int32_t* __restrict__ replay_tokens,
                                              int32_t* __restrict__ n_replay) {
  const int L = cache_len_in[b];
  const int a = accept_len[b];
  const int d = diverge_depth[b];
  const int n = d >= 0 ? max(0, a + 2 - d) : 1;
  replay_tokens[(int64_t)b * P + t] = t < n ? out_tokens[(int64_t)b * P + (d >= 0 ? d - 1 + t : a)] : -1;
  if (t == 0) {
    draft_valid_len[b] = d >= 0 ? L + d : L + a + 1;
    n_replay[b] = n;
    cache_len_out[b] = L + a + 1;
  }
}

__global__ void __launch_bounds__(32 * kWarps)
resync_gather_kernel(int layers, LayerPtrs caches, cure_kv_desc kv, const uint4* __restrict__ tree_k,
                     const uint4* __restrict__ tree_v, int batch, int n_max, int block,
                     const int32_t* __restrict__ path_nodes, const int32_t* __restrict__ accept_len,
                     const int32_t* __restrict__ cache_len_in, int* err, int gather_blocks,
                     const int32_t* __restrict__ diverge_depth, const int32_t* __restrict__ out_tokens,
                     int32_t* cache_len_out, int32_t* __restrict__ draft_valid_len,
                     int32_t* __restrict__ replay_tokens, int32_t* __restrict__ n_replay) {
  pdl_begin();
  if ((int)blockIdx.x >= gather_blocks) {  // the finalize, when cache_len_out is not the input
    const int P = block + 2;
    const int64_t idx = (int64_t)(blockIdx.x - gather_blocks) * blockDim.x + threadIdx.x;
    if (idx < (int64_t)batch * P)
      finalize_slot((int)(idx / P), (int)(idx % P), P, accept_len, diverge_depth, out_tokens,
                    cache_len_in, cache_len_out, draft_valid_len, replay_tokens, n_replay);
    return;
  }
  const int lane = threadIdx.x & 31;
  const int T = block + 1;                      // depths 0..K
  const int groups = (layers + kLayersPerWarp - 1) / kLayersPerWarp;
  const int64_t item = (int64_t)blockIdx.x * kWarps + (threadIdx.x >> 5);
  // item = ((group * 2 + which) * batch + b) * T + t
  const int t = (int)(item % T);
  const int b = (int)((item / T) % batch);
  const int64_t gw = item / ((int64_t)T * batch);
  const int which = (int)(gw & 1), group = (int)(gw >> 1);  // which: 0 = K, 1 = V
  if (group >= groups) return;
  const int a = accept_len[b];
  if (t > a) return;
  const int node = path_nodes[(int64_t)b * (block + 2) + t];
  if (node < 0 || node >= n_max) {
    if (lane == 0) flag(err, CURE_DEVERR_NODES);
    return;
  }
  const bool inplace = tree_k == nullptr;
  if (inplace && node == t) return;  // already in its slot
  const int row_vec = kv.heads_kv * kv.head_dim / 8;  // uint4 per row
  // the cache row of slot `slot`, or -1 (error word set) when it does not exist
  auto row_of = [&](int slot) -> int64_t {
    if (kv.layout == 0) {
      if (slot < 0 || slot >= kv.max_len) {
        if (lane == 0) flag(err, CURE_DEVERR_SLOT);
        return -1;
      }
      return (int64_t)b * kv.max_len + slot;
    }
    const int pi = slot / kv.page_size;
    if (slot < 0 || pi >= kv.max_len) {
      if (lane == 0) flag(err, CURE_DEVERR_SLOT);
      return -1;
    }
    const int page = kv.block_table[(int64_t)b * kv.max_len + pi];
    if (page < 0 || page >= kv.num_pages) {
      if (lane == 0) flag(err, CURE_DEVERR_PAGE);
      return -1;
    }
    return (int64_t)page * kv.page_size + slot % kv.page_size;
  };
  const int L = cache_len_in[b];
  const int64_t dst_row = row_of(L + t);
  if (dst_row < 0) return;
  const int64_t src_row = inplace ? row_of(L + node) : 0;
  if (src_row < 0) return;
  const uint4* tree = which == 0 ? tree_k : tree_v;
  const int l0 = group * kLayersPerWarp, nl = min(kLayersPerWarp, layers - l0);
  for (int i0 = lane; i0 < row_vec; i0 += 32 * 2) {  // two vectors per lane per layer
    uint4 v[kLayersPerWarp][2];
#pragma unroll
    for (int q = 0; q < kLayersPerWarp; ++q) {
      if (q < nl) {
        const uint4* src =
            inplace ? reinterpret_cast<const uint4*>(which == 0 ? caches.k[l0 + q] : caches.v[l0 + q]) +
                          src_row * row_vec
                    : tree + ((((int64_t)(l0 + q) * batch + b) * n_max + node) * row_vec);
#pragma unroll
        for (int h = 0; h < 2; ++h)
          if (i0 + 32 * h < row_vec) v[q][h] = __ldg(src + i0 + 32 * h);
      }
    }
#pragma unroll
    for (int q = 0; q < kLayersPerWarp; ++q) {
      if (q < nl) {
        uint4* dst = reinterpret_cast<uint4*>(which == 0 ? caches.k[l0 + q] : caches.v[l0 + q]) +
                     dst_row * row_vec;
#pragma unroll
        for (int h = 0; h < 2; ++h)
          if (i0 + 32 * h < row_vec) dst[i0 + 32 * h] = v[q][h];
      }
    }
  }
}

// After the gather, so that cache_len_out may alias cache_len_in.
__global__ void resync_finalize_kernel(int batch, int block, const int32_t* __restrict__ accept_len,
                                       const int32_t* __restrict__ diverge_depth,
                                       const int32_t* __restrict__ out_tokens,
                                       const int32_t* cache_len_in, int32_t* cache_len_out,
                                       int32_t* __restrict__ draft_valid_len,
                                       int32_t* __restrict__ replay_tokens,
                                       int32_t* __restrict__ n_replay) {
  pdl_begin();
  const int P = block + 2;
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)batch * P) return;
  finalize_slot((int)(idx / P), (int)(idx % P), P, accept_len, diverge_depth, out_tokens, cache_len_in,
                cache_len_out, draft_valid_len, replay_tokens, n_replay);
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
  const int64_t slots = (int64_t)batch * (block + 2);
  // the finalize rides in the gather's grid unless cache_len_out aliases the
  // input (then it must follow the whole gather)
  const bool fuse = cache_len_out != cache_len_in;
  if (layers > 0) {
    const int64_t items =
        (int64_t)((layers + kLayersPerWarp - 1) / kLayersPerWarp) * 2 * batch * (block + 1);
    const int64_t gather = (items + kWarps - 1) / kWarps;
    const int64_t fin = fuse ? (slots + 32 * kWarps - 1) / (32 * kWarps) : 0;
    const cudaError_t e = launch_pdl(
        resync_gather_kernel, dim3((unsigned)(gather + fin)), dim3(32 * kWarps), 0, s, layers, caches, kv,
        reinterpret_cast<const uint4*>(tree_k), reinterpret_cast<const uint4*>(tree_v), batch, n_max,
        block, path_nodes, accept_len, cache_len_in, err, (int)gather, diverge_depth, out_tokens,
        cache_len_out, draft_valid_len, replay_tokens, n_replay);
    if (e != cudaSuccess || fuse) return e;
  }
  return launch_pdl(resync_finalize_kernel, dim3((unsigned)((slots + 127) / 128)), dim3(128), 0, s, batch, block,
                    accept_len, diverge_depth, out_tokens, cache_len_in, cache_len_out, draft_valid_len,
                    replay_tokens, n_replay);
}

}  // namespace cure
