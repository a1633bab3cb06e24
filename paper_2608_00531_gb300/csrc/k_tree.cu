// Stages 2+3 (UFP selection and repair-tree construction, Sec. 3.1 Eq. 1,
// Sec. 3.3, Sec. 3.4) and the acceptance walk of stage 5 (Sec. 3.5 Eq. 4).
// Both run one warp per sequence: lane i owns draft position i (K <= 32) for
// the tree build, and lanes stride over the nodes (n_max <= 256) for the walk.
#include <limits.h>

#include "common.cuh"

namespace cure {
namespace {

constexpr int kWarpsPerCta = 4;
constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ int warp_excl_scan(int v, int lane) {
  int x = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int y = __shfl_up_sync(kFull, x, off);
    if (lane >= off) x += y;
  }
  return x - v;
}

__device__ __forceinline__ void anc_prefix(uint64_t* dst, int W, int upto) {
  // bits 0..upto (inclusive) set
  for (int w = 0; w < W; ++w) {
    const int lo = w * 64;
    uint64_t word;
    if (upto >= lo + 63) word = ~0ull;
    else if (upto < lo) word = 0ull;
    else word = (upto - lo == 63) ? ~0ull : ((1ull << (upto - lo + 1)) - 1ull);
    dst[w] = word;
  }
}

// Nodes one alternative at position i adds: itself (depth i + 1) and, with
// depth-2 repairs, its successor (depth i + 2), within the block and within
// the maximum depth (0 = none).
__device__ __forceinline__ int repair_cost(int i, int K, int repair_depth, int max_depth) {
  int c = min(repair_depth, K - i);
  if (max_depth > 0) c = min(c, max(0, max_depth - i));
  return c;
}

__global__ void __launch_bounds__(32 * kWarpsPerCta)
build_tree_kernel(cure_tree_params p, const int32_t* __restrict__ top_ids,
                  const float* __restrict__ margin, const int32_t* __restrict__ root_tok,
                  const int32_t* __restrict__ cache_len, const int32_t* __restrict__ redraft,
                  int32_t* __restrict__ n_nodes, int32_t* __restrict__ tok, int32_t* __restrict__ pos,
                  int32_t* __restrict__ parent, int32_t* __restrict__ depth,
                  uint64_t* __restrict__ anc, int32_t* __restrict__ ufp_pos,
                  int32_t* __restrict__ n_ufp) {
  pdl_begin();
  const int lane = threadIdx.x & 31;
  const int wib = threadIdx.x >> 5;
  const int b = blockIdx.x * kWarpsPerCta + wib;
  if (b >= p.batch) return;
  __shared__ int s_pos_by_rank[kWarpsPerCta][32];
  __shared__ int s_cnt[kWarpsPerCta][32];
  __shared__ int s_nalt[kWarpsPerCta][32];
  __shared__ int s_width[kWarpsPerCta][34];  // nodes per depth 0..K+1 during admission

  const int K = p.block;
  const int k = p.topk;
  const int n_max = 1 + K + p.budget;
  const int W = (n_max + 63) >> 6;
  const int nalt = p.branches - 1;
  const int L = cache_len[b];

  // ---- S2: gate and rank by (margin, position)
  const bool valid = lane < K;
  const float m = valid ? margin[(int64_t)b * K + lane] : 0.f;
  bool gated = valid && (m < p.tau);
  int rank = 0;
  for (int j = 0; j < K; ++j) {
    const float mj = __shfl_sync(kFull, m, j);
    const bool gj = __shfl_sync(kFull, gated, j);
    if (gj && (mj < m || (mj == m && j < lane))) ++rank;
  }
  if (p.max_ufp > 0 && rank >= p.max_ufp) gated = false;
  const unsigned gmask = __ballot_sync(kFull, gated);
  const int n_gated = __popc(gmask);
  // alternatives this position offers: the fixed budget, or Eq. (3)'s b_i
  // (u = clip(1 - m/s, 0, 1), b = clip(round(b_min + u (b_max - b_min))),
  // each step a float32 operation rounded to nearest, halves away from zero)
  int nalt_i = nalt;
  if (p.margin_scale > 0.f) {
    const int bmin = p.branch_min, bmax = nalt;
    const float u = fminf(fmaxf(__fsub_rn(1.f, __fdiv_rn(m, p.margin_scale)), 0.f), 1.f);
    const float x = __fadd_rn((float)bmin, __fmul_rn(u, (float)(bmax - bmin)));
    nalt_i = min(max((int)roundf(x), bmin), bmax);
  }
  if (gated) s_pos_by_rank[wib][rank] = lane;
  s_cnt[wib][lane] = 0;
  s_nalt[wib][lane] = nalt_i;
  s_width[wib][lane] = 1;  // the root at depth 0, the chain node at depths 1..K
  if (lane < 2) s_width[wib][32 + lane] = 1;
  __syncwarp();

  // greedy admission in rank order; an alternative that does not fit (the
  // budget, or with a beam width a full depth) is skipped
  if (lane == 0) {
    int used = 0;
    for (int q = 0; q < n_gated; ++q) {
      const int i = s_pos_by_rank[wib][q];
      const int cost = repair_cost(i, K, p.repair_depth, p.max_depth);
      int c = 0;
      const int na = s_nalt[wib][i];
      for (int r = 0; r < na && cost > 0; ++r) {
        bool fits = used + cost <= p.budget;
        if (p.beam > 0)
          for (int dd = i + 1; dd <= i + cost; ++dd) fits = fits && s_width[wib][dd] < p.beam;
        if (fits) {
          used += cost;
          for (int dd = i + 1; dd <= i + cost; ++dd) ++s_width[wib][dd];
          ++c;
        }
      }
      s_cnt[wib][i] = c;
    }
  }
  __syncwarp();

  // ---- S3: nodes in canonical (position, rank, depth) order
  const int cnt = valid ? s_cnt[wib][lane] : 0;
  const int cost = valid ? repair_cost(lane, K, p.repair_depth, p.max_depth) : 0;
  const int mine = cnt * cost;
  const int off = warp_excl_scan(mine, lane);
  const int total_rep = __shfl_sync(kFull, off + mine, 31);
  const int n = 1 + K + total_rep;

  const int64_t nb = (int64_t)b * n_max;
  uint64_t words[4];
  if (lane == 0) {
    tok[nb] = root_tok[b];
    pos[nb] = L;
    parent[nb] = -1;
    depth[nb] = 0;
    anc_prefix(words, W, 0);
    for (int w = 0; w < W; ++w) anc[nb * W + w] = words[w];
    n_nodes[b] = n;
  }
  if (valid) {
    const int j = lane + 1;  // chain node for draft position `lane`
    tok[nb + j] = top_ids[((int64_t)b * K + lane) * k];
    pos[nb + j] = L + j;
    parent[nb + j] = j - 1;
    depth[nb + j] = j;
    anc_prefix(words, W, j);
    for (int w = 0; w < W; ++w) anc[(nb + j) * W + w] = words[w];
    // repair nodes hanging below chain node `lane`
    int node = 1 + K + off;
    for (int a = 0; a < cnt; ++a) {
      const int r = a + 2;  // rank of the alternative
      tok[nb + node] = top_ids[((int64_t)b * K + lane) * k + (r - 1)];
      pos[nb + node] = L + lane + 1;
      parent[nb + node] = lane;
      depth[nb + node] = lane + 1;
      anc_prefix(words, W, lane);
      words[node >> 6] |= 1ull << (node & 63);
      for (int w = 0; w < W; ++w) anc[(nb + node) * W + w] = words[w];
      if (cost == 2) {
        const int sn = node + 1;
        tok[nb + sn] = redraft[((int64_t)b * K + lane) * nalt + (r - 2)];
        pos[nb + sn] = L + lane + 2;
        parent[nb + sn] = node;
        depth[nb + sn] = lane + 2;
        words[sn >> 6] |= 1ull << (sn & 63);
        for (int w = 0; w < W; ++w) anc[(nb + sn) * W + w] = words[w];
      }
      node += cost;
    }
  }
  for (int j = n + lane; j < n_max; j += 32) {
    tok[nb + j] = -1;
    pos[nb + j] = -1;
    parent[nb + j] = -1;
    depth[nb + j] = -1;
    for (int w = 0; w < W; ++w) anc[(nb + j) * W + w] = 0ull;
  }

  // ---- repaired positions in selection order
  const bool took = cnt > 0;
  const unsigned tmask = __ballot_sync(kFull, took);
  int before = 0;
  for (int j = 0; j < K; ++j) {
    const int rj = __shfl_sync(kFull, rank, j);
    if (((tmask >> j) & 1u) && rj < rank) ++before;
  }
  if (valid) ufp_pos[(int64_t)b * K + lane] = -1;
  __syncwarp();
  if (took) ufp_pos[(int64_t)b * K + before] = lane;
  if (lane == 0) n_ufp[b] = __popc(tmask);
}

// One warp per sequence.
__global__ void __launch_bounds__(32 * kWarpsPerCta)
accept_walk_kernel(int batch, int n_max, int block, const int32_t* __restrict__ n_nodes,
                   const int32_t* __restrict__ tok, const int32_t* __restrict__ parent,
                   const int32_t* __restrict__ depth, const uint64_t* __restrict__ anc,
                   const int32_t* __restrict__ targ, int32_t* __restrict__ accept_len,
                   int32_t* __restrict__ best_node, int32_t* __restrict__ path_nodes,
                   int32_t* __restrict__ out_tokens, int32_t* __restrict__ diverge_depth,
                   int* err) {
  pdl_begin();
  const int lane = threadIdx.x & 31;
  const int wib = threadIdx.x >> 5;
  const int b = blockIdx.x * kWarpsPerCta + wib;
  if (b >= batch) return;
  const int W = (n_max + 63) >> 6;
  const int64_t nb = (int64_t)b * n_max;
  int n = n_nodes[b];
  if (n < 1 || n > n_max) {
    if (lane == 0) flag(err, CURE_DEVERR_NODES);
    n = max(1, min(n, n_max));
  }

  // verified bits (the root counts as verified)
  __shared__ uint64_t s_ver[kWarpsPerCta][4];
  if (lane < 4) s_ver[wib][lane] = 0ull;
  __syncwarp();
  for (int j = lane; j < n; j += 32) {
    bool v = (j == 0);
    if (j > 0) {
      const int pj = parent[nb + j];
      if (pj >= 0 && pj < j) v = tok[nb + j] == targ[nb + pj];
      else flag(err, CURE_DEVERR_NODES);
    }
    if (v) atomicOr(reinterpret_cast<unsigned long long*>(&s_ver[wib][j >> 6]),
                    (unsigned long long)(1ull << (j & 63)));
  }
  __syncwarp();

  // deepest accepted node, lowest index on ties
  int bestkey = -1;
  for (int j = lane; j < n; j += 32) {
    bool ok = true;
    for (int w = 0; w < W; ++w) ok &= (anc[(nb + j) * W + w] & ~s_ver[wib][w]) == 0ull;
    if (ok) {
      const int d = depth[nb + j];
      if (d < 0 || d > block) {
        flag(err, CURE_DEVERR_NODES);
      } else {
        bestkey = max(bestkey, (d << 16) | (0xffff - j));
      }
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) bestkey = max(bestkey, __shfl_xor_sync(kFull, bestkey, off));
  if (bestkey < 0) {
    // no node qualified: only a corrupt root depth gets here (the root is
    // always accepted); fall back to the root so every store below stays in
    // the sequence's own rows
    if (lane == 0) {
      flag(err, CURE_DEVERR_NODES);
      path_nodes[(int64_t)b * (block + 2)] = 0;
    }
    bestkey = 0xffff;
  }
  const int best = 0xffff - (bestkey & 0xffff);
  const int a = bestkey >> 16;

  // path by depth, emitted tokens, divergence depth
  const int P = block + 2;
  int div = INT_MAX;
  for (int t = lane; t < P; t += 32) {
    if (t > a) {
      path_nodes[(int64_t)b * P + t] = -1;
      out_tokens[(int64_t)b * P + t] = -1;
    }
  }
  __syncwarp();
  for (int j = lane; j < n; j += 32) {
    if ((anc[(nb + best) * W + (j >> 6)] >> (j & 63)) & 1ull) {
      const int d = depth[nb + j];
      if (d < 0 || d > a) {
        flag(err, CURE_DEVERR_NODES);
        continue;
      }
      path_nodes[(int64_t)b * P + d] = j;
      if (d >= 1) out_tokens[(int64_t)b * P + d - 1] = tok[nb + j];
      if (j > block) div = min(div, d);
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) div = min(div, __shfl_xor_sync(kFull, div, off));
  if (lane == 0) {
    out_tokens[(int64_t)b * P + a] = targ[nb + best];
    accept_len[b] = a;
    best_node[b] = best;
    diverge_depth[b] = (div == INT_MAX) ? -1 : div;
  }
}

}  // namespace

cudaError_t launch_build_tree(const cure_tree_params& p, const int32_t* top_ids,
                              const float* margin, const int32_t* root_tok,
                              const int32_t* cache_len, const int32_t* redraft, int32_t* n_nodes,
                              int32_t* tok, int32_t* pos, int32_t* parent, int32_t* depth,
                              uint64_t* anc, int32_t* ufp_pos, int32_t* n_ufp, int* err,
                              cudaStream_t s) {
  (void)err;
  if (p.batch == 0) return cudaSuccess;
  const int grid = (p.batch + kWarpsPerCta - 1) / kWarpsPerCta;
  return launch_pdl(build_tree_kernel, dim3(grid), dim3(32 * kWarpsPerCta), 0, s, p, top_ids, margin,
                    root_tok, cache_len, redraft, n_nodes, tok, pos, parent, depth, anc, ufp_pos,
                    n_ufp);
}

cudaError_t launch_accept_walk(int batch, int n_max, int block, const int32_t* n_nodes,
                               const int32_t* tok, const int32_t* parent, const int32_t* depth,
                               const uint64_t* anc, const int32_t* targ, int32_t* accept_len,
                               int32_t* best_node, int32_t* path_nodes, int32_t* out_tokens,
                               int32_t* diverge_depth, int* err, cudaStream_t s) {
  if (batch == 0) return cudaSuccess;
  const int grid = (batch + kWarpsPerCta - 1) / kWarpsPerCta;
  return launch_pdl(accept_walk_kernel, dim3(grid), dim3(32 * kWarpsPerCta), 0, s, batch, n_max, block,
                    n_nodes, tok, parent, depth, anc, targ, accept_len, best_node, path_nodes,
                    out_tokens, diverge_depth, err);
}

}  // namespace cure
