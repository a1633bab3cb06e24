// Stage 1 (Sec. 3.3, Eq. 2) and the target argmax of stage 5 (Sec. 3.5, greedy
// decoding): one streaming pass over bf16 vocabulary rows.
//
// A row is scanned by one CTA, or split over a thread-block cluster of S CTAs
// when there are too few rows to fill the GPU.  Every thread streams 16-byte
// vectors (8 bf16 logits) with non-allocating loads, the next vectors loaded
// while the current ones are consumed, and keeps a register top-k list
// ordered by (value desc, id asc) and, for stage 1, an online base-2
// log-sum-exp (running max + rescaled sum).  A logit enters a list only if it
// reaches the warp's threshold: the largest k-th best value over the lanes,
// below which nothing can be in the row's top k (one lane already holds k
// values at or above it).  Lists and sums are merged by warp shuffles, then
// across the warps of the CTA through shared memory, then across the cluster
// through distributed shared memory by the CTA of rank 0, which writes the
// row's result.  No global scratch is used.
#include <cooperative_groups.h>
#include <float.h>
#include <limits.h>

#include "common.cuh"

namespace cg = cooperative_groups;

namespace cure {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kUnroll = 2;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

__device__ __forceinline__ bool better(float a, int ia, float b, int ib) {
  return a > b || (a == b && ia < ib);
}

template <int KT>
struct TopK {
  float v[KT];
  int i[KT];
  __device__ __forceinline__ void init() {
#pragma unroll
    for (int k = 0; k < KT; ++k) {
      v[k] = -INFINITY;
      i[k] = INT_MAX;
    }
  }
  __device__ __forceinline__ void insert(float x, int ix) {
    if (!better(x, ix, v[KT - 1], i[KT - 1])) return;
    bool placed = false;
#pragma unroll
    for (int k = KT - 1; k > 0; --k) {
      const bool up = better(x, ix, v[k - 1], i[k - 1]);
      if (!placed) {
        if (up) {
          v[k] = v[k - 1];
          i[k] = i[k - 1];
        } else {
          v[k] = x;
          i[k] = ix;
          placed = true;
        }
      }
    }
    if (!placed) {
      v[0] = x;
      i[0] = ix;
    }
  }
  __device__ __forceinline__ void merge_shfl(int offset) {
    float pv[KT];
    int pi[KT];
#pragma unroll
    for (int k = 0; k < KT; ++k) {
      pv[k] = __shfl_xor_sync(0xffffffffu, v[k], offset);
      pi[k] = __shfl_xor_sync(0xffffffffu, i[k], offset);
    }
#pragma unroll
    for (int k = 0; k < KT; ++k) insert(pv[k], pi[k]);
  }
};

// Base-2 log-sum-exp state: sum of 2^(x*log2e - mb).
struct Lse2 {
  float m;   // natural-log running max (for the rescale test)
  float mb;  // m * log2e as used in the exponents
  float s;
};

__device__ __forceinline__ void lse_merge(Lse2& a, float mb2, float s2) {
  const float m = fmaxf(a.mb, mb2);
  if (m == -INFINITY) return;
  a.s = a.s * ex2(a.mb - m) + s2 * ex2(mb2 - m);
  a.mb = m;
}

template <int KT, bool LSE>
struct Part {
  float v[KT];
  int i[KT];
  float mb, s;
};

template <int KT, bool LSE>
__device__ __forceinline__ void consume8(const uint4& r, int idx, TopK<KT>& tk, Lse2& ls, float thr) {
  float x[8];
  x[0] = bf16_lo(r.x); x[1] = bf16_hi(r.x);
  x[2] = bf16_lo(r.y); x[3] = bf16_hi(r.y);
  x[4] = bf16_lo(r.z); x[5] = bf16_hi(r.z);
  x[6] = bf16_lo(r.w); x[7] = bf16_hi(r.w);
  const float gm = fmaxf(fmaxf(fmaxf(x[0], x[1]), fmaxf(x[2], x[3])),
                         fmaxf(fmaxf(x[4], x[5]), fmaxf(x[6], x[7])));
  if constexpr (LSE) {
    if (gm > ls.m) {
      const float nb = gm * kLog2e;
      ls.s *= ex2(ls.mb - nb);
      ls.m = gm;
      ls.mb = nb;
    }
    if (ls.m != -INFINITY) {
      float e2[4];
#pragma unroll
      for (int e = 0; e < 4; ++e)
        e2[e] = ex2(fmaf(x[e], kLog2e, -ls.mb)) + ex2(fmaf(x[e + 4], kLog2e, -ls.mb));
      ls.s += (e2[0] + e2[1]) + (e2[2] + e2[3]);
    }
  }
  if (gm >= thr) {
#pragma unroll
    for (int e = 0; e < 8; ++e)
      if (x[e] >= thr) tk.insert(x[e], idx + e);
  }
}

template <int KT, bool LSE>
__device__ __forceinline__ void consume1(float x, int idx, TopK<KT>& tk, Lse2& ls) {
  if constexpr (LSE) {
    if (x > ls.m) {
      const float nb = x * kLog2e;
      ls.s *= ex2(ls.mb - nb);
      ls.m = x;
      ls.mb = nb;
    }
    if (ls.m != -INFINITY) ls.s += ex2(fmaf(x, kLog2e, -ls.mb));
  }
  tk.insert(x, idx);
}

// grid (S, rows) with cluster (S, 1, 1).  TARGET: rows are (b, j) of a
// [batch][n_max] tree and only j < n_nodes[b] are scanned.
template <int KT, bool LSE, bool TARGET>
__global__ void __launch_bounds__(kThreads)
vocab_scan_kernel(const uint16_t* __restrict__ logits, int vocab, int k_out, int n_max,
                  const int32_t* __restrict__ n_nodes, int32_t* __restrict__ top_ids,
                  float* __restrict__ top_vals, float* __restrict__ margin,
                  float* __restrict__ logp1) {
  const int64_t row = blockIdx.y;
  const int S = gridDim.x;
  const int c = blockIdx.x;  // rank within the cluster
  const int tid = threadIdx.x;

  if constexpr (TARGET) {
    const int b = (int)(row / n_max);
    const int j = (int)(row % n_max);
    if (j >= n_nodes[b]) {  // uniform over the cluster: every CTA leaves
      if (c == 0 && tid == 0) top_ids[row] = -1;
      return;
    }
  }

  const uint16_t* rowp = logits + row * (int64_t)vocab;
  const int mis = (int)((reinterpret_cast<uintptr_t>(rowp) >> 1) & 7);
  const int a0 = min((8 - mis) & 7, vocab);
  const int nvec = (vocab - a0) >> 3;
  const int tail0 = a0 + (nvec << 3);
  const int per = (nvec + S - 1) / S;
  const int vb = c * per;
  const int ve = min(nvec, vb + per);

  TopK<KT> tk;
  tk.init();
  Lse2 ls{-INFINITY, -INFINITY, 0.f};

  if (c == 0 && tid < a0) consume1<KT, LSE>(bf16_lo(rowp[tid]), tid, tk, ls);
  if (c == S - 1 && tid < vocab - tail0)
    consume1<KT, LSE>(bf16_lo(rowp[tail0 + tid]), tail0 + tid, tk, ls);

  const uint4* vp = reinterpret_cast<const uint4*>(rowp + a0);
  // the trip count is uniform over the warp, so that every lane takes part in
  // the threshold exchange
  const int lane = tid & 31;
  const int wb0 = vb + (tid & ~31);
  uint4 r[kUnroll];
#pragma unroll
  for (int u = 0; u < kUnroll; ++u) {
    const int vi = wb0 + lane + u * kThreads;
    if (vi < ve) r[u] = ld_stream(vp + vi);
  }
  float thr = tk.v[KT - 1];
  for (int wb = wb0; wb < ve; wb += kUnroll * kThreads) {
    uint4 nx[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int vi = wb + lane + (kUnroll + u) * kThreads;
      if (vi < ve) nx[u] = ld_stream(vp + vi);
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int vi = wb + lane + u * kThreads;
      if (vi < ve) consume8<KT, LSE>(r[u], a0 + (vi << 3), tk, ls, thr);
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) r[u] = nx[u];
    float th = tk.v[KT - 1];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) th = fmaxf(th, __shfl_xor_sync(0xffffffffu, th, off));
    thr = th;
  }

  // ---- warp merge
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    tk.merge_shfl(off);
    if constexpr (LSE) {
      const float mb2 = __shfl_xor_sync(0xffffffffu, ls.mb, off);
      const float s2 = __shfl_xor_sync(0xffffffffu, ls.s, off);
      lse_merge(ls, mb2, s2);
    }
  }

  // ---- CTA merge
  __shared__ Part<KT, LSE> warp_part[kWarps];
  __shared__ Part<KT, LSE> cta_part;
  const int warp = tid >> 5;
  if (lane == 0) {
#pragma unroll
    for (int k = 0; k < KT; ++k) {
      warp_part[warp].v[k] = tk.v[k];
      warp_part[warp].i[k] = tk.i[k];
    }
    warp_part[warp].mb = ls.mb;
    warp_part[warp].s = ls.s;
  }
  __syncthreads();
  if (warp == 0) {
    tk.init();
    ls.mb = -INFINITY;
    ls.s = 0.f;
    if (lane < kWarps) {
#pragma unroll
      for (int k = 0; k < KT; ++k) {
        tk.v[k] = warp_part[lane].v[k];
        tk.i[k] = warp_part[lane].i[k];
      }
      ls.mb = warp_part[lane].mb;
      ls.s = warp_part[lane].s;
    }
#pragma unroll
    for (int off = kWarps / 2; off > 0; off >>= 1) {
      tk.merge_shfl(off);
      if constexpr (LSE) {
        const float mb2 = __shfl_xor_sync(0xffffffffu, ls.mb, off);
        const float s2 = __shfl_xor_sync(0xffffffffu, ls.s, off);
        lse_merge(ls, mb2, s2);
      }
    }
    if (lane == 0) {
#pragma unroll
      for (int k = 0; k < KT; ++k) {
        cta_part.v[k] = tk.v[k];
        cta_part.i[k] = tk.i[k];
      }
      cta_part.mb = ls.mb;
      cta_part.s = ls.s;
    }
  }

  // ---- cluster merge (rank 0 reads its peers' results through DSMEM)
  if (S > 1) {
    cg::cluster_group cluster = cg::this_cluster();
    cluster.sync();
    if (c == 0 && tid == 0) {
      for (int r = 1; r < S; ++r) {
        const Part<KT, LSE>* pp = cluster.map_shared_rank(&cta_part, r);
#pragma unroll
        for (int k = 0; k < KT; ++k) tk.insert(pp->v[k], pp->i[k]);
        if constexpr (LSE) lse_merge(ls, pp->mb, pp->s);
      }
    }
    cluster.sync();
  } else {
    __syncthreads();
  }

  if (c == 0 && tid == 0) {
    if constexpr (TARGET) {
      top_ids[row] = tk.i[0];
    } else {
#pragma unroll
      for (int k = 0; k < KT; ++k) {
        if (k < k_out) {
          top_ids[row * k_out + k] = tk.i[k];
          top_vals[row * k_out + k] = tk.v[k];
        }
      }
      if (margin) margin[row] = tk.v[0] - tk.v[1];
      if constexpr (LSE) {
        if (logp1) {
          const float lse = (ls.mb + log2f(ls.s)) * kLn2;
          logp1[row] = tk.v[0] - lse;
        }
      }
    }
  }
}

// One CTA per row once the rows alone give every SM two CTAs (merging a
// split row costs more than it gains there); else split rows over a cluster
// of up to 8 CTAs, keeping at least two vectors per thread in each.
int pick_split(int64_t rows, int vocab) {
  const int nvec = vocab / 8;
  if (rows >= 2LL * num_sms()) return 1;
  int s = (int)((4LL * num_sms() + rows - 1) / rows);
  s = max(1, min(s, 8));
  while (s > 1 && nvec / s < 2 * kThreads) --s;
  return s;
}

template <int KT, bool LSE, bool TARGET>
cudaError_t launch_scan(const uint16_t* logits, int64_t rows, int vocab, int k_out, int n_max,
                        const int32_t* n_nodes, int32_t* top_ids, float* top_vals, float* margin,
                        float* logp1, cudaStream_t s) {
  const int S = pick_split(rows, vocab);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(S, (unsigned)rows, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = S;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, vocab_scan_kernel<KT, LSE, TARGET>, logits, vocab, k_out,
                            n_max, n_nodes, top_ids, top_vals, margin, logp1);
}

}  // namespace

cudaError_t launch_score(const uint16_t* logits, int64_t rows, int vocab, int topk,
                         int32_t* top_ids, float* top_vals, float* margin, float* logp1,
                         cudaStream_t s) {
  if (rows == 0) return cudaSuccess;
  switch (topk) {
    case 2: return launch_scan<2, true, false>(logits, rows, vocab, topk, 0, nullptr, top_ids, top_vals, margin, logp1, s);
    case 3: return launch_scan<3, true, false>(logits, rows, vocab, topk, 0, nullptr, top_ids, top_vals, margin, logp1, s);
    case 4: return launch_scan<4, true, false>(logits, rows, vocab, topk, 0, nullptr, top_ids, top_vals, margin, logp1, s);
    default: return launch_scan<8, true, false>(logits, rows, vocab, topk, 0, nullptr, top_ids, top_vals, margin, logp1, s);
  }
}

cudaError_t launch_target_argmax(const uint16_t* logits, int batch, int n_max, int vocab,
                                 const int32_t* n_nodes, int32_t* targ, cudaStream_t s) {
  const int64_t rows = (int64_t)batch * n_max;
  if (rows == 0) return cudaSuccess;
  return launch_scan<1, false, true>(logits, rows, vocab, 1, n_max, n_nodes, targ, nullptr,
                                     nullptr, nullptr, s);
}

}  // namespace cure
