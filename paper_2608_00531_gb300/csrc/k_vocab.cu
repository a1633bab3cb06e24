// Stage 1 (Sec. 3.3, Eq. 2) and the target argmax of stage 5 (Sec. 3.5, greedy
// decoding): one streaming pass over bf16 vocabulary rows.
//
// A row is scanned by one CTA, or split over a thread-block cluster of S CTAs
// when there are too few rows to fill the GPU.  Each thread keeps a register
// top-k list ordered by (value desc, id asc) and, for stage 1, an online
// base-2 log-sum-exp (running max + rescaled sum).  A logit enters a list only
// if it reaches the warp's threshold: the largest k-th best value over the
// lanes, below which nothing can be in the row's top k (one lane already holds
// k values at or above it).  Lists and sums are merged by warp shuffles, then
// across the warps of the CTA through shared memory, then across the cluster
// through distributed shared memory by the CTA of rank 0, which writes the
// row's result.  No global scratch is used.  Two ways to feed the lanes:
//  - register streaming (stage 1): every thread loads 16-byte vectors (8 bf16
//    logits) with non-allocating loads, the next vectors loaded while the
//    current ones are consumed; the log-sum-exp work per logit wants the many
//    resident warps this allows;
//  - a ring (the target argmax): a producer warp streams the CTA's part of
//    the row into three 8 KiB shared-memory stages with bulk copies
//    (cp.async.bulk, completing on an mbarrier per stage), so the bytes in
//    flight do not depend on registers; four consumer warps read their
//    vectors from it and free each stage once they hold them.  Ring waits
//    are bounded: on expiry a CTA flags CURE_DEVERR_TIMEOUT, lets its copies
//    land and still takes part in the merge.
#include <cooperative_groups.h>
#include <float.h>
#include <limits.h>

#include <type_traits>

#include "common.cuh"
#include "tc_ptx.cuh"

namespace cg = cooperative_groups;

namespace cure {
namespace {

constexpr int kThreads = 128;              // consumer threads (4 warps)
constexpr int kWarps = kThreads / 32;
constexpr int kCtaThreads = kThreads + 32; // plus one producer warp
constexpr int kUnroll = 2;                 // vectors per consumer lane per step (ring-fed scan)
constexpr int kChunkVec = 512;             // 16-byte vectors per ring stage (8 KiB)
constexpr int kStages = 3;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

using tc::smem_u32;
using tc::wait_bounded;

// One bulk copy of `bytes` (a multiple of 16) from global memory into this
// CTA's shared memory, completing on `bar`.
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}
__device__ __forceinline__ uint4 ld_shared_v4(uint32_t a) {
  uint4 r;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w) : "r"(a));
  return r;
}

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

__device__ __forceinline__ float max3f(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// Pairs of floats in one 64-bit register pair, for the packed f32x2
// arithmetic of sm_100 and later (two lanes of work per instruction).
__device__ __forceinline__ uint64_t f2_pack(float a, float b) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
  return r;
}
__device__ __forceinline__ void f2_unpack(uint64_t r, float& a, float& b) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(r));
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ uint64_t f2_mul(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
  return v;
}

// A lower bound on the warp's k-th best value, the same in every lane: the
// largest lane-local k-th best (that lane holds k values at or above it) and
// the k-th largest of the lane maxima (k lanes each hold one value at or
// above it; a lane that ties the current maximum drops out with it, which can
// only lower the bound).
template <int KT>
__device__ __forceinline__ float warp_kth(const TopK<KT>& tk) {
  float t = warp_max(tk.v[KT - 1]);
  float m = tk.v[0];
#pragma unroll
  for (int k = 0; k < KT; ++k) {
    const float mk = warp_max(m);
    if (k == KT - 1) t = fmaxf(t, mk);
    if (m == mk) m = -INFINITY;
  }
  return t;
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

// Ring-fed variant (used for the target argmax, whose light work per logit
// leaves the loads in flight as the limit).  grid (S, rows) with cluster
// (S, 1, 1).  TARGET: rows are (b, j) of a [batch][n_max] tree and only
// j < n_nodes[b] are scanned.
template <int KT, bool LSE, bool TARGET, int CW>
__global__ void __launch_bounds__(CW * 32 + 32, CW == 4 ? 6 : 4)
vocab_ring_kernel(const uint16_t* __restrict__ logits, int vocab, int k_out, int n_max,
                  const int32_t* __restrict__ n_nodes, int32_t* __restrict__ top_ids,
                  float* __restrict__ top_vals, float* __restrict__ margin,
                  float* __restrict__ logp1, int* err) {
  pdl_begin();
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

  const uint4* vp = reinterpret_cast<const uint4*>(rowp + a0);  // 16-byte aligned
  // The CTA's vectors [vb, ve) stream through a ring of kStages shared-memory
  // stages of kChunkVec vectors, filled by bulk copies that the producer warp
  // issues (bytes in flight do not depend on registers); each consumer warp
  // frees a stage once it has its vectors in registers.
  __shared__ __align__(128) uint4 ring[kStages][kChunkVec];
  __shared__ __align__(8) uint64_t full_bar[kStages], empty_bar[kStages];
  __shared__ int abort_s;
  volatile int* abort_flag = &abort_s;
  const int lane = tid & 31, warp = tid >> 5;
  const int nloc = max(0, ve - vb);
  const int nchunks = (nloc + kChunkVec - 1) / kChunkVec;
  if (tid == 0) {
    for (int st = 0; st < kStages; ++st) {
      tc::mbar_init(smem_u32(&full_bar[st]), 1);
      tc::mbar_init(smem_u32(&empty_bar[st]), CW);
    }
    abort_s = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  float thr = warp_kth(tk);
  float mbw = -INFINITY;
  uint64_t sacc = f2_pack(0.f, 0.f);  // two lane sums, as one f32x2 pair
  // The threshold and the log-sum-exp base are warp-wide values that all
  // lanes take part in (the trip count is uniform over the warp):
  //  - thr: the k-th best value over the warp's lists.  A logit below it
  //    cannot be in the row's top k (the warp already holds k values at or
  //    above it), so lists change only in the rare steps with a logit at or
  //    above it, after which thr is recomputed.
  //  - mbw: base-2 exponent base of the lane sums (sum of 2^(x log2e - mbw));
  //    raised, with the sums rescaled, only when some lane sees a logit more
  //    than 2^8 above it, so the sums stay below 2^8 per term and the rescale
  //    is rare and uniform.
  // One step: kUnroll vectors per lane, r[u] at vector index gi[u] (vb-based);
  // FULL when every lane's vectors are in range, so that no check is needed.
  auto step = [&](const uint4 (&r)[kUnroll], const int (&gi)[kUnroll], int lim, bool first, auto full_tag) {
    constexpr bool FULL = decltype(full_tag)::value;
    uint64_t xp[kUnroll][4];  // (lo, hi) logit pairs of each 32-bit word
    float gmv[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const uint32_t w[4] = {r[u].x, r[u].y, r[u].z, r[u].w};
      float lo[4], hi[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        lo[q] = bf16_lo(w[q]);
        hi[q] = bf16_hi(w[q]);
        xp[u][q] = f2_pack(lo[q], hi[q]);
      }
      const float g = fmaxf(max3f(lo[0], hi[0], lo[1]), max3f(max3f(hi[1], lo[2], hi[2]), lo[3], hi[3]));
      gmv[u] = (FULL || gi[u] < lim) ? g : -INFINITY;
    }
    if constexpr (LSE) {
      float gl = gmv[0];
#pragma unroll
      for (int u = 1; u < kUnroll; ++u) gl = fmaxf(gl, gmv[u]);
      if (__any_sync(0xffffffffu, gl * kLog2e > mbw + 8.f)) {
        const float nb = warp_max(gl) * kLog2e;
        if (mbw != -INFINITY) {
          const float sc = ex2(mbw - nb);
          sacc = f2_mul(sacc, f2_pack(sc, sc));
        }
        mbw = nb;
      }
      if (mbw != -INFINITY) {
        const uint64_t l2 = f2_pack(kLog2e, kLog2e), nb2 = f2_pack(-mbw, -mbw);
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
          if (FULL || gi[u] < lim) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              float a, b;
              f2_unpack(f2_fma(xp[u][q], l2, nb2), a, b);
              sacc = f2_add(sacc, f2_pack(ex2(a), ex2(b)));
            }
          }
        }
      }
    }
    if (first) {
      // first step: the k-th largest of the lanes' maxima of this step is a
      // valid threshold already (each of those maxima is in its lane's list
      // after the inserts below, or that lane holds k values above it), so
      // that a warp does not start by inserting every logit it sees
      float gl = gmv[0];
#pragma unroll
      for (int u = 1; u < kUnroll; ++u) gl = fmaxf(gl, gmv[u]);
#pragma unroll
      for (int k = 0; k < KT; ++k) {
        const float mk = warp_max(gl);
        if (k == KT - 1) thr = fmaxf(thr, mk);
        if (gl == mk) gl = -INFINITY;
      }
    }
    bool cand = false;
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) cand |= (FULL || gi[u] < lim) && gmv[u] >= thr;
    if (__any_sync(0xffffffffu, cand)) {
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        if ((FULL || gi[u] < lim) && gmv[u] >= thr) {
          const int idx = a0 + ((vb + gi[u]) << 3);
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            float a, b;
            f2_unpack(xp[u][q], a, b);
            if (a >= thr) tk.insert(a, idx + 2 * q);
            if (b >= thr) tk.insert(b, idx + 2 * q + 1);
          }
        }
      }
      thr = warp_kth(tk);
    }
  };

  if (warp == CW) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      int issued = 0;
      for (int ch = 0; ch < nchunks; ++ch, ++issued) {
        const int st = ch % kStages;
        if (ch >= kStages &&
            !wait_bounded(smem_u32(&empty_bar[st]), ((ch / kStages) & 1) ^ 1, abort_flag, err, true))
          break;
        const uint32_t bytes = (uint32_t)min(kChunkVec, nloc - ch * kChunkVec) * 16u;
        tc::mbar_arrive_expect_tx(smem_u32(&full_bar[st]), bytes);
        bulk_load(smem_u32(&ring[st][0]), vp + vb + ch * kChunkVec, bytes, smem_u32(&full_bar[st]));
      }
      // the copies in flight land before the CTA's shared memory goes away
      for (int ch = max(0, issued - kStages); ch < issued; ++ch)
        wait_bounded(smem_u32(&full_bar[ch % kStages]), (ch / kStages) & 1, abort_flag, err, false);
    }
  } else {
    // ---------------------------------------------------------------- consumers
    bool first = true;
    for (int ch = 0; ch < nchunks; ++ch) {
      const int st = ch % kStages;
      const bool ok = wait_bounded(smem_u32(&full_bar[st]), (ch / kStages) & 1, abort_flag, err, true);
      if (!__all_sync(0xffffffffu, ok)) break;
      const int cb = ch * kChunkVec;              // chunk's first vector (vb-based)
      const int lim = nloc;
      const bool full = cb + kChunkVec <= nloc;
      // the warp's two steps of this chunk: vectors warp*32 + lane + u*128,
      // u = 0..3; the stage is freed once the second step's vectors are read
      uint4 r[kUnroll];
      int gi[kUnroll];
#pragma unroll
      constexpr int kSteps = kChunkVec / (CW * 32 * kUnroll);  // steps per chunk
#pragma unroll
      for (int half = 0; half < kSteps; ++half) {
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
          const int o = warp * 32 + lane + (half * kUnroll + u) * (CW * 32);
          gi[u] = cb + o;
          if (full || gi[u] < lim) r[u] = ld_shared_v4(smem_u32(&ring[st][o]));
        }
        if (half == kSteps - 1) {
          __syncwarp();
          if (lane == 0) tc::mbar_arrive(smem_u32(&empty_bar[st]));  // this warp's vectors are in registers
        }
        if (full) step(r, gi, lim, first && half == 0, std::integral_constant<bool, true>());
        else step(r, gi, lim, first && half == 0, std::integral_constant<bool, false>());
      }
      first = false;
    }
  }
  float sa, sb2;
  f2_unpack(sacc, sa, sb2);
  const float s0 = sa, s1 = sb2;
  if constexpr (LSE) lse_merge(ls, mbw, s0 + s1);

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
  __shared__ Part<KT, LSE> warp_part[CW];
  __shared__ Part<KT, LSE> cta_part;
  if (lane == 0 && warp < CW) {
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
    if (lane < CW) {
#pragma unroll
      for (int k = 0; k < KT; ++k) {
        tk.v[k] = warp_part[lane].v[k];
        tk.i[k] = warp_part[lane].i[k];
      }
      ls.mb = warp_part[lane].mb;
      ls.s = warp_part[lane].s;
    }
#pragma unroll
    for (int off = CW / 2; off > 0; off >>= 1) {
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

// Register-streaming variant (used for stage 1, whose log-sum-exp work per
// logit wants many resident warps): every thread streams 16-byte vectors with
// non-allocating loads, the next vectors loaded while the current ones are
// consumed.  grid (S, rows) with cluster (S, 1, 1).
// Vectors per lane per step of the register-streaming scan: three 16-byte
// loads in flight per lane (70 registers, still one wave of the grid).
constexpr int kUnrollS = 3;

template <int KT, bool LSE, bool TARGET>
__global__ void __launch_bounds__(kThreads)
vocab_scan_kernel(const uint16_t* __restrict__ logits, int vocab, int k_out, int n_max,
                  const int32_t* __restrict__ n_nodes, int32_t* __restrict__ top_ids,
                  float* __restrict__ top_vals, float* __restrict__ margin,
                  float* __restrict__ logp1) {
  pdl_begin();
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
  // The trip count is uniform over the warp: the threshold and the log-sum-exp
  // base are warp-wide values that all lanes take part in.
  //  - thr: the k-th best value over the warp's lists.  A logit below it
  //    cannot be in the row's top k (the warp already holds k values at or
  //    above it), so lists change only in the rare steps with a logit at or
  //    above it, after which thr is recomputed.
  //  - mbw: base-2 exponent base of the lane sums s0 + s1 (sum of
  //    2^(x log2e - mbw)); raised, with the sums rescaled, only when some lane
  //    sees a logit more than 2^8 above it, so the sums stay below 2^8 per
  //    term and the rescale is rare and uniform.
  const int lane = tid & 31;
  const int wb0 = vb + (tid & ~31);
  uint4 r[kUnrollS];
#pragma unroll
  for (int u = 0; u < kUnrollS; ++u) {
    const int vi = wb0 + lane + u * kThreads;
    if (vi < ve) r[u] = ld_stream(vp + vi);
  }
  float thr = warp_kth(tk);
  float mbw = -INFINITY;
  uint64_t sacc = f2_pack(0.f, 0.f);  // two lane sums, as one f32x2 pair
  // one step: kUnrollS vectors per lane; FULL when every lane's vectors are in
  // range (all but a warp's last step), so that no per-vector check is needed
  auto step = [&](int wb, auto full_tag) {
    constexpr bool FULL = decltype(full_tag)::value;
    uint4 nx[kUnrollS];
#pragma unroll
    for (int u = 0; u < kUnrollS; ++u) {
      const int vi = wb + lane + (kUnrollS + u) * kThreads;
      if (vi < ve) nx[u] = ld_stream(vp + vi);
    }
    uint64_t xp[kUnrollS][4];  // (lo, hi) logit pairs of each 32-bit word
    float gmv[kUnrollS];
#pragma unroll
    for (int u = 0; u < kUnrollS; ++u) {
      const uint32_t w[4] = {r[u].x, r[u].y, r[u].z, r[u].w};
      float lo[4], hi[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        lo[q] = bf16_lo(w[q]);
        hi[q] = bf16_hi(w[q]);
        xp[u][q] = f2_pack(lo[q], hi[q]);
      }
      const float g = fmaxf(max3f(lo[0], hi[0], lo[1]), max3f(max3f(hi[1], lo[2], hi[2]), lo[3], hi[3]));
      gmv[u] = (FULL || wb + lane + u * kThreads < ve) ? g : -INFINITY;
    }
    if constexpr (LSE) {
      float gl = gmv[0];
#pragma unroll
      for (int u = 1; u < kUnrollS; ++u) gl = fmaxf(gl, gmv[u]);
      if (__any_sync(0xffffffffu, gl * kLog2e > mbw + 8.f)) {
        const float nb = warp_max(gl) * kLog2e;
        if (mbw != -INFINITY) {
          const float sc = ex2(mbw - nb);
          sacc = f2_mul(sacc, f2_pack(sc, sc));
        }
        mbw = nb;
      }
      if (mbw != -INFINITY) {
        const uint64_t l2 = f2_pack(kLog2e, kLog2e), nb2 = f2_pack(-mbw, -mbw);
#pragma unroll
        for (int u = 0; u < kUnrollS; ++u) {
          if (FULL || wb + lane + u * kThreads < ve) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              float a, b;
              f2_unpack(f2_fma(xp[u][q], l2, nb2), a, b);
              sacc = f2_add(sacc, f2_pack(ex2(a), ex2(b)));
            }
          }
        }
      }
    }
    if (wb == wb0) {
      // first step: the k-th largest of the lanes' maxima of this step is a
      // valid threshold already (each of those maxima is in its lane's list
      // after the inserts below, or that lane holds k values above it), so
      // that a warp does not start by inserting every logit it sees
      float gl = gmv[0];
#pragma unroll
      for (int u = 1; u < kUnrollS; ++u) gl = fmaxf(gl, gmv[u]);
#pragma unroll
      for (int k = 0; k < KT; ++k) {
        const float mk = warp_max(gl);
        if (k == KT - 1) thr = fmaxf(thr, mk);
        if (gl == mk) gl = -INFINITY;
      }
    }
    bool cand = false;
#pragma unroll
    for (int u = 0; u < kUnrollS; ++u) cand |= (FULL || wb + lane + u * kThreads < ve) && gmv[u] >= thr;
    if (__any_sync(0xffffffffu, cand)) {
#pragma unroll
      for (int u = 0; u < kUnrollS; ++u) {
        if ((FULL || wb + lane + u * kThreads < ve) && gmv[u] >= thr) {
          const int idx = a0 + ((wb + lane + u * kThreads) << 3);
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            float a, b;
            f2_unpack(xp[u][q], a, b);
            if (a >= thr) tk.insert(a, idx + 2 * q);
            if (b >= thr) tk.insert(b, idx + 2 * q + 1);
          }
        }
      }
      thr = warp_kth(tk);
    }
#pragma unroll
    for (int u = 0; u < kUnrollS; ++u) r[u] = nx[u];
  };
  int wb = wb0;
  for (; wb + 31 + (kUnrollS - 1) * kThreads < ve; wb += kUnrollS * kThreads)
    step(wb, std::integral_constant<bool, true>());
  for (; wb < ve; wb += kUnrollS * kThreads) step(wb, std::integral_constant<bool, false>());
  float sa, sb2;
  f2_unpack(sacc, sa, sb2);
  const float s0 = sa, s1 = sb2;
  if constexpr (LSE) lse_merge(ls, mbw, s0 + s1);

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

// One CTA per row once the rows alone give every SM six CTAs (24 warps, the
// occupancy the scan needs to hide its load and exponential latencies); else
// split rows over a cluster of up to 8 CTAs, keeping at least two vectors per
// thread in each.
int pick_split_lsu(int64_t rows, int vocab) {
  const int nvec = vocab / 8;
  if (rows >= 6LL * num_sms()) return 1;
  int s = (int)((6LL * num_sms() + rows - 1) / rows);
  s = max(1, min(s, 8));
  while (s > 1 && nvec / s < 2 * kThreads) --s;
  return s;
}

// The grid is kept to one wave of at most six CTAs per SM (the occupancy the
// kernel is built for): one CTA per row when the rows alone reach that,
// else rows split over a cluster of up to 8 CTAs, each keeping at least two
// vectors per consumer thread.  Bytes in flight come from each CTA's ring, so
// a CTA that streams a whole row keeps the SM as busy as several would.
int pick_split_ring(int64_t rows, int vocab, int per_sm) {
  const int nvec = vocab / 8;
  const int64_t slots = (int64_t)per_sm * num_sms();
  if (rows >= slots) return 1;
  int s = (int)(slots / rows);
  s = max(1, min(s, 8));
  while (s > 1 && nvec / s < 2 * kThreads) --s;
  return s;
}

template <int KT, bool LSE, bool TARGET, bool RING, int CW = 4>
cudaError_t launch_scan(const uint16_t* logits, int64_t rows, int vocab, int k_out, int n_max,
                        const int32_t* n_nodes, int32_t* top_ids, float* top_vals, float* margin,
                        float* logp1, cudaStream_t s) {
  const int S = RING ? pick_split_ring(rows, vocab, CW == 4 ? 6 : 4) : pick_split_lsu(rows, vocab);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(S, (unsigned)rows, 1);
  cfg.blockDim = dim3(RING ? CW * 32 + 32 : kThreads, 1, 1);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = S;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // see pdl_begin()
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  if constexpr (RING)
    return cudaLaunchKernelEx(&cfg, vocab_ring_kernel<KT, LSE, TARGET, CW>, logits, vocab, k_out, n_max, n_nodes,
                              top_ids, top_vals, margin, logp1, device_error_word());
  else
    return cudaLaunchKernelEx(&cfg, vocab_scan_kernel<KT, LSE, TARGET>, logits, vocab, k_out, n_max, n_nodes,
                              top_ids, top_vals, margin, logp1);
}

}  // namespace

cudaError_t launch_score(const uint16_t* logits, int64_t rows, int vocab, int topk,
                         int32_t* top_ids, float* top_vals, float* margin, float* logp1,
                         cudaStream_t s) {
  if (rows == 0) return cudaSuccess;
  switch (topk) {
    case 2: return launch_scan<2, true, false, false>(logits, rows, vocab, topk, 0, nullptr, top_ids, top_vals, margin, logp1, s);
    case 3: return launch_scan<3, true, false, false>(logits, rows, vocab, topk, 0, nullptr, top_ids, top_vals, margin, logp1, s);
    case 4: return launch_scan<4, true, false, false>(logits, rows, vocab, topk, 0, nullptr, top_ids, top_vals, margin, logp1, s);
    default: return launch_scan<8, true, false, false>(logits, rows, vocab, topk, 0, nullptr, top_ids, top_vals, margin, logp1, s);
  }
}

cudaError_t launch_target_argmax(const uint16_t* logits, int batch, int n_max, int vocab,
                                 const int32_t* n_nodes, int32_t* targ, cudaStream_t s) {
  const int64_t rows = (int64_t)batch * n_max;
  if (rows == 0) return cudaSuccess;
  return launch_scan<1, false, true, true>(logits, rows, vocab, 1, n_max, n_nodes, targ, nullptr,
                                     nullptr, nullptr, s);
}

}  // namespace cure
