// Stage 4: tree-masked GQA attention (Sec. 3.2 / 3.4 / 3.5: the target
// verifies every path of the repair tree in one pass with Tree Attention).
//
// Decomposition.  For sequence b and kv head h the query rows are the
// (node j, group head g) pairs, r = j * G + g, so all G query heads that share
// a kv head read each K/V tile once.  Rows are cut into blocks of 128 (one CTA
// each); the cache keys 0..L_b-1 are cut into splits of `chunk` keys (split-KV
// flash decoding); the split that holds the last cache key also takes the
// tree keys, masked per row by the node's ancestor bits.  Each CTA writes a
// partial (normalised output, base-2 log-sum-exp) per row; a reduce kernel
// merges the splits and writes bf16.
//
// This version computes QK^T and PV with warp-level bf16 tensor-core MMAs
// (16 query rows per warp, 64-key tiles double-buffered through shared memory
// with cp.async) and keeps the online softmax in registers.
#include <cuda_bf16.h>

#include <algorithm>
#include <atomic>

#include "common.cuh"

namespace cure {
namespace {

constexpr int D = 128;
constexpr int kWarps = 8;
constexpr int kThreads = 32 * kWarps;
constexpr int kRowsCta = 16 * kWarps;  // 128
constexpr int kKeys = 64;              // keys per tile
constexpr int kLd = D + 8;             // smem row stride in bf16 (272 B): conflict-free ldmatrix
constexpr int kSmemBytes = (kRowsCta + 4 * kKeys) * kLd * 2;
constexpr float kLog2e = 1.4426950408889634f;

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

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
  const int n = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(n));
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;"); }
template <int N>
__device__ __forceinline__ void cp_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N));
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1,
                                          uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void mma16816(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__global__ void __launch_bounds__(kThreads, 1) tree_attn_mma_kernel(AttnArgs A) {
  extern __shared__ __align__(128) uint16_t smem[];
  uint16_t* Qs = smem;
  uint16_t* Ks = Qs + kRowsCta * kLd;  // [2][kKeys][kLd]
  uint16_t* Vs = Ks + 2 * kKeys * kLd;

  const int rb = blockIdx.x;
  const int split = blockIdx.y;
  const int Hkv = A.kv.heads_kv;
  const int b = blockIdx.z / Hkv;
  const int h = blockIdx.z % Hkv;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  int L = A.cache_len[b];
  int n = A.n_nodes[b];
  if (L < 0 || L > A.cap || n < 1 || n > A.n_max) {
    if (tid == 0) flag(A.err, (L < 0 || L > A.cap) ? CURE_DEVERR_SLOT : CURE_DEVERR_NODES);
    L = max(0, min(L, A.cap));
    n = max(1, min(n, A.n_max));
  }
  const int rows_valid = n * A.G;
  const int r0 = rb * kRowsCta;
  if (r0 >= rows_valid) return;
  const int nsplit = max(1, (L + A.chunk - 1) / A.chunk);
  if (split >= nsplit) return;
  const int key_beg = split * A.chunk;
  const int key_end = min(L, key_beg + A.chunk);
  const bool has_tree = split == nsplit - 1;
  const int n_cache_tiles = (key_end - key_beg + kKeys - 1) / kKeys;
  const int n_tiles = n_cache_tiles + (has_tree ? (n + kKeys - 1) / kKeys : 0);

  const int64_t kv_row = (int64_t)Hkv * D;  // elements between consecutive tokens
  // ---- Q rows of this block
  for (int c = tid; c < kRowsCta * (D / 8); c += kThreads) {
    const int row = c >> 4, ch = c & 15;
    const int r = r0 + row;
    const bool v = r < rows_valid;
    const int j = v ? r / A.G : 0, g = v ? r % A.G : 0;
    const uint16_t* src = A.q + (((int64_t)b * A.n_max + j) * A.heads_q + h * A.G + g) * D + ch * 8;
    cp_async16(smem_u32(Qs + row * kLd + ch * 8), v ? src : A.q, v);
  }

  auto load_tile = [&](int i, int stage) {
    uint16_t* ks = Ks + stage * kKeys * kLd;
    uint16_t* vs = Vs + stage * kKeys * kLd;
    for (int c = tid; c < kKeys * (D / 8); c += kThreads) {
      const int row = c >> 4, ch = c & 15;
      const uint16_t* ksrc = A.kc;
      const uint16_t* vsrc = A.vc;
      bool v = false;
      if (i < n_cache_tiles) {
        const int t = key_beg + i * kKeys + row;
        if (t < key_end) {
          int64_t tok_row;
          if (A.kv.layout == 0) {
            tok_row = (int64_t)b * A.kv.max_len + t;
            v = true;
          } else {
            const int page = A.kv.block_table[(int64_t)b * A.kv.max_len + t / A.kv.page_size];
            v = page >= 0 && page < A.kv.num_pages;
            if (!v) flag(A.err, CURE_DEVERR_PAGE);
            tok_row = (int64_t)page * A.kv.page_size + t % A.kv.page_size;
          }
          if (v) {
            const int64_t off = tok_row * kv_row + (int64_t)h * D + ch * 8;
            ksrc = A.kc + off;
            vsrc = A.vc + off;
          }
        }
      } else {
        const int u = (i - n_cache_tiles) * kKeys + row;
        if (u < n) {
          const int64_t off = (((int64_t)b * A.n_max + u) * Hkv + h) * D + ch * 8;
          ksrc = A.tk + off;
          vsrc = A.tv + off;
          v = true;
        }
      }
      cp_async16(smem_u32(ks + row * kLd + ch * 8), ksrc, v);
      cp_async16(smem_u32(vs + row * kLd + ch * 8), vsrc, v);
    }
  };

  load_tile(0, 0);
  cp_commit();

  // rows owned by this thread: rA (c0,c1) and rB = rA + 8 (c2,c3)
  const int rA = r0 + warp * 16 + (lane >> 2);
  const int rB = rA + 8;
  const bool warp_active = r0 + warp * 16 < rows_valid;
  uint64_t ancA[4] = {0, 0, 0, 0}, ancB[4] = {0, 0, 0, 0};
  if (has_tree) {
    const int jA = rA < rows_valid ? rA / A.G : -1;
    const int jB = rB < rows_valid ? rB / A.G : -1;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      if (w < A.W && jA >= 0) ancA[w] = A.anc[((int64_t)b * A.n_max + jA) * A.W + w];
      if (w < A.W && jB >= 0) ancB[w] = A.anc[((int64_t)b * A.n_max + jB) * A.W + w];
    }
  }

  uint32_t qf[8][4];
  float o[16][4];
#pragma unroll
  for (int i = 0; i < 16; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float mA = -INFINITY, mB = -INFINITY, lA = 0.f, lB = 0.f;

  for (int i = 0; i < n_tiles; ++i) {
    const int stage = i & 1;
    if (i + 1 < n_tiles) load_tile(i + 1, stage ^ 1);
    cp_commit();
    cp_wait<1>();
    __syncthreads();
    if (i == 0 && warp_active) {
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) {
        const int row = warp * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        const int col = ks * 16 + (lane >> 4) * 8;
        ldsm_x4(smem_u32(Qs + row * kLd + col), qf[ks][0], qf[ks][1], qf[ks][2], qf[ks][3]);
      }
    }
    if (warp_active) {
      const uint16_t* ks_ = Ks + stage * kKeys * kLd;
      const uint16_t* vs_ = Vs + stage * kKeys * kLd;
      float s[8][4];
#pragma unroll
      for (int t = 0; t < 8; ++t) s[t][0] = s[t][1] = s[t][2] = s[t][3] = 0.f;
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
#pragma unroll
        for (int np = 0; np < 4; ++np) {
          const int key = np * 16 + (lane & 7) + (lane >> 4) * 8;
          const int col = kk * 16 + ((lane >> 3) & 1) * 8;
          uint32_t b0, b1, b2, b3;
          ldsm_x4(smem_u32(ks_ + key * kLd + col), b0, b1, b2, b3);
          mma16816(s[2 * np], qf[kk], b0, b1);
          mma16816(s[2 * np + 1], qf[kk], b2, b3);
        }
      }
      // scale + mask
      const bool tree_tile = i >= n_cache_tiles;
      const int base = tree_tile ? (i - n_cache_tiles) * kKeys : key_beg + i * kKeys;
#pragma unroll
      for (int t = 0; t < 8; ++t) {
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const int key = base + t * 8 + 2 * (lane & 3) + (c & 1);
          bool vis;
          if (tree_tile) {
            const uint64_t* an = (c < 2) ? ancA : ancB;
            const int w = key >> 6;
            uint64_t word = 0;
#pragma unroll
            for (int q = 0; q < 4; ++q) word = (q == w) ? an[q] : word;
            vis = (word >> (key & 63)) & 1ull;
          } else {
            vis = key < key_end;
          }
          s[t][c] = vis ? s[t][c] * A.scale_log2 : -INFINITY;
        }
      }
      // online softmax
      float mxA = -INFINITY, mxB = -INFINITY;
#pragma unroll
      for (int t = 0; t < 8; ++t) {
        mxA = fmaxf(mxA, fmaxf(s[t][0], s[t][1]));
        mxB = fmaxf(mxB, fmaxf(s[t][2], s[t][3]));
      }
#pragma unroll
      for (int off = 1; off < 4; off <<= 1) {
        mxA = fmaxf(mxA, __shfl_xor_sync(0xffffffffu, mxA, off));
        mxB = fmaxf(mxB, __shfl_xor_sync(0xffffffffu, mxB, off));
      }
      const float nA = fmaxf(mA, mxA), nB = fmaxf(mB, mxB);
      const float bA = nA == -INFINITY ? 0.f : nA;
      const float bB = nB == -INFINITY ? 0.f : nB;
      const float aA = ex2(mA - bA), aB = ex2(mB - bB);
      mA = nA;
      mB = nB;
      float sumA = 0.f, sumB = 0.f;
      uint32_t pa[4][4];
#pragma unroll
      for (int t = 0; t < 8; ++t) {
        const float p0 = ex2(s[t][0] - bA), p1 = ex2(s[t][1] - bA);
        const float p2 = ex2(s[t][2] - bB), p3 = ex2(s[t][3] - bB);
        sumA += p0 + p1;
        sumB += p2 + p3;
        const int kk = t >> 1;
        if ((t & 1) == 0) {
          pa[kk][0] = pack_bf16(p0, p1);
          pa[kk][1] = pack_bf16(p2, p3);
        } else {
          pa[kk][2] = pack_bf16(p0, p1);
          pa[kk][3] = pack_bf16(p2, p3);
        }
      }
      lA = lA * aA + sumA;
      lB = lB * aB + sumB;
#pragma unroll
      for (int t = 0; t < 16; ++t) {
        o[t][0] *= aA;
        o[t][1] *= aA;
        o[t][2] *= aB;
        o[t][3] *= aB;
      }
      // O += P V
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
        for (int dp = 0; dp < 8; ++dp) {
          const int key = kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
          const int col = dp * 16 + (lane >> 4) * 8;
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(smem_u32(vs_ + key * kLd + col), b0, b1, b2, b3);
          mma16816(o[2 * dp], pa[kk], b0, b1);
          mma16816(o[2 * dp + 1], pa[kk], b2, b3);
        }
      }
    }
    __syncthreads();
  }

  if (!warp_active) return;
#pragma unroll
  for (int off = 1; off < 4; off <<= 1) {
    lA += __shfl_xor_sync(0xffffffffu, lA, off);
    lB += __shfl_xor_sync(0xffffffffu, lB, off);
  }
  const int64_t pbase = ((int64_t)blockIdx.z * A.splits + split) * A.rows_pad;
  const float iA = lA > 0.f ? 1.f / lA : 0.f;
  const float iB = lB > 0.f ? 1.f / lB : 0.f;
  if (rA < rows_valid) {
    float* dst = A.ws_o + (pbase + rA) * D;
#pragma unroll
    for (int t = 0; t < 16; ++t)
      *reinterpret_cast<float2*>(dst + t * 8 + 2 * (lane & 3)) = make_float2(o[t][0] * iA, o[t][1] * iA);
    if ((lane & 3) == 0) A.ws_lse[pbase + rA] = mA + log2f(lA);
  }
  if (rB < rows_valid) {
    float* dst = A.ws_o + (pbase + rB) * D;
#pragma unroll
    for (int t = 0; t < 16; ++t)
      *reinterpret_cast<float2*>(dst + t * 8 + 2 * (lane & 3)) = make_float2(o[t][2] * iB, o[t][3] * iB);
    if ((lane & 3) == 0) A.ws_lse[pbase + rB] = mB + log2f(lB);
  }
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
  if (cap < p.chunk) p.chunk = (int)std::max<int64_t>(kKeys, ((cap + kKeys - 1) / kKeys) * kKeys);
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
  // the shared-memory opt-in is a per-device function attribute
  static std::atomic<uint64_t> attr_done{0};
  int dev = 0;
  cudaError_t e0 = cudaGetDevice(&dev);
  if (e0 != cudaSuccess) return e0;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(attr_done.load() & bit)) {
    e0 = cudaFuncSetAttribute(tree_attn_mma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              kSmemBytes);
    if (e0 != cudaSuccess) return e0;
    attr_done.fetch_or(bit);
  }
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
  tree_attn_mma_kernel<<<grid, kThreads, kSmemBytes, s>>>(A);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int64_t items = (int64_t)batch * n_max * heads_q;
  tree_attn_reduce_kernel<<<(unsigned)((items + 7) / 8), 256, 0, s>>>(A);
  return cudaGetLastError();
}

}  // namespace cure
