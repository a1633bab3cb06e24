// Stage 4 main kernel: tree-masked GQA attention on tcgen05 tensor cores
// (Sec. 3.2 / 3.4 / 3.5, Tree Attention).
//
// One CTA = 128 query rows (packed (node, group head) pairs of one sequence and
// kv head) x one split of the cache keys (plus the tree keys on the last
// split).  Six warps:
//   warps 0-3  softmax: thread t owns query row t = TMEM lane t
//   warp 4     TMA producer: 64-key K and V tiles, 128-byte swizzled,
//              double-buffered
//   warp 5     MMA issuer (one lane): S = Q K^T (M128 N64 K128) into one of two
//              TMEM S buffers, O += P V (M128 N128 K64) into the TMEM O buffer
// TMEM: S[2] (2 x 64 columns) + O (128 columns) = 256 columns, so two CTAs
// share an SM.  P goes through swizzled shared memory.  The online softmax
// keeps a lazily updated row max: O in TMEM is rescaled only when the max
// grows by more than 2^8, which keeps every probability below 256.
// Every wait on an mbarrier is bounded; on a timeout the CTA raises
// CURE_DEVERR_TIMEOUT, drains its copies and MMAs, frees TMEM and leaves.
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <atomic>

#include "attn_common.cuh"
#include "tc_ptx.cuh"

namespace cure {
namespace {

using namespace tc;

constexpr int BM = kAttnRowsCta;  // 128
constexpr int BN = kAttnKeys;     // 64
constexpr int D = kAttnD;         // 128
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kColS = 0;    // S buffers: columns [0, 64) and [64, 128)
constexpr uint32_t kColO = 128;  // O: columns [128, 256)

constexpr int kQHalf = BM * 64 * 2;   // 16 KiB: [128 rows][64 d]
constexpr int kKVHalf = BN * 64 * 2;  // 8 KiB: [64 keys][64 d]
constexpr int kTile = 2 * kKVHalf;    // one K or V tile
constexpr int kOffQ = 0;
constexpr int kOffK = kOffQ + 2 * kQHalf;
constexpr int kOffV = kOffK + 2 * kTile;
constexpr int kOffP = kOffV + 2 * kTile;
constexpr int kOffBar = kOffP + BM * BN * 2;
enum { B_KFULL = 0, B_VFULL = 2, B_KEMPTY = 4, B_VEMPTY = 6, B_SFULL = 8, B_SFREE = 10,
       B_PFULL = 12, B_PVDONE = 13, B_DRAIN = 14, kNumBars = 15 };
constexpr int kOffTmemSlot = kOffBar + 8 * kNumBars;
constexpr int kOffAbort = kOffTmemSlot + 4;
constexpr int kSmemBytes = kOffBar + 128;
static_assert(kOffAbort + 4 <= kSmemBytes, "bookkeeping fits");

constexpr long long kTimeoutCycles = 1LL << 30;  // about half a second

__device__ __forceinline__ bool wait_bounded(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                             int* err, bool honour_abort) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (honour_abort && *abort_flag) return false;
    if (clock64() - t0 > kTimeoutCycles) {
      *abort_flag = 1;
      flag(err, CURE_DEVERR_TIMEOUT);
      return false;
    }
  }
}

// All lanes of the warp wait; the warp proceeds only if every lane succeeded.
__device__ __forceinline__ bool wait_warp(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                          int* err) {
  const bool ok = wait_bounded(bar, parity, abort_flag, err, true);
  return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c,
                                             uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c),
               "r"(d)
               : "memory");
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
               "r"(valid ? 16 : 0)
               : "memory");
}

__global__ void __launch_bounds__(kThreads, 2)
tree_attn_tc_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                    const __grid_constant__ CUtensorMap tm_tk,
                    const __grid_constant__ CUtensorMap tm_tv, const AttnArgs A) {
  extern __shared__ __align__(1024) uint8_t smem[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t sb = smem_u32(smem);
  if (sb & 1023u) {  // the swizzled tiles need a 1 KiB-aligned base
    if (tid == 0) flag(A.err, CURE_DEVERR_ALIGN);
    return;
  }

  const int rb = blockIdx.x, split = blockIdx.y;
  const int Hkv = A.kv.heads_kv;
  const int b = blockIdx.z / Hkv, h = blockIdx.z % Hkv;
  int L = A.cache_len[b];
  int n = A.n_nodes[b];
  if (L < 0 || L > A.cap || n < 1 || n > A.n_max) {
    if (tid == 0 && rb == 0 && split == 0 && h == 0)
      flag(A.err, (L < 0 || L > A.cap) ? CURE_DEVERR_SLOT : CURE_DEVERR_NODES);
    L = max(0, min(L, A.cap));
    n = max(1, min(n, A.n_max));
  }
  const int rows_valid = n * A.G;
  const int r0 = rb * BM;
  if (r0 >= rows_valid) return;
  const int nsplit = max(1, (L + A.chunk - 1) / A.chunk);
  if (split >= nsplit) return;
  const int key_beg = split * A.chunk;
  const int key_end = min(L, key_beg + A.chunk);
  const bool has_tree = split == nsplit - 1;
  const int n_cache_tiles = (key_end - key_beg + BN - 1) / BN;
  const int n_tiles = n_cache_tiles + (has_tree ? (n + BN - 1) / BN : 0);

  const uint32_t bar0 = sb + kOffBar;
  auto bar = [&](int i) -> uint32_t { return bar0 + 8u * (uint32_t)i; };
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + kOffAbort);

  if (tid == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(B_KFULL + i), 1);
      mbar_init(bar(B_VFULL + i), 1);
      mbar_init(bar(B_KEMPTY + i), 1);
      mbar_init(bar(B_VEMPTY + i), 1);
      mbar_init(bar(B_SFULL + i), 1);
      mbar_init(bar(B_SFREE + i), 128);
    }
    mbar_init(bar(B_PFULL), 128);
    mbar_init(bar(B_PVDONE), 1);
    mbar_init(bar(B_DRAIN), 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(sb + kOffTmemSlot, kTmemCols);
  if (warp == 4 && lane == 0) {
    tma_prefetch_desc(&tm_k);
    tma_prefetch_desc(&tm_v);
    if (has_tree) {
      tma_prefetch_desc(&tm_tk);
      tma_prefetch_desc(&tm_tv);
    }
  }

  // Q rows of this block into the swizzled K-major layout (zero past the valid rows)
  for (int c = tid; c < BM * 16; c += kThreads) {
    const int row = c >> 4, ch = c & 15, half = ch >> 3, cc = ch & 7;
    const int r = r0 + row;
    const bool v = r < rows_valid;
    const int j = v ? r / A.G : 0, g = v ? r % A.G : 0;
    const uint16_t* src =
        v ? A.q + (((int64_t)b * A.n_max + j) * A.heads_q + h * A.G + g) * D + ch * 8 : A.q;
    cp_async16(sb + kOffQ + half * kQHalf + row * 128 + ((cc ^ (row & 7)) << 4), src, v);
  }
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_all;" ::: "memory");
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(smem + kOffTmemSlot);

  if (warp == 4) {
    // ------------------------------------------------------------ TMA producer
    // One 64-key tile of K (or V) into `dst`: cache tiles come from the
    // contiguous or paged cache, the tree tiles from this step's tree rows.
    // Physical page ids of the split are fetched 32 tiles at a time, one tile
    // per lane (up to 8 pages of a 64-key tile in registers), and handed to
    // lane 0 by shuffles: no dependent global load sits in front of a copy.
    const int ps = A.kv.page_size;
    const int ppt = A.kv.layout == 1 ? BN / ps : 0;  // pages per tile
    int pg[8];
    auto fetch_pages = [&](int window) {
      const int j = window * 32 + lane;
#pragma unroll
      for (int p = 0; p < 8; ++p) {
        pg[p] = -1;
        if (p < ppt && j < n_cache_tiles) {
          const int tok = key_beg + j * BN + p * ps;
          if (tok < key_end) {
            const int page = A.kv.block_table[(int64_t)b * A.kv.max_len + tok / ps];
            if (page < 0 || page >= A.kv.num_pages) flag(A.err, CURE_DEVERR_PAGE);
            else pg[p] = page;  // a missing page stays -1: its box reads zeros
          }
        }
      }
    };
    int tile_pg[8];
    // One 64-key tile of K (or V) into `dst`: cache tiles come from the
    // contiguous or paged cache, the tree tiles from this step's tree rows.
    auto load_tile = [&](int j, uint32_t dst, uint32_t fb, const CUtensorMap* cache_map,
                         const CUtensorMap* tree_map) {
      if (j < n_cache_tiles) {
        const int t0 = key_beg + j * BN;
        if (A.kv.layout == 0) {
          const int row = b * A.kv.max_len + t0;
          for (int hf = 0; hf < 2; ++hf) tma_load_3d(dst + hf * kKVHalf, cache_map, fb, hf * 64, h, row);
        } else {
#pragma unroll
          for (int p = 0; p < 8; ++p) {
            if (p < ppt) {
              for (int hf = 0; hf < 2; ++hf)
                tma_load_3d(dst + hf * kKVHalf + p * ps * 128, cache_map, fb, hf * 64, h,
                            tile_pg[p] * ps);
            }
          }
        }
      } else {
        const int row = b * A.n_max + (j - n_cache_tiles) * BN;
        for (int hf = 0; hf < 2; ++hf) tma_load_3d(dst + hf * kKVHalf, tree_map, fb, hf * 64, h, row);
      }
    };
    int k_issued = 0, v_issued = 0;
    for (int j = 0; j < n_tiles; ++j) {
      const int s = j & 1;
      const uint32_t use = (uint32_t)j >> 1;
      if (ppt > 0 && j < n_cache_tiles) {
        if ((j & 31) == 0) fetch_pages(j >> 5);
#pragma unroll
        for (int p = 0; p < 8; ++p) tile_pg[p] = __shfl_sync(0xffffffffu, pg[p], j & 31);
      }
      // K stage s frees when S(j-2) completes, V stage s when PV(j-2) does
      if (!wait_warp(bar(B_KEMPTY + s), (use & 1u) ^ 1u, abort_flag, A.err)) break;
      if (lane == 0) {
        const uint32_t dk = sb + kOffK + s * kTile;
        mbar_arrive_expect_tx(bar(B_KFULL + s), kTile);
        load_tile(j, dk, bar(B_KFULL + s), &tm_k, &tm_tk);
      }
      __syncwarp();
      k_issued = j + 1;
      if (!wait_warp(bar(B_VEMPTY + s), (use & 1u) ^ 1u, abort_flag, A.err)) break;
      if (lane == 0) {
        const uint32_t dv = sb + kOffV + s * kTile;
        mbar_arrive_expect_tx(bar(B_VFULL + s), kTile);
        load_tile(j, dv, bar(B_VFULL + s), &tm_v, &tm_tv);
      }
      __syncwarp();
      v_issued = j + 1;
    }
    if (*abort_flag) {  // let copies in flight land before the CTA's smem goes away
      for (int jj = max(0, k_issued - 2); jj < k_issued; ++jj)
        wait_bounded(bar(B_KFULL + (jj & 1)), ((uint32_t)jj >> 1) & 1u, abort_flag, A.err, false);
      for (int jj = max(0, v_issued - 2); jj < v_issued; ++jj)
        wait_bounded(bar(B_VFULL + (jj & 1)), ((uint32_t)jj >> 1) & 1u, abort_flag, A.err, false);
    }
  } else if (warp == 5) {
    // ------------------------------------------------------------ MMA issuer
    constexpr uint32_t idS = idesc_bf16_f32(BM, BN, false);
    constexpr uint32_t idO = idesc_bf16_f32(BM, D, true);
    auto issue_s = [&](int j) -> bool {
      const int s = j & 1;
      const uint32_t use = (uint32_t)j >> 1;
      if (!wait_warp(bar(B_KFULL + s), use & 1u, abort_flag, A.err)) return false;
      if (!wait_warp(bar(B_SFREE + s), (use & 1u) ^ 1u, abort_flag, A.err)) return false;
      tc_fence_after();
      if (lane == 0) {
        const uint32_t qa = sb + kOffQ, ka = sb + kOffK + s * kTile;
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
          const uint32_t oq = (ks >> 2) * kQHalf + (ks & 3) * 32;
          const uint32_t okk = (ks >> 2) * kKVHalf + (ks & 3) * 32;
          mma_bf16_ss(tmem + kColS + s * BN, sdesc_sw128(qa + oq, 16, 1024),
                      sdesc_sw128(ka + okk, 16, 1024), idS, ks > 0 ? 1u : 0u);
        }
        mma_commit(bar(B_SFULL + s));
        mma_commit(bar(B_KEMPTY + s));
      }
      __syncwarp();
      return true;
    };
    bool ok = issue_s(0) && (n_tiles < 2 || issue_s(1));
    for (int j = 0; ok && j < n_tiles; ++j) {
      const int s = j & 1;
      const uint32_t use = (uint32_t)j >> 1;
      if (!wait_warp(bar(B_PFULL), (uint32_t)j & 1u, abort_flag, A.err)) break;
      if (!wait_warp(bar(B_VFULL + s), use & 1u, abort_flag, A.err)) break;
      tc_fence_after();
      if (lane == 0) {
        const uint32_t pa = sb + kOffP, va = sb + kOffV + s * kTile;
#pragma unroll
        for (int ks = 0; ks < 4; ++ks) {
          mma_bf16_ss(tmem + kColO, sdesc_sw128(pa + ks * 32, 16, 1024),
                      sdesc_sw128(va + ks * 16 * 128, kKVHalf, 1024), idO,
                      (j > 0 || ks > 0) ? 1u : 0u);
        }
        mma_commit(bar(B_PVDONE));
        mma_commit(bar(B_VEMPTY + s));
      }
      __syncwarp();
      // S(j+2) reuses the S buffer that softmax(j) has finished reading
      if (j + 2 < n_tiles && !issue_s(j + 2)) break;
    }
    // every MMA issued by this warp has completed once the drain barrier flips
    if (lane == 0) mma_commit(bar(B_DRAIN));
    __syncwarp();
    wait_bounded(bar(B_DRAIN), 0, abort_flag, A.err, false);
  } else {
    // ------------------------------------------------------------ softmax (rows)
    const int row = tid;
    const int r = r0 + row;
    const bool vrow = r < rows_valid;
    const int jrow = vrow ? r / A.G : 0;
    uint64_t an[4] = {0ull, 0ull, 0ull, 0ull};
    if (has_tree && vrow) {
#pragma unroll
      for (int w = 0; w < 4; ++w)
        if (w < A.W) an[w] = A.anc[((int64_t)b * A.n_max + jrow) * A.W + w];
    }
    const uint32_t tl = tmem + ((uint32_t)(warp * 32) << 16);
    const float c = A.scale_log2;
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    for (int j = 0; j < n_tiles; ++j) {
      const int s = j & 1;
      const uint32_t use = (uint32_t)j >> 1;
      if (!wait_warp(bar(B_SFULL + s), use & 1u, abort_flag, A.err)) {
        ok = false;
        break;
      }
      tc_fence_after();
      uint32_t u0[32], u1[32];
      tmem_ld32(tl + kColS + s * BN, u0);
      tmem_ld32(tl + kColS + s * BN + 32, u1);
      tmem_wait_ld();
      tc_fence_before();
      mbar_arrive(bar(B_SFREE + s));

      const bool tree = j >= n_cache_tiles;
      float x[64];
      if (tree) {
        const int wi = j - n_cache_tiles;
        const uint64_t word = wi == 0 ? an[0] : wi == 1 ? an[1] : wi == 2 ? an[2] : an[3];
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          x[i] = ((word >> i) & 1ull) ? __uint_as_float(u0[i]) * c : -INFINITY;
          x[32 + i] = ((word >> (32 + i)) & 1ull) ? __uint_as_float(u1[i]) * c : -INFINITY;
        }
      } else {
        const int lim = key_end - (key_beg + j * BN);
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          x[i] = i < lim ? __uint_as_float(u0[i]) * c : -INFINITY;
          x[32 + i] = 32 + i < lim ? __uint_as_float(u1[i]) * c : -INFINITY;
        }
      }
      float mx[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) mx[i] = x[i];
#pragma unroll
      for (int i = 8; i < 64; ++i) mx[i & 7] = fmaxf(mx[i & 7], x[i]);
      const float mt = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                             fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
      const float m_new = fmaxf(m_run, mt);
      const bool need = m_new > m_run + 8.0f;
      // the row max used for this tile's probabilities (lazily updated)
      const float m_use = need ? m_new : m_run;
      const float base = m_use == -INFINITY ? 0.f : m_use;
      uint32_t pk[32];
      float sm[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const float p0 = ex2(x[2 * i] - base), p1 = ex2(x[2 * i + 1] - base);
        sm[i & 3] += p0 + p1;
        pk[i] = pack_bf16(p0, p1);
      }

      // P and O are free once the previous PV product has completed
      if (j > 0) {
        if (!wait_warp(bar(B_PVDONE), (uint32_t)(j - 1) & 1u, abort_flag, A.err)) {
          ok = false;
          break;
        }
        tc_fence_after();
        if (__any_sync(0xffffffffu, need)) {
          const float alpha = need ? ex2(m_run - m_new) : 1.f;
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            uint32_t o[32];
            tmem_ld32(tl + kColO + q * 32, o);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
            tmem_st32(tl + kColO + q * 32, o);
          }
          tmem_wait_st();
        }
      }
      if (need) {
        l_run *= ex2(m_run - m_new);
        m_run = m_new;
      }
      l_run += (sm[0] + sm[1]) + (sm[2] + sm[3]);
      const uint32_t prow = sb + kOffP + row * 128;
#pragma unroll
      for (int q = 0; q < 8; ++q)
        st_shared_v4(prow + ((q ^ (row & 7)) << 4), pk[4 * q], pk[4 * q + 1], pk[4 * q + 2],
                     pk[4 * q + 3]);

      // a partial tile: zero the V rows past the last valid key so that their
      // (unspecified) contents cannot reach O through 0 * NaN
      const int valid = tree ? min(BN, n - (j - n_cache_tiles) * BN)
                             : min(BN, key_end - (key_beg + j * BN));
      if (valid < BN) {
        if (!wait_warp(bar(B_VFULL + s), use & 1u, abort_flag, A.err)) {
          ok = false;
          break;
        }
        const uint32_t vb = sb + kOffV + s * kTile;
        const int nch = (BN - valid) * 16;
        for (int q = row; q < nch; q += BM) {
          const int rr = valid + (q >> 4), hf = (q >> 3) & 1, cc = q & 7;
          st_shared_v4(vb + hf * kKVHalf + rr * 128 + cc * 16, 0u, 0u, 0u, 0u);
        }
      }
      fence_proxy_async_smem();
      tc_fence_before();
      mbar_arrive(bar(B_PFULL));
    }
    if (ok && wait_warp(bar(B_PVDONE), (uint32_t)(n_tiles - 1) & 1u, abort_flag, A.err)) {
      tc_fence_after();
      const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
      const int64_t pbase = ((int64_t)blockIdx.z * A.splits + split) * A.rows_pad;
      float* dst = A.ws_o + (pbase + r) * D;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        uint32_t o[32];
        tmem_ld32(tl + kColO + q * 32, o);
        tmem_wait_ld();
        if (vrow) {
#pragma unroll
          for (int i = 0; i < 32; i += 4)
            *reinterpret_cast<float4*>(dst + q * 32 + i) =
                make_float4(__uint_as_float(o[i]) * inv, __uint_as_float(o[i + 1]) * inv,
                            __uint_as_float(o[i + 2]) * inv, __uint_as_float(o[i + 3]) * inv);
        }
      }
      if (vrow) A.ws_lse[pbase + r] = m_run + log2f(l_run);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::atomic<bool> tried{false};
  if (!fn && !tried.exchange(true)) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// [rows][Hkv][128] bf16 viewed as a 3-D tensor (d, head, row); boxes of
// 64 d x 1 head x box_rows rows with 128-byte swizzle.
bool make_map(CUtensorMap* m, const void* base, uint64_t rows, int Hkv, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)Hkv, (cuuint64_t)rows};
  cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)Hkv * D * 2};
  cuuint32_t box[3] = {64, 1, (cuuint32_t)box_rows};
  cuuint32_t es[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

cudaError_t launch_tree_attn_tc(const AttnArgs& A, dim3 grid, cudaStream_t s) {
  static std::atomic<uint64_t> attr_done{0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(attr_done.load() & bit)) {
    e = cudaFuncSetAttribute(tree_attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             kSmemBytes);
    if (e != cudaSuccess) return e;
    attr_done.fetch_or(bit);
  }
  const int Hkv = A.kv.heads_kv;
  CUtensorMap mk, mv, mtk, mtv;
  bool ok;
  if (A.kv.layout == 0) {
    const uint64_t rows = (uint64_t)A.batch * A.kv.max_len;
    ok = make_map(&mk, A.kc, rows, Hkv, BN) && make_map(&mv, A.vc, rows, Hkv, BN);
  } else {
    const uint64_t rows = (uint64_t)A.kv.num_pages * A.kv.page_size;
    ok = make_map(&mk, A.kc, rows, Hkv, A.kv.page_size) &&
         make_map(&mv, A.vc, rows, Hkv, A.kv.page_size);
  }
  const uint64_t trows = (uint64_t)A.batch * A.n_max;
  ok = ok && make_map(&mtk, A.tk, trows, Hkv, BN) && make_map(&mtv, A.tv, trows, Hkv, BN);
  if (!ok) return cudaErrorInvalidValue;
  tree_attn_tc_kernel<<<grid, kThreads, kSmemBytes, s>>>(mk, mv, mtk, mtv, A);
  return cudaGetLastError();
}

}  // namespace cure
