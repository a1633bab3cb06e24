// Stage 4: tree-masked GQA attention on tcgen05 tensor cores (Sec. 3.2 / 3.4 /
// 3.5, Tree Attention), one persistent CTA per SM.
//
// Work.  A unit is (sequence b, kv head h, row group rg): up to 256 query rows,
// the packed (node, group head) pairs of 2 * npb tree nodes (npb = 128 / G
// nodes per 128-row M tile).  A unit's keys are cut into 64-key tiles: the
// cache tiles 0..ceil(L_b/64)-1, then the tree tiles (the ancestor mask of a
// node for tree tile t is one 64-bit word).  All units' tiles are laid end to
// end and CTA c takes the contiguous range [c*T/P, (c+1)*T/P) ("stream-K"), so
// every SM gets the same number of tiles whatever the ragged cache lengths.
// A unit wholly inside one CTA writes its bf16 output directly; a unit cut by
// range boundaries writes one partial (normalised O, base-2 log-sum-exp) per
// piece, and the CTA that completes the unit's last piece (a per-unit counter,
// fence + atomic, no waiting) merges the pieces and writes the output.
//
// Roles (12 warps):
//   warps 0-3 / 4-7   softmax of M tile 0 / 1: thread t owns row t = TMEM lane t
//                     and writes its bf16 probabilities back into TMEM
//   warp 8            TMA producer: Q rows (4-D box: d x group head x node),
//                     64-key K and V tiles into 5-stage rings (128-byte
//                     swizzle), page ids prefetched, boxes issued from
//                     several lanes.  A tile from a paged cache is
//                     [8-key group][d half][8 keys][64 d] for K and V alike:
//                     one box per page of one head (a 5-D map), 2 KiB apart
//                     groups, so a 16-token page costs one 4 KiB box per
//                     operand.  A producer warp sustains only so many boxes a
//                     microsecond, so fewer, larger boxes load faster.  Tree
//                     tiles and contiguous caches use [d half][64 keys][64 d]
//                     for K and [16-key chunk][d half][16 keys][64 d] for V.
//   warps 9 / 10      S issuers (one lane each) of M tile 0 / 1:
//                     S_m = Q_m K^T (M128 N64 K128) into TMEM S_m
//   warp 11           PV issuer (one lane) of both M tiles:
//                     O_m += P_m V (A = P_m in TMEM, M128 N128 K64); it
//                     releases the K/V stage after the tile's last product.
//                     S is on the softmax's critical path and PV is not, so
//                     an S product never queues behind a PV issue.  The
//                     products of one group go out from one asm block with
//                     constant descriptor steps, which keeps the issuing
//                     lanes' instruction count low while the softmax warps
//                     share their schedulers.
// TMEM (512 columns): S[2] (2 x 64) | P[2][2] (4 x 32, bf16 pairs) | O[2]
// (2 x 128).  The softmax releases S_m as soon as it has loaded it, so the
// next tile's S product runs while this tile's exponentials are computed; P
// is double-buffered so that it can be written while the previous PV product
// still reads the other buffer.  S(j + 1) is issued as soon as the softmax
// has loaded S(j); PV(j) as soon as it has published P(j); a K/V ring stage
// is released when the PV products of its tile are done.
// The online softmax keeps a lazily updated row max (O is rescaled in TMEM only
// when the max grows by more than 2^8).  Every mbarrier wait is bounded; on a
// timeout the CTA raises CURE_DEVERR_TIMEOUT, drains and leaves.
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <atomic>

#include "attn_common.cuh"
#include "tc_ptx.cuh"

namespace cure {
namespace {

using namespace tc;

constexpr int BM = kAttnRowsCta;  // 128 rows per M tile
constexpr int BN = kAttnKeys;     // 64 keys per tile
constexpr int D = kAttnD;         // 128
constexpr int NS = 5;             // K and V ring stages
constexpr int kThreads = 384;     // 12 warps
constexpr uint32_t kTmemCols = 512;

constexpr int kQHalf = BM * 64 * 2;   // 16 KiB: [128 rows][64 d]
constexpr int kKVHalf = BN * 64 * 2;  // 8 KiB: [64 keys][64 d]
constexpr int kTile = 2 * kKVHalf;    // one K or V tile (16 KiB)
constexpr int kVChunk = 16 * D * 2;   // 4 KiB: V keys 16c..16c+15, both d halves
constexpr int kVHalf = kVChunk / 2;   // 2 KiB: one d half of a V chunk
// Tiles from a paged cache: [8-key group][d half][8 keys][64 d], one TMA box
// per page (its ps / 8 groups, both halves); 8-key groups 2 KiB apart.
constexpr int kPgGroup = 8 * D * 2;   // 2 KiB
constexpr int kPgHalf = kPgGroup / 2; // 1 KiB
constexpr int kOffQ = 0;                          // Q[m][half]
constexpr int kOffK = kOffQ + 4 * kQHalf;         // K[stage]
constexpr int kOffV = kOffK + NS * kTile;         // V[stage]
constexpr int kOffMisc = kOffV + NS * kTile;      // 196608
enum {
  B_QFULL = 0, B_QEMPTY = 1, B_KFULL = 2, B_VFULL = B_KFULL + NS, B_KVEMPTY = B_VFULL + NS,
  B_SFULL = B_KVEMPTY + NS, B_SFREE = B_SFULL + 2, B_PFULL = B_SFREE + 2, B_PVDONE = B_PFULL + 4,
  B_OFREE = B_PVDONE + 4, B_DRAIN = B_OFREE + 2, kNumBars = B_DRAIN + 3
};
constexpr int kOffTmemSlot = kOffMisc + 8 * kNumBars;
constexpr int kOffAbort = kOffTmemSlot + 4;
constexpr int kOffLast = kOffAbort + 4;
constexpr int kOffPrefix = kOffLast + 8;             // int tiles_start[B+1], units_start[B+1]
constexpr int kSmemBytes = kOffPrefix + 8 * (kAttnMaxBatch + 1);
static_assert(kSmemBytes <= 232448, "fits the 227 KiB opt-in");

constexpr uint32_t kColS = 0;    // S[m]:      columns m*64
constexpr uint32_t kColP = 128;  // P[m][buf]: columns 128 + m*64 + buf*32
constexpr uint32_t kColO = 256;  // O[m]:      columns 256 + m*128

// One S product group, S_m = Q_m K^T over K = 128 (8 MMAs), in one asm
// block: the descriptors step by constant adds (16-byte units: 32 bytes
// within a 64-element half); kd and kd2 describe the two d halves of K.
__device__ __forceinline__ void mma_s_group(uint32_t d, uint64_t qd, uint64_t kd, uint64_t kd2, uint32_t idesc) {
  asm volatile(
      "{\n\t.reg .pred pf, pt;\n\t.reg .b64 a, b;\n\t"
      "setp.ne.b32 pf, %4, %4;\n\t"
      "setp.eq.b32 pt, %4, %4;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, pf;\n\t"
      "add.s64 a, %1, 2;\n\tadd.s64 b, %2, 2;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %3, pt;\n\t"
      "add.s64 a, %1, 4;\n\tadd.s64 b, %2, 4;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %3, pt;\n\t"
      "add.s64 a, %1, 6;\n\tadd.s64 b, %2, 6;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %3, pt;\n\t"
      "add.s64 a, %1, %5;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], a, %6, %3, pt;\n\t"
      "add.s64 a, %1, %5 + 2;\n\tadd.s64 b, %6, 2;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %3, pt;\n\t"
      "add.s64 a, %1, %5 + 4;\n\tadd.s64 b, %6, 4;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %3, pt;\n\t"
      "add.s64 a, %1, %5 + 6;\n\tadd.s64 b, %6, 6;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %3, pt;\n\t}\n" ::"r"(d),
      "l"(qd), "l"(kd), "r"(idesc), "r"(0), "n"(kQHalf >> 4), "l"(kd2)
      : "memory");
}
// One PV product group, O_m (+)= P_m V over 64 keys (4 MMAs): A from TMEM
// (8 columns of bf16 pairs per step), B stepping by one V chunk.
__device__ __forceinline__ void mma_pv_group(uint32_t d, uint32_t pa, uint64_t vd, uint32_t idesc,
                                             uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p0, pt;\n\t.reg .b64 b;\n\t.reg .b32 t;\n\t"
      "setp.ne.b32 p0, %4, 0;\n\t"
      "setp.eq.b32 pt, %4, %4;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p0;\n\t"
      "add.u32 t, %1, 8;\n\tadd.s64 b, %2, %5;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [t], b, %3, pt;\n\t"
      "add.u32 t, %1, 16;\n\tadd.s64 b, %2, 2 * %5;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [t], b, %3, pt;\n\t"
      "add.u32 t, %1, 24;\n\tadd.s64 b, %2, 3 * %5;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [t], b, %3, pt;\n\t}\n" ::"r"(d),
      "r"(pa), "l"(vd), "r"(idesc), "r"(accumulate), "n"(kVChunk >> 4)
      : "memory");
}

struct Bar {
  uint32_t base;
  __device__ __forceinline__ uint32_t operator()(int i) const { return base + 8u * (uint32_t)i; }
};

// All lanes of the warp wait; the warp proceeds only if every lane succeeded.
__device__ __forceinline__ bool wait_warp(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                          int* err) {
  const bool ok = wait_bounded(bar, parity, abort_flag, err, true);
  return __all_sync(0xffffffffu, ok);
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

// max of three (sm_100 and later have a three-input float max)
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
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

// A unit's piece counter holds (launch tag << 9) | pieces arrived.  A word
// whose tag is not this launch's (left by an aborted launch, or never
// written) counts as zero, so the workspace needs no reset; a completed unit
// leaves zero behind, so an old word can only match a later tag if its launch
// was aborted exactly 2^23 - 1 launches earlier.
constexpr int kCountBits = 9;
constexpr int kCountMask = (1 << kCountBits) - 1;
__device__ __forceinline__ int count_of(int v, uint32_t tag) {
  return ((uint32_t)v >> kCountBits) == tag ? (v & kCountMask) : 0;
}
// This piece's arrival (after its release fence): the pieces arrived so far,
// this one included.
__device__ __forceinline__ int arrive(int* cnt, uint32_t tag) {
  int old = *reinterpret_cast<volatile int*>(cnt);
  while (true) {
    const int nw = (int)((tag << kCountBits) | (uint32_t)(count_of(old, tag) + 1));
    const int prev = atomicCAS(cnt, old, nw);
    if (prev == old) return nw & kCountMask;
    old = prev;
  }
}

__device__ __forceinline__ int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void named_sync_softmax() {  // warps 0-7
  asm volatile("bar.sync 1, 256;" ::: "memory");
}

__device__ __forceinline__ void tma_load_5d(uint32_t dst, const CUtensorMap* map, uint32_t bar,
                                            int c0, int c1, int c2, int c3, int c4) {
  asm volatile(
      "cp.async.bulk.tensor.5d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5, %6, %7}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(c4)
      : "memory");
}
// An L2 prefetch of one 4-D box (no shared memory, no barrier).
__device__ __forceinline__ void tma_prefetch_4d(const CUtensorMap* map, int c0, int c1, int c2, int c3) {
  asm volatile("cp.async.bulk.prefetch.tensor.4d.L2.global.tile [%0, {%1, %2, %3, %4}];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(c0), "r"(c1), "r"(c2), "r"(c3)
               : "memory");
}
__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap* map, uint32_t bar,
                                            int c0, int c1, int c2, int c3) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5, %6}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
      : "memory");
}

// One unit piece owned by this CTA.
struct Seg {
  int b, h, rg;    // unit
  int u;           // global unit id
  int t0, t1;      // tile range within the unit
  int T;           // tiles of the unit
  int nct;         // cache tiles of the unit
  int L, n;        // cache length, tree nodes
  int part, parts; // piece index and piece count of the unit
  int slot;        // first workspace slot of the unit
  long long next;  // cost position after the piece
};

// Work is laid out in cost positions: each unit takes C positions of fixed
// cost (its piece start-up, epilogue and merge, in tile times) followed by
// one position per 64-key tile.  The CTA ranges split the cost positions
// evenly, so a CTA that starts more units gets fewer tiles.
struct Sched {
  const int* tiles_start;  // smem [B+1]: first cost position of each sequence's units
  const int* units_start;  // smem [B+1]
  int B, Hkv, P, C;
  long long Ttot;          // total cost positions
  const int* cache_len;
  const int* n_nodes;
  int cap, n_max;
  bool inplace;            // tree rows at cache slots L + j: one key range [0, L + n)
  __device__ int owner(long long g) const {  // the CTA whose range holds position g
    return (int)(((g + 1) * (long long)P - 1) / Ttot);
  }
  // The piece that starts at cost position g (or at the first tile after it,
  // when g is one of a unit's fixed-cost positions) and ends no later than
  // g_end; s.next is the position after it.  s.t0 == s.t1 when the range
  // holds no tile of that unit.
  __device__ Seg at(long long g, long long g_end) const {
    int lo = 0, hi = B;  // largest b with tiles_start[b] <= g
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (tiles_start[mid] <= g) lo = mid;
      else hi = mid;
    }
    Seg s;
    s.b = lo;
    s.L = max(0, min(cache_len[lo], cap));
    s.n = max(1, min(n_nodes[lo], n_max));
    if (inplace && s.L + s.n > cap) s.L = max(0, cap - s.n);
    // cache tiles (0..nct-1), then the tree tiles of separate tree tensors;
    // in the in-place layout every tile is a cache tile over keys 0..L+n-1
    s.nct = ((inplace ? s.L + s.n : s.L) + BN - 1) / BN;
    s.T = inplace ? s.nct : s.nct + (s.n + BN - 1) / BN;
    const long long local = g - tiles_start[lo];
    const int Tc = s.T + C;
    const int uib = (int)(local / Tc);
    s.rg = uib / Hkv;
    s.h = uib % Hkv;
    s.u = units_start[lo] + uib;
    const int o = (int)(local % Tc);
    const long long ustart = g - o + C;  // cost position of the unit's first tile
    const long long gs = o < C ? ustart : g;
    s.t0 = (int)(gs - ustart);
    s.t1 = gs < g_end ? (int)min((long long)s.T, (long long)s.t0 + (g_end - gs)) : s.t0;
    s.next = o < C && gs >= g_end ? g_end : gs + (s.t1 - s.t0);
    const int o0 = owner(ustart), o1 = owner(ustart + s.T - 1);
    s.parts = o1 - o0 + 1;
    s.part = owner(gs) - o0;
    s.slot = s.u + o0;
    return s;
  }
};

// INPLACE: the in-place layout (no tree tensors; node j's rows at cache slot
// L + j), a template parameter so that the separate-tensor kernel carries
// none of its tests.
template <bool INPLACE>
__global__ void __launch_bounds__(kThreads, 1)
tree_attn_tc_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                    const __grid_constant__ CUtensorMap tm_tk, const __grid_constant__ CUtensorMap tm_tv,
                    const __grid_constant__ CUtensorMap tm_q, const AttnArgs A) {
  extern __shared__ __align__(1024) uint8_t smem[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t sb = smem_u32(smem);
  if (sb & 1023u) {  // the swizzled tiles need a 1 KiB-aligned base
    if (tid == 0) flag(A.err, CURE_DEVERR_ALIGN);
    return;
  }
  const int B = A.batch, Hkv = A.kv.heads_kv, G = A.G;
  const int npb = BM / G;  // tree nodes per M tile
  const Bar bar{sb + kOffMisc};
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + kOffAbort);
  volatile int* last_flag = reinterpret_cast<volatile int*>(smem + kOffLast);
  int* tiles_start = reinterpret_cast<int*>(smem + kOffPrefix);
  int* units_start = tiles_start + (kAttnMaxBatch + 1);

  // ---------------------------------------------------------------- set-up
  if (tid == 0) {
    mbar_init(bar(B_QFULL), 1);
    mbar_init(bar(B_QEMPTY), 2);
    for (int i = 0; i < NS; ++i) {
      mbar_init(bar(B_KFULL + i), 1);
      mbar_init(bar(B_VFULL + i), 1);
      mbar_init(bar(B_KVEMPTY + i), 1);
    }
    for (int m = 0; m < 2; ++m) {
      mbar_init(bar(B_SFULL + m), 1);
      mbar_init(bar(B_SFREE + m), 128);
      mbar_init(bar(B_PFULL + 2 * m), 128);
      mbar_init(bar(B_PFULL + 2 * m + 1), 128);
      mbar_init(bar(B_PVDONE + 2 * m), 1);
      mbar_init(bar(B_PVDONE + 2 * m + 1), 1);
      mbar_init(bar(B_OFREE + m), 128);
      mbar_init(bar(B_DRAIN + m), 1);
    }
    mbar_init(bar(B_DRAIN + 2), 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(sb + kOffTmemSlot, kTmemCols);
  if (warp == 8 && lane == 0) {
    tma_prefetch_desc(&tm_q);
    tma_prefetch_desc(&tm_k);
    tma_prefetch_desc(&tm_v);
    tma_prefetch_desc(&tm_tk);
    tma_prefetch_desc(&tm_tv);
  }
  // Q rows at or past npb * G are never written by the Q copies: zero them once
  const int pad_rows = BM - npb * G;
  for (int c = tid; c < 4 * pad_rows * 8; c += kThreads) {
    const int q16 = c & 7, rr = npb * G + ((c >> 3) % pad_rows), mh = (c >> 3) / pad_rows;
    st_shared_v4(sb + kOffQ + mh * kQHalf + rr * 128 + q16 * 16, 0u, 0u, 0u, 0u);
  }
  // the set-up above reads no global memory; wait for the previous kernel on
  // the stream before the first read (programmatic dependent launch)
  pdl_begin();
  // per-sequence tiles and units, and their prefix sums (warp 9 scans)
  if (warp == 9) {
    int run_t = 0, run_u = 0;
    for (int base = 0; base < B; base += 32) {
      const int b = base + lane;
      int tb = 0, ub = 0;
      if (b < B) {
        int L = A.cache_len[b], n = A.n_nodes[b];
        if (L < 0 || L > A.cap) {
          if (blockIdx.x == 0) flag(A.err, CURE_DEVERR_SLOT);
          L = max(0, min(L, A.cap));
        }
        if (n < 1 || n > A.n_max) {
          if (blockIdx.x == 0) flag(A.err, CURE_DEVERR_NODES);
          n = max(1, min(n, A.n_max));
        }
        if (INPLACE && L + n > A.cap) {  // the tree rows must fit in the cache
          if (blockIdx.x == 0) flag(A.err, CURE_DEVERR_SLOT);
          L = max(0, A.cap - n);
        }
        const int rg = (n + 2 * npb - 1) / (2 * npb);
        ub = rg * Hkv;
        const int T = INPLACE ? (L + n + BN - 1) / BN : (L + BN - 1) / BN + (n + BN - 1) / BN;
        tb = ub * (T + A.unit_cost);
      }
      int it = tb, iu = ub;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int yt = __shfl_up_sync(0xffffffffu, it, off);
        const int yu = __shfl_up_sync(0xffffffffu, iu, off);
        if (lane >= off) {
          it += yt;
          iu += yu;
        }
      }
      if (b < B) {
        tiles_start[b] = run_t + it - tb;
        units_start[b] = run_u + iu - ub;
      }
      run_t += __shfl_sync(0xffffffffu, it, 31);
      run_u += __shfl_sync(0xffffffffu, iu, 31);
    }
    if (lane == 0) {
      tiles_start[B] = run_t;
      units_start[B] = run_u;
    }
  }
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(smem + kOffTmemSlot);

  Sched sch;
  sch.tiles_start = tiles_start;
  sch.units_start = units_start;
  sch.B = B;
  sch.Hkv = Hkv;
  sch.C = A.unit_cost;
  sch.Ttot = tiles_start[B];
  // with fewer tiles than CTAs only the first Ttot CTAs take part, so that every
  // taking part owns at least one tile and a unit's pieces are its owners
  sch.P = (int)min((long long)gridDim.x, sch.Ttot);
  sch.cache_len = A.cache_len;
  sch.n_nodes = A.n_nodes;
  sch.cap = A.cap;
  sch.n_max = A.n_max;
  sch.inplace = INPLACE;
  const bool takes_part = (int)blockIdx.x < sch.P;
  const long long g_begin = takes_part ? (long long)blockIdx.x * sch.Ttot / sch.P : 0;
  const long long g_end = takes_part ? (long long)(blockIdx.x + 1) * sch.Ttot / sch.P : 0;
  // M tile 1 of a piece is active when its first node is a tree node
  auto active1 = [&](const Seg& s) { return (2 * s.rg + 1) * npb < s.n; };

  if (warp == 8) {
    // ================================================================ producer
    const int ps = A.kv.page_size;
    const int ppt = A.kv.layout == 1 ? BN / ps : 0;
    const uint32_t qbytes = (uint32_t)(npb * G * 128);
    uint32_t qc = 0, gk = 0;  // pieces started, tiles issued (ring position)
    uint32_t k_issued = 0, v_issued = 0;
    bool ok = true;
    for (long long g = g_begin; ok && g < g_end;) {
      const Seg s = sch.at(g, g_end);
      g = s.next;
      if (s.t1 <= s.t0) continue;
      // the next piece's Q boxes are prefetched into L2 now, so that its Q
      // load at the piece boundary is served from L2
      if (g < g_end && lane == 0) {
        const Seg nx = sch.at(g, g_end);
        if (nx.t1 > nx.t0) {
          for (int m = 0; m < (active1(nx) ? 2 : 1); ++m)
            for (int hf = 0; hf < 2; ++hf)
              tma_prefetch_4d(&tm_q, hf * 64, 0, nx.h, nx.b * A.n_max + (2 * nx.rg + m) * npb);
        }
      }
      // Q of both M tiles once the previous piece's S products are done; it
      // is requested after the piece's first K/V tile, whose ring stage frees
      // up independently, so that the ring refills across the piece boundary
      auto load_q = [&]() -> bool {
        if (!wait_warp(bar(B_QEMPTY), (qc & 1u) ^ 1u, abort_flag, A.err)) return false;
        ++qc;
        if (lane == 0) {
          mbar_arrive_expect_tx(bar(B_QFULL), 4 * qbytes);
          for (int m = 0; m < 2; ++m) {
            const int node0 = (2 * s.rg + m) * npb;
            for (int hf = 0; hf < 2; ++hf)
              tma_load_4d(sb + kOffQ + (2 * m + hf) * kQHalf, &tm_q, bar(B_QFULL), hf * 64, 0, s.h,
                          s.b * A.n_max + node0);
          }
        }
        __syncwarp();
        return true;
      };
      int pg[8];
      for (int t = s.t0; ok && t < s.t1; ++t) {
        // page ids of up to 32 tiles, one tile per lane, fetched together
        if (ppt > 0 && t < s.nct && ((t - s.t0) & 31) == 0) {
          const int tl = t + lane;
#pragma unroll
          for (int p = 0; p < 8; ++p) {
            pg[p] = -1;
            if (p < ppt && tl < s.nct && tl < s.t1) {
              const int tok = tl * BN + p * ps;
              if (tok < s.L + (INPLACE ? s.n : 0) && tok / ps < A.kv.max_len) {
                const int page = A.kv.block_table[(int64_t)s.b * A.kv.max_len + tok / ps];
                if (page < 0 || page >= A.kv.num_pages) flag(A.err, CURE_DEVERR_PAGE);
                else pg[p] = page;  // a missing page stays -1: its box reads zeros
              }
            }
          }
        }
        int tpg[8];
#pragma unroll
        for (int p = 0; p < 8; ++p) tpg[p] = -1;
        if (ppt > 0 && t < s.nct) {
#pragma unroll
          for (int p = 0; p < 8; ++p) tpg[p] = __shfl_sync(0xffffffffu, pg[p], (t - s.t0) & 31);
        }
        const int st = (int)(gk % NS);
        const uint32_t ph = ((gk / NS) & 1u) ^ 1u;
        // The boxes of one tile are issued by several lanes at once (one box
        // each): a single issuing thread sustains only a few boxes per
        // microsecond, and a paged tile is 2 * (64 / page_size) boxes.
        auto page_of = [&](int p) {
          int pgv = tpg[0];
#pragma unroll
          for (int q = 1; q < 8; ++q) pgv = (q == p) ? tpg[q] : pgv;
          return pgv;
        };
        // A paged cache tile is one box per page (lane p: page p of the
        // tile, ps * 256 bytes into the stage); a contiguous cache tile or a
        // tree tile is two 64-key K boxes (one per d half) and four 16-key V
        // chunks.
        auto issue_k = [&](uint32_t dst, uint32_t fb) {
          if (t < s.nct) {
            if (A.kv.layout == 0) {
              if (lane < 2)
                tma_load_3d(dst + lane * kKVHalf, &tm_k, fb, lane * 64, s.h, s.b * A.kv.max_len + t * BN);
            } else if (lane < ppt) {
              tma_load_5d(dst + lane * ps * 256, &tm_k, fb, 0, 0, 2 * s.h, 0, page_of(lane));
            }
          } else if (lane < 2) {
            tma_load_3d(dst + lane * kKVHalf, &tm_tk, fb, lane * 64, s.h, s.b * A.n_max + (t - s.nct) * BN);
          }
        };
        auto issue_v = [&](uint32_t dst, uint32_t fb) {
          if (t < s.nct) {
            if (A.kv.layout == 0) {
              if (lane < 4)
                tma_load_4d(dst + lane * kVChunk, &tm_v, fb, 0, s.b * A.kv.max_len + t * BN + 16 * lane, 0, s.h);
            } else if (lane < ppt) {
              tma_load_5d(dst + lane * ps * 256, &tm_v, fb, 0, 0, 2 * s.h, 0, page_of(lane));
            }
          } else if (lane < 4) {
            tma_load_4d(dst + lane * kVChunk, &tm_tv, fb, 0, s.b * A.n_max + (t - s.nct) * BN + 16 * lane, 0, s.h);
          }
        };
        if (!wait_warp(bar(B_KVEMPTY + st), ph, abort_flag, A.err)) { ok = false; break; }
        if (lane == 0) mbar_arrive_expect_tx(bar(B_KFULL + st), kTile);
        __syncwarp();
        issue_k(sb + kOffK + st * kTile, bar(B_KFULL + st));
        __syncwarp();
        ++k_issued;
        if (lane == 0) mbar_arrive_expect_tx(bar(B_VFULL + st), kTile);
        __syncwarp();
        issue_v(sb + kOffV + st * kTile, bar(B_VFULL + st));
        __syncwarp();
        ++v_issued;
        ++gk;
        if (t == s.t0 && !load_q()) { ok = false; break; }
      }
    }
    if (*abort_flag) {  // let copies in flight land before the CTA's smem goes away
      for (uint32_t i = (k_issued > NS ? k_issued - NS : 0); i < k_issued; ++i)
        wait_bounded(bar(B_KFULL + i % NS), (i / NS) & 1u, abort_flag, A.err, false);
      for (uint32_t i = (v_issued > NS ? v_issued - NS : 0); i < v_issued; ++i)
        wait_bounded(bar(B_VFULL + i % NS), (i / NS) & 1u, abort_flag, A.err, false);
      if (qc > 0) wait_bounded(bar(B_QFULL), (qc - 1) & 1u, abort_flag, A.err, false);
    }
  } else if (warp == 9 || warp == 10) {
    // ================================================================ S issuers
    // warp 9 + m issues S_m = Q_m K^T as soon as the softmax has loaded the
    // previous S_m and the tile's K has landed
    const int m = warp - 9;
    constexpr uint32_t idS = idesc_bf16_f32(BM, BN, false);
    uint32_t qc = 0, gk = 0, sc = 0;
    bool ok = true;
    for (long long g = g_begin; ok && g < g_end;) {
      const Seg s = sch.at(g, g_end);
      g = s.next;
      if (s.t1 <= s.t0) continue;
      const int n = s.t1 - s.t0;
      const uint32_t gk0 = gk;
      gk += (uint32_t)n;
      if (!wait_warp(bar(B_QFULL), qc & 1u, abort_flag, A.err)) { ok = false; break; }
      ++qc;
      if (!(m == 0 || active1(s))) {  // no rows in this M tile: Q is free at once
        if (lane == 0) mbar_arrive(bar(B_QEMPTY));
        __syncwarp();
        continue;
      }
      const uint64_t qd = sdesc_sw128(sb + kOffQ + 2 * m * kQHalf, 16, 1024);
      for (int j = 0; ok && j < n; ++j) {
        const uint32_t gt = gk0 + (uint32_t)j;
        if (sc > 0 && !wait_warp(bar(B_SFREE + m), (sc - 1) & 1u, abort_flag, A.err)) { ok = false; break; }
        if (!wait_warp(bar(B_KFULL + gt % NS), (gt / NS) & 1u, abort_flag, A.err)) { ok = false; break; }
        tc_fence_after();
        if (lane == 0) {
          // a paged cache tile interleaves the d halves per 8-key group
          const bool pgd = A.kv.layout == 1 && s.t0 + j < s.nct;
          const uint32_t ka = sb + kOffK + (gt % NS) * kTile;
          const uint32_t sbo = pgd ? kPgGroup : 1024u, kh = pgd ? kPgHalf : kKVHalf;
          mma_s_group(tmem + kColS + m * 64, qd, sdesc_sw128(ka, 16, sbo), sdesc_sw128(ka + kh, 16, sbo), idS);
          mma_commit(bar(B_SFULL + m));
          if (j == n - 1) mma_commit(bar(B_QEMPTY));  // the piece's last use of Q
        }
        __syncwarp();
        ++sc;
      }
    }
    if (lane == 0) mma_commit(bar(B_DRAIN + m));
    __syncwarp();
    wait_bounded(bar(B_DRAIN + m), 0, abort_flag, A.err, false);
  } else if (warp == 11) {
    // ================================================================ PV issuer
    // O_m += P_m V for both M tiles as soon as the softmax has published P_m;
    // the K/V stage is released after the tile's last PV product
    constexpr uint32_t idO = idesc_bf16_f32(BM, D, true);
    uint32_t gk = 0, pc0 = 0, pc1 = 0, oc0 = 0, oc1 = 0;
    bool ok = true;
    for (long long g = g_begin; ok && g < g_end;) {
      const Seg s = sch.at(g, g_end);
      g = s.next;
      if (s.t1 <= s.t0) continue;
      const int n = s.t1 - s.t0;
      const uint32_t gk0 = gk;
      gk += (uint32_t)n;
      const bool two = active1(s);
      auto issue_pv = [&](int m, uint32_t& pc, uint32_t& oc, int j, uint32_t gt) -> bool {
        if (!wait_warp(bar(B_PFULL + 2 * m + (pc & 1u)), (pc >> 1) & 1u, abort_flag, A.err)) return false;
        if (j == 0) {  // O_m holds the previous piece until its epilogue has read it
          if (!wait_warp(bar(B_OFREE + m), (oc & 1u) ^ 1u, abort_flag, A.err)) return false;
          ++oc;
        }
        tc_fence_after();
        if (lane == 0) {
          // V as an MN-major operand: the d halves LBO apart, 8-key groups SBO
          // apart; a K = 16 step is 4 KiB in both layouts
          const bool pgd = A.kv.layout == 1 && s.t0 + j < s.nct;
          mma_pv_group(tmem + kColO + m * 128, tmem + kColP + m * 64 + (pc & 1u) * 32,
                       sdesc_sw128(sb + kOffV + (gt % NS) * kTile, pgd ? kPgHalf : kVHalf,
                                   pgd ? kPgGroup : 1024u),
                       idO, j > 0 ? 1u : 0u);
          mma_commit(bar(B_PVDONE + 2 * m + (pc & 1u)));
        }
        __syncwarp();
        ++pc;
        return true;
      };
      for (int j = 0; ok && j < n; ++j) {
        const uint32_t gt = gk0 + (uint32_t)j;
        if (!wait_warp(bar(B_VFULL + gt % NS), (gt / NS) & 1u, abort_flag, A.err)) { ok = false; break; }
        if (!issue_pv(0, pc0, oc0, j, gt) || (two && !issue_pv(1, pc1, oc1, j, gt))) { ok = false; break; }
        if (lane == 0) mma_commit(bar(B_KVEMPTY + gt % NS));  // the tile's K and V are consumed
        __syncwarp();
      }
    }
    if (lane == 0) mma_commit(bar(B_DRAIN + 2));
    __syncwarp();
    wait_bounded(bar(B_DRAIN + 2), 0, abort_flag, A.err, false);
  } else {
    // ================================================================ softmax
    const int m = warp >> 2;   // M tile
    const int row = tid & 127; // row within the M tile = TMEM lane
    const uint32_t tl = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    const float c = A.scale_log2;
    uint32_t sc = 0, gk = 0;
    bool ok = true;
    for (long long g = g_begin; g < g_end;) {
      const Seg s = sch.at(g, g_end);
      g = s.next;
      if (s.t1 <= s.t0) continue;
      const int n = s.t1 - s.t0;
      const uint32_t gk0 = gk;
      gk += (uint32_t)n;
      const bool act = m == 0 || active1(s);
      const int node0 = (2 * s.rg + m) * npb;
      const int node = node0 + row / G, gh = row % G;
      const bool vrow = act && row < npb * G && node < s.n;
      float m_run = -INFINITY, l_run = 0.f;
      if (act && ok) {
        for (int jj = 0; jj < n; ++jj) {
          const int t = s.t0 + jj;
          if (!wait_warp(bar(B_SFULL + m), sc & 1u, abort_flag, A.err)) { ok = false; break; }
          const uint32_t tcur = sc;  // this M tile's tile count: P buffer tcur & 1
          const uint32_t pbuf = tcur & 1u;
          ++sc;
          tc_fence_after();
          uint32_t u0[32], u1[32];
          tmem_ld32(tl + kColS + m * 64, u0);
          tmem_ld32(tl + kColS + m * 64 + 32, u1);
          tmem_wait_ld();
          tc_fence_before();
          mbar_arrive(bar(B_SFREE + m));  // S_m may be overwritten by the next product

          // raw scores, -inf where masked; the scale is applied in the exponent
          const bool tree = t >= s.nct;
          const int kend = INPLACE ? s.L + s.n : s.L;  // keys of the cache tiles
          const int valid = tree ? min(BN, s.n - (t - s.nct) * BN) : min(BN, kend - t * BN);
          // in the in-place layout, a tile that reaches past L holds tree rows
          // (key k is node k - L): cache keys below L are visible, tree keys
          // through the row's ancestor bits, read at the tile's offset
          const bool mixed = INPLACE && (t + 1) * BN > s.L;
          float x[64];
          if (mixed) {
            const int off = t * BN - s.L;  // node of the tile's first key, > -64
            uint64_t vis = 0ull;
            if (vrow) {
              const uint64_t* ar = A.anc + ((int64_t)s.b * A.n_max + node) * A.W;
              if (off < 0) {
                vis = (ar[0] << (-off)) | ((1ull << (-off)) - 1ull);
              } else {
                const int wi = off >> 6, sh = off & 63;
                const uint64_t lo = wi < A.W ? ar[wi] : 0ull;
                const uint64_t hi = (sh != 0 && wi + 1 < A.W) ? ar[wi + 1] : 0ull;
                vis = (lo >> sh) | (sh != 0 ? hi << (64 - sh) : 0ull);
              }
            } else if (off < 0) {
              vis = (1ull << (-off)) - 1ull;
            }
            const uint32_t w0 = (uint32_t)vis, w1 = (uint32_t)(vis >> 32);
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              x[i] = ((w0 >> i) & 1u) ? __uint_as_float(u0[i]) : -INFINITY;
              x[32 + i] = ((w1 >> i) & 1u) ? __uint_as_float(u1[i]) : -INFINITY;
            }
          } else if (tree) {
            const int wi = t - s.nct;
            const uint64_t word = vrow ? A.anc[((int64_t)s.b * A.n_max + node) * A.W + wi] : 0ull;
            const uint32_t w0 = (uint32_t)word, w1 = (uint32_t)(word >> 32);
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              x[i] = ((w0 >> i) & 1u) ? __uint_as_float(u0[i]) : -INFINITY;
              x[32 + i] = ((w1 >> i) & 1u) ? __uint_as_float(u1[i]) : -INFINITY;
            }
          } else if (valid == BN) {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              x[i] = __uint_as_float(u0[i]);
              x[32 + i] = __uint_as_float(u1[i]);
            }
          } else {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              x[i] = i < valid ? __uint_as_float(u0[i]) : -INFINITY;
              x[32 + i] = 32 + i < valid ? __uint_as_float(u1[i]) : -INFINITY;
            }
          }
          float mx[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) mx[i] = fmax3(x[i], x[8 + i], x[16 + i]);
#pragma unroll
          for (int i = 0; i < 8; ++i) mx[i] = fmax3(mx[i], x[24 + i], x[32 + i]);
#pragma unroll
          for (int i = 0; i < 8; ++i) mx[i] = fmax3(mx[i], x[40 + i], x[48 + i]);
#pragma unroll
          for (int i = 0; i < 8; ++i) mx[i] = fmaxf(mx[i], x[56 + i]);
          const float mt = fmax3(fmax3(mx[0], mx[1], mx[2]), fmax3(mx[3], mx[4], mx[5]),
                                 fmaxf(mx[6], mx[7])) * c;
          const float m_new = fmaxf(m_run, mt);
          const bool need = m_new > m_run + 8.0f;
          const float m_use = need ? m_new : m_run;
          const float nbase = m_use == -INFINITY ? 0.f : -m_use;
          // P(t) goes into buffer t & 1 once PV(t - 2), which read it last, is
          // done (each buffer has its own done barrier: PV(t) completes phase
          // t >> 1 of barrier t & 1, and PV(t) cannot start before P(t) is
          // published, so a wait is never two phases behind)
          if (tcur >= 2) {
            if (!wait_warp(bar(B_PVDONE + 2 * m + pbuf), ((tcur >> 1) & 1u) ^ 1u, abort_flag, A.err)) { ok = false; break; }
            tc_fence_after();
          }
          // exponent arguments and row sums two at a time (packed f32x2); each
          // half of P goes to TMEM as soon as it is computed, so that the first
          // half's store runs under the second half's exponentials
          uint32_t pk[32];
          const uint64_t c2 = f2_pack(c, c), nb2 = f2_pack(nbase, nbase);
          uint64_t sm2[2] = {f2_pack(0.f, 0.f), f2_pack(0.f, 0.f)};
          auto exp_pair = [&](int i) {
            float a0, a1;
            f2_unpack(f2_fma(f2_pack(x[2 * i], x[2 * i + 1]), c2, nb2), a0, a1);
            const float p0 = ex2(a0), p1 = ex2(a1);
            sm2[i & 1] = f2_add(sm2[i & 1], f2_pack(p0, p1));
            pk[i] = pack_bf16(p0, p1);
          };
#pragma unroll
          for (int i = 0; i < 16; ++i) exp_pair(i);
          tmem_st16(tl + kColP + m * 64 + pbuf * 32, pk);
#pragma unroll
          for (int i = 16; i < 32; ++i) exp_pair(i);
          tmem_st16(tl + kColP + m * 64 + pbuf * 32 + 16, pk + 16);
          float sm[4];
          f2_unpack(sm2[0], sm[0], sm[1]);
          f2_unpack(sm2[1], sm[2], sm[3]);
          // O_m is rescaled only once PV(t - 1) is done
          if (jj > 0 && __any_sync(0xffffffffu, need)) {
            const uint32_t tp = tcur - 1;
            if (!wait_warp(bar(B_PVDONE + 2 * m + (tp & 1u)), (tp >> 1) & 1u, abort_flag, A.err)) { ok = false; break; }
            tc_fence_after();
            {
              const float alpha = need ? ex2(m_run - m_new) : 1.f;
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                uint32_t o[32];
                tmem_ld32(tl + kColO + m * 128 + q * 32, o);
                tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
                tmem_st32(tl + kColO + m * 128 + q * 32, o);
              }
            }
          }
          if (need) {
            l_run *= ex2(m_run - m_new);
            m_run = m_new;
          }
          l_run += (sm[0] + sm[1]) + (sm[2] + sm[3]);
          // the V rows past the last valid key of a partial tile are zeroed (by
          // both M tiles: the second writes the same zeros) so that their
          // unspecified contents cannot reach O through 0 * NaN
          if (valid < BN) {
            const uint32_t gt = gk0 + (uint32_t)jj;
            const int st = (int)(gt % NS);
            if (!wait_warp(bar(B_VFULL + st), (gt / NS) & 1u, abort_flag, A.err)) { ok = false; break; }
            const uint32_t vb = sb + kOffV + st * kTile;
            const int nch = (BN - valid) * 16;
            const bool pgd = A.kv.layout == 1 && !tree;
            for (int q = row; q < nch; q += BM) {
              const int rr = valid + (q >> 4), hf = (q >> 3) & 1, cc = q & 7;
              const uint32_t off = pgd ? (rr >> 3) * kPgGroup + hf * kPgHalf + (rr & 7) * 128
                                       : (rr >> 4) * kVChunk + hf * kVHalf + (rr & 15) * 128;
              st_shared_v4(vb + off + cc * 16, 0u, 0u, 0u, 0u);
            }
            fence_proxy_async_smem();
          }
          tmem_wait_st();
          tc_fence_before();
          mbar_arrive(bar(B_PFULL + 2 * m + pbuf));
        }
        if (ok) {  // O_m is final once the piece's last PV product is done
          const uint32_t tl_ = sc - 1;
          if (!wait_warp(bar(B_PVDONE + 2 * m + (tl_ & 1u)), (tl_ >> 1) & 1u, abort_flag, A.err)) ok = false;
        }
        if (ok) tc_fence_after();
      }
      // ---- epilogue of the piece
      const bool whole = s.t0 == 0 && s.t1 == s.T;
      const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
      // a piece's partial: fp32 float4 columns [32][256 rows], so that the 32
      // rows of a warp touch 512 contiguous bytes at every column
      const int prow = m * BM + row;
      float4* pslot = reinterpret_cast<float4*>(A.ws_o) + (int64_t)(s.slot + s.part) * (32 * 2 * BM);
      uint16_t* orow =
          A.out + (((int64_t)s.b * A.n_max + min(node, A.n_max - 1)) * A.heads_q + s.h * G + gh) * D;
      if (whole) {
        if (act && ok) {
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            uint32_t o[32];
            tmem_ld32(tl + kColO + m * 128 + q * 32, o);
            tmem_wait_ld();
            if (vrow) {
#pragma unroll
              for (int i = 0; i < 32; i += 8) {
                uint4 v;
                v.x = pack_bf16(__uint_as_float(o[i]) * inv, __uint_as_float(o[i + 1]) * inv);
                v.y = pack_bf16(__uint_as_float(o[i + 2]) * inv, __uint_as_float(o[i + 3]) * inv);
                v.z = pack_bf16(__uint_as_float(o[i + 4]) * inv, __uint_as_float(o[i + 5]) * inv);
                v.w = pack_bf16(__uint_as_float(o[i + 6]) * inv, __uint_as_float(o[i + 7]) * inv);
                *reinterpret_cast<uint4*>(orow + q * 32 + i) = v;
              }
            }
          }
          tc_fence_before();
          mbar_arrive(bar(B_OFREE + m));
        }
      } else {
        // A piece whose unit's other pieces have all published already is the
        // last one for sure: it neither writes its own partial nor publishes,
        // and merges with its O read straight from TMEM.  Otherwise it writes
        // its partial, publishes (release fence + counter), and merges if the
        // counter says it came last.  O_m is released after the merge.
        const float lse_own = m_run + log2f(l_run);
        named_sync_softmax();
        if (tid == 0)
          *last_flag = (!*abort_flag && count_of(ld_acquire(A.cnt + s.u), A.tag) == s.parts - 1) ? 2 : 0;
        named_sync_softmax();
        int last = *last_flag;
        if (last != 2) {
          if (act && ok) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              uint32_t o[32];
              tmem_ld32(tl + kColO + m * 128 + q * 32, o);
              tmem_wait_ld();
              if (vrow) {
#pragma unroll
                for (int i = 0; i < 8; ++i)
                  pslot[(q * 8 + i) * (2 * BM) + prow] =
                      make_float4(__uint_as_float(o[4 * i]) * inv, __uint_as_float(o[4 * i + 1]) * inv,
                                  __uint_as_float(o[4 * i + 2]) * inv, __uint_as_float(o[4 * i + 3]) * inv);
              }
            }
          }
          if (vrow && ok) A.ws_lse[(int64_t)(s.slot + s.part) * (2 * BM) + prow] = lse_own;
          __threadfence();
          named_sync_softmax();
          if (tid == 0) {
            int l = 0;
            if (!*abort_flag) {
              l = arrive(A.cnt + s.u, A.tag) == s.parts;
              if (l) A.cnt[s.u] = 0;  // a completed unit leaves a zero word behind
            }
            *last_flag = l;
          }
          named_sync_softmax();
          last = *last_flag;
        } else if (tid == 0) {
          A.cnt[s.u] = 0;  // a completed unit leaves a zero word behind
        }
        if (last && act && ok) {
          __threadfence();
          // O = sum_p w_p O_p with w_p = 2^(lse_p - M) / sum_q 2^(lse_q - M);
          // this piece's O_p comes from TMEM, the others' from the workspace,
          // their loads batched (two pieces x eight float4 columns per thread)
          const int own = s.part, no = s.parts - 1;  // other pieces: k -> k < own ? k : k + 1
          const float* lse0 = A.ws_lse + (int64_t)s.slot * (2 * BM) + prow;
          float M = lse_own;
          if (vrow)
            for (int k = 0; k < no; ++k) M = fmaxf(M, __ldcg(lse0 + (int64_t)(k < own ? k : k + 1) * 2 * BM));
          float wsum = ex2(lse_own - M);
          if (vrow)
            for (int k = 0; k < no; ++k) wsum += ex2(__ldcg(lse0 + (int64_t)(k < own ? k : k + 1) * 2 * BM) - M);
          const float winv = 1.f / wsum;
          const float wown = ex2(lse_own - M) * winv * inv;
          const float4* base = reinterpret_cast<const float4*>(A.ws_o) + (int64_t)s.slot * (32 * 2 * BM) + prow;
#pragma unroll 1
          for (int q = 0; q < 4; ++q) {
            uint32_t o[32];
            tmem_ld32(tl + kColO + m * 128 + q * 32, o);
            tmem_wait_ld();
            if (vrow) {
              float4 acc[8];
#pragma unroll
              for (int i = 0; i < 8; ++i)
                acc[i] = make_float4(__uint_as_float(o[4 * i]) * wown, __uint_as_float(o[4 * i + 1]) * wown,
                                     __uint_as_float(o[4 * i + 2]) * wown, __uint_as_float(o[4 * i + 3]) * wown);
#pragma unroll 1
              for (int k0 = 0; k0 < no; k0 += 2) {
                const bool two = k0 + 1 < no;
                const int pa_i = k0 < own ? k0 : k0 + 1, pb_i = k0 + 1 < own ? k0 + 1 : k0 + 2;
                float4 va[8], vb[8];
                const float4* pa = base + (int64_t)pa_i * (32 * 2 * BM) + q * 8 * (2 * BM);
                const float4* pbp = base + (int64_t)pb_i * (32 * 2 * BM) + q * 8 * (2 * BM);
#pragma unroll
                for (int i = 0; i < 8; ++i) va[i] = __ldcg(pa + i * (2 * BM));
                if (two) {
#pragma unroll
                  for (int i = 0; i < 8; ++i) vb[i] = __ldcg(pbp + i * (2 * BM));
                }
                const float wa = ex2(__ldcg(lse0 + (int64_t)pa_i * 2 * BM) - M) * winv;
                const float wb = two ? ex2(__ldcg(lse0 + (int64_t)pb_i * 2 * BM) - M) * winv : 0.f;
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                  acc[i].x += wa * va[i].x; acc[i].y += wa * va[i].y;
                  acc[i].z += wa * va[i].z; acc[i].w += wa * va[i].w;
                  if (two) {
                    acc[i].x += wb * vb[i].x; acc[i].y += wb * vb[i].y;
                    acc[i].z += wb * vb[i].z; acc[i].w += wb * vb[i].w;
                  }
                }
              }
#pragma unroll
              for (int i = 0; i < 8; i += 2) {
                uint4 v;
                v.x = pack_bf16(acc[i].x, acc[i].y);
                v.y = pack_bf16(acc[i].z, acc[i].w);
                v.z = pack_bf16(acc[i + 1].x, acc[i + 1].y);
                v.w = pack_bf16(acc[i + 1].z, acc[i + 1].w);
                *reinterpret_cast<uint4*>(orow + q * 32 + i * 4) = v;
              }
            }
          }
        }
        if (act && ok) {
          tc_fence_before();
          mbar_arrive(bar(B_OFREE + m));
        }
      }
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

// [rows][Hkv][128] bf16 viewed as (d, head, row); boxes of 64 d x 1 head x box_rows.
bool make_kv_map(CUtensorMap* m, const void* base, uint64_t rows, int Hkv, int box_rows) {
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

// V rows [rows][Hkv][128] bf16 viewed as (d in half, row, d half, head);
// boxes of 64 d x 16 rows x 2 halves: [half][16 rows][64 d], one 4 KiB chunk.
bool make_v_rows_map(CUtensorMap* m, const void* base, uint64_t rows, int Hkv) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[4] = {64, (cuuint64_t)rows, 2, (cuuint64_t)Hkv};
  cuuint64_t strides[3] = {(cuuint64_t)Hkv * D * 2, 128, (cuuint64_t)D * 2};
  cuuint32_t box[4] = {64, 16, 2, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Paged K or V [pages][ps][Hkv][128] bf16 viewed as (d in half, row in an
// 8-row group, d half + 2 * head, group in page, page); one box is a whole
// page of one head: [group][d half][8 rows][64 d], ps * 256 bytes.
bool make_page_map(CUtensorMap* m, const void* base, uint64_t pages, int ps, int Hkv) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[5] = {64, 8, 2 * (cuuint64_t)Hkv, (cuuint64_t)(ps / 8), (cuuint64_t)pages};
  cuuint64_t strides[4] = {(cuuint64_t)Hkv * D * 2, 128, (cuuint64_t)8 * Hkv * D * 2,
                           (cuuint64_t)ps * Hkv * D * 2};
  cuuint32_t box[5] = {64, 8, 2, (cuuint32_t)(ps / 8), 1};
  cuuint32_t es[5] = {1, 1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// q [tokens][Hkv][G][128] bf16 viewed as (d, group head, kv head, token); boxes
// of 64 d x G x 1 x npb tokens: the rows of one M tile, (node, g) packed.
bool make_q_map(CUtensorMap* m, const void* base, uint64_t tokens, int Hkv, int G, int npb) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)G, (cuuint64_t)Hkv, (cuuint64_t)tokens};
  cuuint64_t strides[3] = {(cuuint64_t)D * 2, (cuuint64_t)G * D * 2, (cuuint64_t)Hkv * G * D * 2};
  cuuint32_t box[4] = {64, (cuuint32_t)G, 1, (cuuint32_t)npb};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, es,
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
    e = cudaFuncSetAttribute(tree_attn_tc_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             kSmemBytes);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(tree_attn_tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               kSmemBytes);
    if (e != cudaSuccess) return e;
    attr_done.fetch_or(bit);
  }
  const int Hkv = A.kv.heads_kv;
  CUtensorMap mk, mv, mtk, mtv, mq;
  bool ok;
  if (A.kv.layout == 0) {
    const uint64_t rows = (uint64_t)A.batch * A.kv.max_len;
    ok = make_kv_map(&mk, A.kc, rows, Hkv, BN) && make_v_rows_map(&mv, A.vc, rows, Hkv);
  } else {
    const int ps = A.kv.page_size;
    ok = make_page_map(&mk, A.kc, (uint64_t)A.kv.num_pages, ps, Hkv) &&
         make_page_map(&mv, A.vc, (uint64_t)A.kv.num_pages, ps, Hkv);
  }
  const uint64_t trows = (uint64_t)A.batch * A.n_max;
  // in the in-place layout the tree maps are never used for a copy; they are
  // encoded over Q (at least as large) so that every map passed is valid
  const void* tk = A.inplace ? static_cast<const void*>(A.q) : A.tk;
  const void* tv = A.inplace ? static_cast<const void*>(A.q) : A.tv;
  ok = ok && make_kv_map(&mtk, tk, trows, Hkv, BN) && make_v_rows_map(&mtv, tv, trows, Hkv) &&
       make_q_map(&mq, A.q, trows, Hkv, A.G, BM / A.G);
  if (!ok) return cudaErrorInvalidValue;
  // a fresh tag per launch makes the piece counters left in the workspace
  // count as zero (1 .. 2^23 - 1; zero-filled memory is never current)
  static std::atomic<uint32_t> launches{0};
  AttnArgs a = A;
  a.tag = launches.fetch_add(1) % ((1u << (32 - kCountBits)) - 1) + 1;
  e = A.inplace ? launch_pdl(tree_attn_tc_kernel<true>, grid, dim3(kThreads), kSmemBytes, s, mk, mv, mtk,
                             mtv, mq, a)
                : launch_pdl(tree_attn_tc_kernel<false>, grid, dim3(kThreads), kSmemBytes, s, mk, mv, mtk,
                             mtv, mq, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace cure
