// Stochastic verification (temperature T > 0): the target's token at every
// tree node drawn from softmax(logits / T) by inverse CDF with a uniform the
// caller supplies.  Speculative decoding is lossless sampling from the target
// (Sec. 2); the paper's own runs are greedy (Sec. 4.1), where the argmax of
// cure_accept takes this kernel's place.  The acceptance walk is the same in
// both cases: a child is accepted when its token equals the parent's sample.
//
// One CTA of four warps per (sequence, node) row.  The row is cut into eight-id
// groups on 16-byte boundaries (only the first and the last group can be
// partial) and each warp owns a contiguous quarter of the groups, which its
// lanes stream as 16-byte vectors, 32 adjacent groups per warp instruction:
//   1. one pass: a warp step covers 128 contiguous groups (four per lane);
//      every lane sums p_v = 2^((l_v - base) log2(e) / T) over them against a
//      warp-wide base, raised (and the running sums rescaled) only when a
//      logit lies more than 2^8 above it in p units; the warp's step masses
//      are summed into blocks of consecutive steps (at most 64 per segment),
//      and each block's mass is kept with its base in shared memory;
//   2. the segment masses are brought to the row's largest base and scanned in
//      id order: segment w covers the cumulative range [E_w, E_w + S_w), the
//      row total is Z, the target point is r = u Z;
//   3. the last segment with mass whose E_w <= r is searched by its warp: a
//      scan of its block masses finds the block holding r, whose groups are
//      then read again in id order, 32 at a time (a warp scan of the group
//      masses), down to the first id whose running sum exceeds r (the last id
//      with mass if rounding leaves r past the block's end).
// The exponent is formed as (l - base) * (log2(e) / T), never as a difference
// of two products, so it cannot overflow for any finite T > 0: at very small T
// every id below the maximum gets mass 0 and the draw picks among the maxima.
#include <float.h>

#include <type_traits>

#include "common.cuh"

namespace cure {
namespace {

constexpr int kSampleThreads = 128;
constexpr int kSampleWarps = kSampleThreads / 32;
constexpr int kSampleUnroll = 4;  // groups per lane per step (loads one step ahead)
constexpr float kLog2eS = 1.4426950408889634f;
constexpr float kRaise = 8.f;     // base raised when a term would exceed 2^8
constexpr int kMaxBlocks = 64;    // recorded block masses per warp segment

__device__ __forceinline__ float ex2s(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint4 ld_row(const uint4* p) {
  uint4 r;
  asm volatile("ld.global.nc.L2::256B.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

// The eight logits of group g (ids 8g - mis .. 8g - mis + 7) as packed bf16
// pairs; ids outside the row read as -inf (0xff80).  Whole groups are one
// 16-byte load, partial ones (the first and the last) are loaded element by
// element.
struct RowView {
  const uint16_t* rowp;  // the row's first logit
  const uint4* vbase;    // 16-byte aligned address of group 0 (may precede rowp)
  int mis;               // logits between vbase and rowp (0..7)
  int vocab;
  int ngroups;

  __device__ __forceinline__ uint4 load(int g) const {
    const int id0 = 8 * g - mis;
    if (id0 >= 0 && id0 + 8 <= vocab) return ld_row(vbase + g);
    uint32_t w[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int a = id0 + 2 * q, c = a + 1;
      const uint32_t lo = (a >= 0 && a < vocab) ? rowp[a] : 0xff80u;
      const uint32_t hi = (c >= 0 && c < vocab) ? rowp[c] : 0xff80u;
      w[q] = lo | (hi << 16);
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
  }
};

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
__device__ __forceinline__ float max3s(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// The (lo, hi) logit pair of one 32-bit word of a group.
__device__ __forceinline__ uint64_t pair_of(uint32_t w) {
  return f2_pack(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}

// The largest of a group's eight logits.
__device__ __forceinline__ float group_max_raw(const uint4& r) {
  const uint32_t w[4] = {r.x, r.y, r.z, r.w};
  float v[8];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    v[2 * q] = __uint_as_float(w[q] << 16);
    v[2 * q + 1] = __uint_as_float(w[q] & 0xffff0000u);
  }
  return max3s(max3s(v[0], v[1], v[2]), max3s(v[3], v[4], v[5]), fmaxf(v[6], v[7]));
}

__device__ __forceinline__ void unpack8(const uint4& r, float x[8]) {
  const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    x[2 * q] = __uint_as_float(w[q] << 16);
    x[2 * q + 1] = __uint_as_float(w[q] & 0xffff0000u);
  }
}

__device__ __forceinline__ float warp_max_s(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float warp_sum_s(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Mass of one group against `base` (a finite logit value).
__device__ __forceinline__ float group_mass(const float x[8], float base, float scale) {
  float s = 0.f;
#pragma unroll
  for (int e = 0; e < 8; ++e) s += ex2s((x[e] - base) * scale);
  return s;
}

__global__ void __launch_bounds__(kSampleThreads)
sample_target_kernel(const uint16_t* __restrict__ logits, const float* __restrict__ uniforms, float scale,
                     int n_max, int vocab, const int32_t* __restrict__ n_nodes, int32_t* __restrict__ targ,
                     int* err) {
  pdl_begin();
  const int64_t row = blockIdx.x;
  const int b = (int)(row / n_max), j = (int)(row % n_max);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int n = n_nodes[b];
  if (n < 1 || n > n_max) {
    if (tid == 0 && j == 0) flag(err, CURE_DEVERR_NODES);
    n = max(1, min(n, n_max));
  }
  if (j >= n) {  // uniform over the CTA
    if (tid == 0) targ[row] = -1;
    return;
  }

  RowView rv;
  rv.rowp = logits + row * (int64_t)vocab;
  rv.mis = (int)((reinterpret_cast<uintptr_t>(rv.rowp) >> 1) & 7);
  rv.vbase = reinterpret_cast<const uint4*>(rv.rowp - rv.mis);
  rv.vocab = vocab;
  rv.ngroups = (vocab + rv.mis + 7) >> 3;
  const int gpw = (rv.ngroups + kSampleWarps - 1) / kSampleWarps;  // groups per warp segment
  const int g_lo = min(rv.ngroups, warp * gpw), g_hi = min(rv.ngroups, g_lo + gpw);
  constexpr int kStepGroups = 32 * kSampleUnroll;  // contiguous groups one warp step covers
  const int steps = (g_hi - g_lo + kStepGroups - 1) / kStepGroups;
  // a block is `bstride` consecutive steps; at most kMaxBlocks per segment
  const int bstride = max(1, (steps + kMaxBlocks - 1) / kMaxBlocks);
  __shared__ float s_blk[kSampleWarps][kMaxBlocks], s_blkbase[kSampleWarps][kMaxBlocks];

  // ---- 1. block masses of the segment against a lazily raised warp base
  float base = -INFINITY;  // warp-uniform
  float bm = 0.f;          // current block's mass (warp-uniform)
  int blk = 0, in_blk = 0;
  uint64_t acc2 = f2_pack(0.f, 0.f);  // this lane's part of the current step's mass, as a pair
  // interior groups need no per-element bounds: [gf_lo, gf_hi) lie wholly inside the row
  const int gf_lo = rv.mis == 0 ? 0 : 1;
  const int gf_hi = (vocab + rv.mis) >> 3;
  const uint64_t sc2 = f2_pack(scale, scale);
  uint4 r4[kSampleUnroll];
#pragma unroll
  for (int u = 0; u < kSampleUnroll; ++u) {
    const int g = g_lo + lane + 32 * u;
    if (g < g_hi) r4[u] = rv.load(g);
  }
  // one warp step over groups g0 .. g0 + 127; FULL: every group of every lane
  // is whole and inside the segment, so no check is needed
  auto step = [&](int g0, auto full_tag) {
    constexpr bool FULL = decltype(full_tag)::value;
    uint4 nx[kSampleUnroll];
#pragma unroll
    for (int u = 0; u < kSampleUnroll; ++u) {
      const int g = g0 + lane + 32 * (kSampleUnroll + u);
      if (g < g_hi) nx[u] = (g >= gf_lo && g < gf_hi) ? ld_row(rv.vbase + g) : rv.load(g);
    }
    float gm = -INFINITY;
#pragma unroll
    for (int u = 0; u < kSampleUnroll; ++u)
      if (FULL || g0 + lane + 32 * u < g_hi) gm = fmaxf(gm, group_max_raw(r4[u]));
    // raise the base when some lane's terms would exceed 2^kRaise
    if (__any_sync(0xffffffffu, gm > base && (base == -INFINITY || (gm - base) * scale > kRaise))) {
      const float nb = warp_max_s(gm);
      if (base != -INFINITY) {
        const float f = ex2s((base - nb) * scale);
        bm *= f;
        acc2 = f2_mul(acc2, f2_pack(f, f));
      }
      base = nb;
    }
    if (base != -INFINITY) {
      // p = 2^((l - base) scale): a packed subtraction and product per pair;
      // never l * scale - base * scale, whose rounding error can be huge in
      // exponent units when scale is large
      const uint64_t nb2 = f2_pack(-base, -base);
#pragma unroll
      for (int u = 0; u < kSampleUnroll; ++u) {
        if (FULL || g0 + lane + 32 * u < g_hi) {
          const uint32_t w[4] = {r4[u].x, r4[u].y, r4[u].z, r4[u].w};
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            float a, b;
            f2_unpack(f2_mul(f2_add(pair_of(w[q]), nb2), sc2), a, b);
            acc2 = f2_add(acc2, f2_pack(ex2s(a), ex2s(b)));
          }
        }
      }
    }
    if (++in_blk == bstride || g0 + kStepGroups >= g_hi) {
      float a, b;
      f2_unpack(acc2, a, b);
      bm += warp_sum_s(a + b);
      acc2 = f2_pack(0.f, 0.f);
      if (lane == 0) {
        s_blk[warp][blk] = bm;
        s_blkbase[warp][blk] = base;
      }
      ++blk;
      bm = 0.f;
      in_blk = 0;
    }
#pragma unroll
    for (int u = 0; u < kSampleUnroll; ++u) r4[u] = nx[u];
  };
  int g0 = g_lo;
  // a partial first group (a row not on a 16-byte boundary) is checked; then
  // full steps while this step's groups and the next step's loads are whole
  // and in range; then the checked tail
  for (; g0 < g_hi && g0 < gf_lo; g0 += kStepGroups) step(g0, std::integral_constant<bool, false>());
  for (; g0 + 2 * kStepGroups <= min(g_hi, gf_hi); g0 += kStepGroups) step(g0, std::integral_constant<bool, true>());
  for (; g0 < g_hi; g0 += kStepGroups) step(g0, std::integral_constant<bool, false>());
  __syncwarp();
  // the segment's mass at its final base (bases only grow)
  float sm = 0.f;
  for (int i = lane; i < blk; i += 32)
    if (s_blkbase[warp][i] != -INFINITY) sm += s_blk[warp][i] * ex2s((s_blkbase[warp][i] - base) * scale);
  sm = warp_sum_s(sm);

  // ---- 2. segment masses at the row's base, scanned in id order
  __shared__ float s_base[kSampleWarps], s_mass[kSampleWarps];
  if (lane == 0) {
    s_base[warp] = base;
    s_mass[warp] = sm;
  }
  __syncthreads();
  float m = -INFINITY;
#pragma unroll
  for (int w = 0; w < kSampleWarps; ++w) m = fmaxf(m, s_base[w]);
  if (m == -INFINITY) {  // no finite logit: id 0, as the argmax's tie rule gives
    if (tid == 0) targ[row] = 0;
    return;
  }
  float E[kSampleWarps], S[kSampleWarps], total = 0.f;
#pragma unroll
  for (int w = 0; w < kSampleWarps; ++w) {
    S[w] = s_base[w] == -INFINITY ? 0.f : s_mass[w] * ex2s((s_base[w] - m) * scale);
    E[w] = total;
    total += S[w];
  }
  float u = uniforms[row];
  u = fminf(fmaxf(u, 0.f), 0x1.fffffep-1f);  // [0, 1); NaN -> 0
  const float r = u * total;
  int owner = 0;
#pragma unroll
  for (int w = 0; w < kSampleWarps; ++w)
    if (S[w] > 0.f && E[w] <= r) owner = w;
  if (warp != owner) return;

  // ---- 3a. the block of the owning segment that holds r
  float acc = E[owner];
  int bsel = -1, blast = -1;
  float bstart = acc, blast_start = acc;
  for (int i0 = 0; i0 < blk && bsel < 0; i0 += 32) {
    const int i = i0 + lane;
    const float q = (i < blk && s_blkbase[warp][i] != -INFINITY)
                        ? s_blk[warp][i] * ex2s((s_blkbase[warp][i] - m) * scale) : 0.f;
    float inc = q;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float y = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += y;
    }
    const unsigned hit = __ballot_sync(0xffffffffu, q > 0.f && acc + inc > r);
    const unsigned has = __ballot_sync(0xffffffffu, q > 0.f);
    if (hit) {
      const int l = __ffs(hit) - 1;
      bsel = i0 + l;
      bstart = acc + __shfl_sync(0xffffffffu, inc - q, l);
    } else if (has) {
      const int l = 31 - __clz(has);
      blast = i0 + l;
      blast_start = acc + __shfl_sync(0xffffffffu, inc - q, l);
    }
    acc += __shfl_sync(0xffffffffu, inc, 31);
  }
  if (bsel < 0) {  // rounding left r past the segment's end: its last block with mass
    bsel = blast >= 0 ? blast : 0;
    bstart = blast >= 0 ? blast_start : E[owner];
  }

  // ---- 3b. that block's groups in id order, 32 at a time
  const int c_lo = g_lo + bsel * bstride * kStepGroups;
  const int c_hi = min(g_hi, c_lo + bstride * kStepGroups);
  acc = bstart;
  int last = -1;  // the block's last id with mass seen so far (warp-uniform)
  for (int c0 = c_lo; c0 < c_hi; c0 += 32) {
    const int g = c0 + lane;
    float xv[8];
    float q = 0.f;
    if (g < c_hi) {
      unpack8(rv.load(g), xv);
      q = group_mass(xv, m, scale);
    }
    float inc = q;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float y = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += y;
    }
    const float tot = __shfl_sync(0xffffffffu, inc, 31);
    const unsigned has = __ballot_sync(0xffffffffu, q > 0.f);
    const unsigned hit = __ballot_sync(0xffffffffu, q > 0.f && acc + inc > r);
    if (hit) {
      const int l = __ffs(hit) - 1;  // first group whose running sum passes r
      if (lane == l) {
        float a = acc + inc - q;
        int pick = -1, lastv = -1;
        for (int e = 0; e < 8; ++e) {
          const float p = ex2s((xv[e] - m) * scale);
          if (p > 0.f) {
            lastv = 8 * g - rv.mis + e;
            if (a + p > r) {
              pick = lastv;
              break;
            }
          }
          a += p;
        }
        targ[row] = pick >= 0 ? pick : lastv;
      }
      return;
    }
    if (has) {
      // the last group with mass in this chunk: its last id with mass
      const int l = 31 - __clz(has);
      int lv = -1;
      if (lane == l)
        for (int e = 0; e < 8; ++e)
          if (ex2s((xv[e] - m) * scale) > 0.f) lv = 8 * g - rv.mis + e;
      last = __shfl_sync(0xffffffffu, lv, l);
    }
    acc += tot;
  }
  // rounding left r past the block's end: its last id with mass
  if (lane == 0) targ[row] = last >= 0 ? last : 0;
}

}  // namespace

cudaError_t launch_sample_target(const uint16_t* logits, const float* uniforms, float temperature, int batch,
                                 int n_max, int vocab, const int32_t* n_nodes, int32_t* targ, int* err,
                                 cudaStream_t s) {
  if (batch == 0) return cudaSuccess;
  const unsigned rows = (unsigned)((int64_t)batch * n_max);
  return launch_pdl(sample_target_kernel, dim3(rows), dim3(kSampleThreads), 0, s, logits, uniforms,
                    kLog2eS / temperature, n_max, vocab, n_nodes, targ, err);
}

}  // namespace cure
