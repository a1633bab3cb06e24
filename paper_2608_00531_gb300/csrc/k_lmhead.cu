// Stage 5 fused with the target's LM head (Sec. 3.5, Eq. 4; greedy decoding,
// Sec. 4.1): the target's greedy token at every tree node computed from the
// node's final hidden state, as the epilogue of the LM-head contraction
//   logits[r][v] = hidden[r] . w_lm[v],   targ[r] = first argmax_v logits[r][v],
// so that the rows x vocab logits never reach HBM.
//
// The contraction runs on the tcgen05 tensor cores: one persistent CTA per SM
// owns one 128-row M tile of `hidden` and a contiguous range of the vocabulary
// in 128-id halves, taken as 256-id (N) tiles and, for an odd count, one
// 128-id tile at its end; the CTAs that share a vocab range run side by side,
// so each weight tile is read from HBM about once and served to the other M
// tiles from L2.
//   warp 0   producer: TMA loads of the 64-wide K slices of the hidden tile
//            [128 x 64] and of the weight tile [256 x 64] (128-byte swizzle)
//            into a 4-stage ring;
//   warp 1   MMA issuer (one lane): per K slice four M128 N256 K16 bf16
//            products accumulating in float32 in TMEM; two accumulators of
//            256 columns alternate between N tiles;
//   warps 2-5 epilogue: each thread owns one TMEM lane (one row), reads the
//            finished accumulator 32 columns at a time and keeps the row's
//            running (max, first id), strictly greater replacing, so the lowest
//            id wins ties; then frees the accumulator for the tile after next.
// Each CTA writes one (max, id) per row for its vocab range; a second kernel
// takes the first maximum over the ranges in vocab order.  Waits are bounded:
// on expiry a CTA flags CURE_DEVERR_TIMEOUT, drains its copies and products,
// frees its TMEM and leaves.
#include <cudaTypedefs.h>
#include <float.h>

#include <atomic>

#include "common.cuh"
#include "tc_ptx.cuh"

namespace cure {
namespace {

using namespace tc;

constexpr int BM = 128;           // rows per M tile (TMEM lanes)
constexpr int BN = 256;           // vocab ids per N tile (accumulator columns)
constexpr int BK = 64;            // K slice: one 128-byte swizzled row
constexpr int NS = 4;             // ring stages
constexpr int kThreads = 192;     // 6 warps
constexpr uint32_t kTmemCols = 512;
constexpr int kABytes = BM * BK * 2;       // 16 KiB
constexpr int kBBytes = BN * BK * 2;       // 32 KiB
constexpr int kStage = kABytes + kBBytes;  // 48 KiB
constexpr int kOffBars = NS * kStage;      // 196608
enum { B_FULL = 0, B_EMPTY = NS, B_ACCFULL = 2 * NS, B_ACCEMPTY = 2 * NS + 2, B_DRAIN = 2 * NS + 4,
       kNumBars = 2 * NS + 5 };
constexpr int kOffTmemSlot = kOffBars + 8 * kNumBars;
constexpr int kOffAbort = kOffTmemSlot + 4;
constexpr int kSmemUsed = kOffAbort + 4;
constexpr int kSmemBytes = kSmemUsed + 1024;  // room to align the base to 1024 bytes
static_assert(kSmemBytes <= 232448, "fits the 227 KiB opt-in");

struct LmArgs {
  int M, d, V;
  int m_tiles, groups, h_tiles;  // M tiles, vocab ranges, 128-id vocab halves
  float* part_val;   // [groups][M]
  int32_t* part_idx; // [groups][M]
  int* err;
};

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint32_t bar, int c0, int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1)
      : "memory");
}

// Four M128 N256 K16 products over one 64-wide K slice (descriptors step by
// 32 bytes, 2 in 16-byte units, inside the 128-byte swizzled rows).
__device__ __forceinline__ void mma_kslice(uint32_t d, uint64_t ad, uint64_t bd, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p0, pt;\n\t.reg .b64 a, b;\n\t"
      "setp.ne.b32 p0, %4, 0;\n\t"
      "setp.eq.b32 pt, %4, %4;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p0;\n\t"
      "add.s64 a, %1, 2;\n\tadd.s64 b, %2, 2;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %3, pt;\n\t"
      "add.s64 a, %1, 4;\n\tadd.s64 b, %2, 4;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %3, pt;\n\t"
      "add.s64 a, %1, 6;\n\tadd.s64 b, %2, 6;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %3, pt;\n\t}\n" ::"r"(d),
      "l"(ad), "l"(bd), "r"(idesc), "r"(acc)
      : "memory");
}

__global__ void __launch_bounds__(kThreads, 1)
lm_head_argmax_kernel(const __grid_constant__ CUtensorMap mh, const __grid_constant__ CUtensorMap mw,
                      const LmArgs A) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t sb = (raw + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (sb - raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  auto bar = [&](int i) { return sb + kOffBars + 8u * (uint32_t)i; };
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + kOffAbort);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + kOffTmemSlot);

  const int m_tile = blockIdx.x % A.m_tiles;
  const int g = blockIdx.x / A.m_tiles;
  const int h_lo = (int)((int64_t)g * A.h_tiles / A.groups);
  const int h_hi = (int)((int64_t)(g + 1) * A.h_tiles / A.groups);
  const int ntl = (h_hi - h_lo + 1) / 2;  // N tiles: 256 ids, the last one 128 for an odd count
  auto wide = [&](int t) { return h_hi - h_lo - 2 * t >= 2; };
  const int KS = A.d / BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(bar(B_FULL + s), 1);
      mbar_init(bar(B_EMPTY + s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(bar(B_ACCFULL + a), 1);
      mbar_init(bar(B_ACCEMPTY + a), 4);  // one arrival per epilogue warp
    }
    mbar_init(bar(B_DRAIN), 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&mh);
    tma_prefetch_desc(&mw);
  }
  if (warp == 1) tmem_alloc(sb + kOffTmemSlot, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_begin();

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      int it = 0;
      bool ok = true;
      for (int t = 0; t < ntl && ok; ++t) {
        const int v0 = (h_lo + 2 * t) * 128;
        for (int k = 0; k < KS; ++k, ++it) {
          const int s = it % NS;
          if (it >= NS && !wait_bounded(bar(B_EMPTY + s), ((it / NS) & 1) ^ 1, abort_flag, A.err, true)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(bar(B_FULL + s), kStage);
          const uint32_t st = sb + s * kStage;
          tma_load_2d(st, &mh, bar(B_FULL + s), k * BK, m_tile * BM);
          // a 128-id tile still loads a whole box; its second half goes unused
          tma_load_2d(st + kABytes, &mw, bar(B_FULL + s), k * BK, v0);
        }
      }
      if (!ok) {  // let the copies in flight land before the CTA's smem goes away
        for (int j = max(0, it - NS); j < it; ++j)
          wait_bounded(bar(B_FULL + j % NS), (j / NS) & 1, abort_flag, A.err, false);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_w = idesc_bf16_f32(BM, BN, false);
      constexpr uint32_t idesc_h = idesc_bf16_f32(BM, BN / 2, false);
      int it = 0;
      bool ok = true;
      for (int t = 0; t < ntl && ok; ++t) {
        const int a = t & 1;
        if (t >= 2 && !wait_bounded(bar(B_ACCEMPTY + a), ((t >> 1) & 1) ^ 1, abort_flag, A.err, true)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t idesc = wide(t) ? idesc_w : idesc_h;
        for (int k = 0; k < KS; ++k, ++it) {
          const int s = it % NS;
          if (!wait_bounded(bar(B_FULL + s), (it / NS) & 1, abort_flag, A.err, true)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t st = sb + s * kStage;
          mma_kslice(tmem + a * BN, sdesc_sw128(st, 16, 1024), sdesc_sw128(st + kABytes, 16, 1024), idesc,
                     k > 0 ? 1u : 0u);
          mma_commit(bar(B_EMPTY + s));
        }
        if (ok) mma_commit(bar(B_ACCFULL + a));
      }
      // every product issued has completed before TMEM is freed
      mma_commit(bar(B_DRAIN));
      wait_bounded(bar(B_DRAIN), 0, abort_flag, A.err, false);
    }
  } else {
    // ---------------------------------------------------------------- epilogue
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    const int row = m_tile * BM + q * 32 + lane;
    float best = -INFINITY;
    int bi = -1;
    for (int t = 0; t < ntl; ++t) {
      const int a = t & 1;
      const bool ok = wait_bounded(bar(B_ACCFULL + a), (t >> 1) & 1, abort_flag, A.err, true);
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      const int v0 = (h_lo + 2 * t) * 128;
      const int nc = wide(t) ? BN / 32 : BN / 64;
#pragma unroll 1
      for (int c = 0; c < nc; ++c) {
        uint32_t r[32];
        tmem_ld32(tmem + ((uint32_t)(q * 32) << 16) + a * BN + c * 32, r);
        tmem_wait_ld();
        const int vc = v0 + c * 32;
        if (vc + 32 <= A.V) {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const float x = __uint_as_float(r[j]);
            if (x > best) {
              best = x;
              bi = vc + j;
            }
          }
        } else {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const float x = __uint_as_float(r[j]);
            if (vc + j < A.V && x > best) {
              best = x;
              bi = vc + j;
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(B_ACCEMPTY + a));
    }
    if (row < A.M && !*abort_flag) {
      A.part_val[(int64_t)g * A.M + row] = best;
      A.part_idx[(int64_t)g * A.M + row] = bi;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// The first maximum over the vocab ranges, in vocab order.
__global__ void __launch_bounds__(256)
lm_head_reduce_kernel(const float* __restrict__ part_val, const int32_t* __restrict__ part_idx, int groups, int M,
                      int32_t* __restrict__ out, const int32_t* __restrict__ out_index) {
  pdl_begin();
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= M) return;
  float best = -INFINITY;
  int bi = -1;
  for (int g = 0; g < groups; ++g) {
    const float v = part_val[(int64_t)g * M + r];
    const int i = part_idx[(int64_t)g * M + r];
    if (i >= 0 && (bi < 0 || v > best)) {
      best = v;
      bi = i;
    }
  }
  out[out_index ? out_index[r] : r] = bi < 0 ? 0 : bi;
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

// [rows][d] bf16, K-major: boxes of 64 (K) x box_rows, 128-byte swizzle.
bool make_rows_map(CUtensorMap* m, const void* base, uint64_t rows, int d, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)d * 2};
  cuuint32_t box[2] = {BK, (cuuint32_t)box_rows};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

LmPlan plan_lm_head(int rows, int vocab) {
  LmPlan p;
  p.m_tiles = (rows + BM - 1) / BM;
  p.h_tiles = (vocab + 127) / 128;
  const int sms = num_sms();
  int groups = sms / (p.m_tiles > 0 ? p.m_tiles : 1);
  if (groups < 1) groups = 1;
  if (groups > p.h_tiles) groups = p.h_tiles;
  p.groups = groups;
  p.ws_bytes = ((size_t)groups * rows * (sizeof(float) + sizeof(int32_t)) + 255) / 256 * 256;
  return p;
}

cudaError_t launch_lm_head_argmax(const LmPlan& p, const uint16_t* hidden, const uint16_t* w_lm, int rows, int d,
                                  int vocab, int32_t* out, const int32_t* out_index, void* workspace, int* err,
                                  cudaStream_t s) {
  if (rows == 0) return cudaSuccess;
  static std::atomic<uint64_t> attr_done{0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(attr_done.load() & bit)) {
    e = cudaFuncSetAttribute(lm_head_argmax_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
    if (e != cudaSuccess) return e;
    attr_done.fetch_or(bit);
  }
  CUtensorMap mh, mw;
  if (!make_rows_map(&mh, hidden, (uint64_t)rows, d, BM) || !make_rows_map(&mw, w_lm, (uint64_t)vocab, d, BN))
    return cudaErrorInvalidValue;
  LmArgs a;
  a.M = rows;
  a.d = d;
  a.V = vocab;
  a.m_tiles = p.m_tiles;
  a.groups = p.groups;
  a.h_tiles = p.h_tiles;
  a.part_val = static_cast<float*>(workspace);
  a.part_idx = reinterpret_cast<int32_t*>(static_cast<char*>(workspace) + (size_t)p.groups * rows * sizeof(float));
  a.err = err;
  e = launch_pdl(lm_head_argmax_kernel, dim3(p.m_tiles * p.groups), dim3(kThreads), kSmemBytes, s, mh, mw, a);
  if (e != cudaSuccess) return e;
  e = launch_pdl(lm_head_reduce_kernel, dim3((rows + 255) / 256), dim3(256), 0, s, a.part_val, a.part_idx, p.groups,
                 rows, out, out_index);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace cure
