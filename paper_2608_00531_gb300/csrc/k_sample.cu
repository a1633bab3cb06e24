// Stochastic verification (temperature T > 0): the target's token at every
// tree node drawn from softmax(logits / T) by inverse CDF with a uniform the
// caller supplies.  Speculative decoding is lossless sampling from the target
// (Sec. 2); the paper's own runs are greedy (Sec. 4.1), where the argmax of
// cure_accept takes this kernel's place.  The acceptance walk is the same in
// both cases: a child is accepted when its token equals the parent's sample.
//
// One CTA per (sequence, node) row; thread t owns the contiguous ids
// [t * chunk, (t + 1) * chunk):
//   1. the row max m, from the threads' chunk maxima;
//   2. each chunk's sum of p_v = 2^((l_v - m) log2(e) / T), and an exclusive
//      scan of the chunk sums over the threads: chunk t covers the cumulative
//      range [E_t, E_t + S_t), the row total is Z;
//   3. r = u Z; the last chunk with mass whose E_t <= r walks its ids again in
//      the same order from E_t and takes the first id whose running sum
//      exceeds r (its last id with mass if rounding leaves r past its end).
#include "common.cuh"

namespace cure {
namespace {

constexpr int kSampleThreads = 512;
constexpr int kSampleWarps = kSampleThreads / 32;
constexpr float kLog2eS = 1.4426950408889634f;

__device__ __forceinline__ float ex2s(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float bf16_to_f32(uint16_t h) { return __uint_as_float((uint32_t)h << 16); }

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
  const uint16_t* x = logits + row * (int64_t)vocab;
  const int chunk = (vocab + kSampleThreads - 1) / kSampleThreads;
  const int v0 = min(vocab, tid * chunk), v1 = min(vocab, v0 + chunk);
  __shared__ float s_warp[kSampleWarps];
  __shared__ int s_owner;

  // 1. row max
  float m = -INFINITY;
  for (int v = v0; v < v1; ++v) m = fmaxf(m, bf16_to_f32(x[v]));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  if (lane == 0) s_warp[warp] = m;
  if (tid == 0) s_owner = -1;
  __syncthreads();
  m = s_warp[0];
#pragma unroll
  for (int w = 1; w < kSampleWarps; ++w) m = fmaxf(m, s_warp[w]);
  if (m == -INFINITY) {  // no finite logit: id 0, as the argmax's tie rule gives
    if (tid == 0) targ[row] = 0;
    return;
  }
  __syncthreads();  // every thread has read s_warp before it is reused

  // 2. chunk sums, their exclusive scan and the total
  const float nm = -m * scale;
  float sum = 0.f;
  for (int v = v0; v < v1; ++v) sum += ex2s(fmaf(bf16_to_f32(x[v]), scale, nm));
  float inc = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float y = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc += y;
  }
  float exc = __shfl_up_sync(0xffffffffu, inc, 1);
  if (lane == 0) exc = 0.f;
  if (lane == 31) s_warp[warp] = inc;
  __syncthreads();
  float base = 0.f, total = 0.f;
#pragma unroll
  for (int w = 0; w < kSampleWarps; ++w) {
    const float sw = s_warp[w];
    if (w < warp) base += sw;
    total += sw;
  }
  const float start = base + exc;
  float u = uniforms[row];
  u = fminf(fmaxf(u, 0.f), 0x1.fffffep-1f);  // [0, 1); NaN -> 0
  const float r = u * total;

  // 3. the owning chunk walks its ids
  if (sum > 0.f && start <= r) atomicMax(&s_owner, tid);
  __syncthreads();
  if (tid == s_owner) {
    float acc = start;
    int y = -1, last = -1;
    for (int v = v0; v < v1; ++v) {
      const float p = ex2s(fmaf(bf16_to_f32(x[v]), scale, nm));
      if (p > 0.f) {
        last = v;
        if (acc + p > r) {
          y = v;
          break;
        }
      }
      acc += p;
    }
    targ[row] = y >= 0 ? y : last;
  }
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
