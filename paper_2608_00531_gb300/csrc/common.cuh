// Internal declarations shared by the translation units of libcure.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/cure.h"

namespace cure {

constexpr int kMaxNodes = 256;     // n_max limit: 4 ancestor words
constexpr int kMaxLayers = 128;    // resync: layers passed by value
constexpr int kAttnBatchLimit = 256;  // tree attention: sequences per call

// An NVTX range named after the entry point, for the duration of the host
// call (header-only NVTX: a no-op unless a profiler's tool is attached).
struct ApiRange {
  explicit ApiRange(const char* name);
  ~ApiRange();
};

// Device error word of the current device (see cure_device_error).
int* device_error_word();
int num_sms();

// Device address of a __device__ variable of this library in the current
// device's current context.  The address belongs to the context (a reset or
// a re-created primary context gets a new one), so the cache is keyed by the
// driver's unique context id, and looked up again whenever that id changes or
// cannot be read.  `symbol` is the variable's host-side stand-in.
struct SymbolCache;
SymbolCache* new_symbol_cache();
cudaError_t device_symbol_address(SymbolCache* cache, const void* symbol, void** out);

__device__ __forceinline__ void flag(int* err, int bits) {
  if (err) atomicOr(err, bits);
}

// ---- programmatic dependent launch ----
// The library's kernels are launched so that each may be scheduled while the
// previous kernel on the stream finishes (its set-up then overlaps that
// kernel's tail); every kernel calls pdl_begin() before its first read of
// global memory, which waits for the previous kernel to complete and lets
// the next one be scheduled.  Without a programmatic launch both are no-ops.
__device__ __forceinline__ void pdl_begin() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// ---- launchers (all asynchronous on `s`; return the launch's cudaError_t) ----
cudaError_t launch_score(const uint16_t* logits, int64_t rows, int vocab, int topk,
                         int32_t* top_ids, float* top_vals, float* margin, float* logp1,
                         cudaStream_t s);
// Target argmax over rows (b, j) with j < n_nodes[b]; other rows get -1.
cudaError_t launch_target_argmax(const uint16_t* logits, int batch, int n_max, int vocab,
                                 const int32_t* n_nodes, int32_t* targ, cudaStream_t s);
// Target token sampled at temperature T > 0 over rows (b, j) with j < n_nodes[b]
// (inverse CDF with uniforms[b][j]); other rows get -1.
cudaError_t launch_sample_target(const uint16_t* logits, const float* uniforms, float temperature,
                                 int batch, int n_max, int vocab, const int32_t* n_nodes, int32_t* targ,
                                 int* err, cudaStream_t s);

cudaError_t launch_build_tree(const cure_tree_params& p, const int32_t* top_ids,
                              const float* margin, const int32_t* root_tok,
                              const int32_t* cache_len, const int32_t* redraft, int32_t* n_nodes,
                              int32_t* tok, int32_t* pos, int32_t* parent, int32_t* depth,
                              uint64_t* anc, int32_t* ufp_pos, int32_t* n_ufp, int* err,
                              cudaStream_t s);

cudaError_t launch_accept_walk(int batch, int n_max, int block, const int32_t* n_nodes,
                               const int32_t* tok, const int32_t* parent, const int32_t* depth,
                               const uint64_t* anc, const int32_t* targ, int32_t* accept_len,
                               int32_t* best_node, int32_t* path_nodes, int32_t* out_tokens,
                               int32_t* diverge_depth, int* err, cudaStream_t s);

struct LayerPtrs {
  void* k[kMaxLayers];
  void* v[kMaxLayers];
};

cudaError_t launch_resync(int layers, const LayerPtrs& caches, const cure_kv_desc& kv,
                          const uint16_t* tree_k, const uint16_t* tree_v, int batch, int n_max,
                          int block, const int32_t* path_nodes, const int32_t* accept_len,
                          const int32_t* diverge_depth, const int32_t* out_tokens,
                          const int32_t* cache_len_in, int32_t* cache_len_out,
                          int32_t* draft_valid_len, int32_t* replay_tokens, int32_t* n_replay,
                          int* err, cudaStream_t s);

// Fused LM head + argmax: launch plan for a shape (persistent CTAs, one
// 128-row M tile each, the vocabulary's 128-id halves split into `groups`
// ranges).
struct LmPlan {
  int m_tiles = 0, h_tiles = 0, groups = 0;
  size_t ws_bytes = 0;  // per-range (max, id) partials: groups * rows * 8 bytes
};
LmPlan plan_lm_head(int rows, int vocab);
cudaError_t launch_lm_head_argmax(const LmPlan& p, const uint16_t* hidden, const uint16_t* w_lm, int rows, int d,
                                  int vocab, int32_t* out, const int32_t* out_index, void* workspace, int* err,
                                  cudaStream_t s);

// Tree attention: workspace layout for a shape.
struct AttnPlan {
  int units_max;   // (sequence, kv head, row group) units at n_max
  size_t ws_cnt;   // bytes of per-unit piece counters (256-byte rounded)
  size_t ws_o;     // bytes of partial outputs
  size_t ws_lse;   // bytes of partial log-sum-exps
  size_t total() const { return ws_cnt + ws_o + ws_lse; }
};
bool plan_tree_attn(int batch, int n_max, int heads_q, const cure_kv_desc& kv, AttnPlan* plan);

cudaError_t launch_tree_attn(const AttnPlan& plan, const uint16_t* q, const uint16_t* tree_k,
                             const uint16_t* tree_v, const uint16_t* k_cache,
                             const uint16_t* v_cache, const cure_kv_desc& kv,
                             const int32_t* cache_len, const int32_t* n_nodes,
                             const uint64_t* anc, int batch, int n_max, int heads_q, float scale,
                             uint16_t* out, void* workspace, int* err, cudaStream_t s);

}  // namespace cure
