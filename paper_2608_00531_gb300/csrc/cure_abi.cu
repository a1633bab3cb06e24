// The C ABI (include/cure.h): host-side argument checks, then the launches.
// Nothing here allocates device memory.
#include <cuda.h>
#include <float.h>
#include <nvtx3/nvToolsExt.h>

#include <mutex>

#include "common.cuh"

namespace cure {
namespace {

__device__ int g_err_word;  // device error word, one per device that loads the library

std::mutex g_mu;
int g_sms[64];

int current_device() {
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess) return 0;
  return d & 63;
}

inline bool aligned(const void* p, size_t a) {
  return (reinterpret_cast<uintptr_t>(p) % a) == 0;
}

inline cure_status from_cuda(cudaError_t e) { return e == cudaSuccess ? CURE_OK : CURE_ERR_CUDA; }

bool kv_ok(const cure_kv_desc* kv, cure_status* why) {
  *why = CURE_ERR_INVALID_ARG;
  if (!kv) return false;
  if (kv->layout != 0 && kv->layout != 1) return false;
  if (kv->heads_kv < 1 || kv->max_len < 0) return false;
  if (kv->head_dim != 128) {
    *why = CURE_ERR_UNSUPPORTED;
    return false;
  }
  if (kv->layout == 1) {
    if (kv->page_size < 1 || kv->num_pages < 1 || !kv->block_table) return false;
    if ((int64_t)kv->max_len * kv->page_size > INT32_MAX ||
        (int64_t)kv->num_pages * kv->page_size > INT32_MAX)
      return false;
    // a page is whole TMA boxes of a 64-key tile
    if (kv->page_size != 8 && kv->page_size != 16 && kv->page_size != 32 && kv->page_size != 64) {
      *why = CURE_ERR_UNSUPPORTED;
      return false;
    }
  }
  return true;
}

}  // namespace

// ---- context-keyed device addresses of the library's __device__ variables
namespace {

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);
CtxGetCurrentFn g_ctx_get_current = nullptr;
CtxGetIdFn g_ctx_get_id = nullptr;
std::once_flag g_ctx_once;

// The driver's id of the calling thread's current context; false when there
// is none or it cannot be read (the caller then does not cache).
bool current_context_id(unsigned long long* id) {
  std::call_once(g_ctx_once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      g_ctx_get_current = reinterpret_cast<CtxGetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      g_ctx_get_id = reinterpret_cast<CtxGetIdFn>(p);
  });
  if (!g_ctx_get_current || !g_ctx_get_id) return false;
  CUcontext c = nullptr;
  if (g_ctx_get_current(&c) != CUDA_SUCCESS || !c) return false;
  return g_ctx_get_id(c, id) == CUDA_SUCCESS;
}

}  // namespace

struct SymbolCache {
  std::mutex mu;
  unsigned long long ctx[64] = {};
  void* ptr[64] = {};
};

SymbolCache* new_symbol_cache() { return new SymbolCache(); }

cudaError_t device_symbol_address(SymbolCache* cache, const void* symbol, void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  unsigned long long id = 0;
  const bool have_id = current_context_id(&id);
  std::lock_guard<std::mutex> lk(cache->mu);
  if (have_id && cache->ptr[dev] && cache->ctx[dev] == id) {
    *out = cache->ptr[dev];
    return cudaSuccess;
  }
  void* p = nullptr;
  e = cudaGetSymbolAddress(&p, symbol);  // loads the module into the context if needed
  if (e != cudaSuccess) return e;
  // the look-up may have created the context: read its id again
  cache->ptr[dev] = current_context_id(&id) ? p : nullptr;
  cache->ctx[dev] = id;
  *out = p;
  return cudaSuccess;
}

ApiRange::ApiRange(const char* name) { nvtxRangePushA(name); }
ApiRange::~ApiRange() { nvtxRangePop(); }

int* device_error_word() {
  static SymbolCache* cache = new_symbol_cache();
  void* p = nullptr;
  if (device_symbol_address(cache, &g_err_word, &p) != cudaSuccess) return nullptr;
  return static_cast<int*>(p);
}

int num_sms() {
  const int d = current_device();
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_sms[d]) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, d) != cudaSuccess || v <= 0)
      v = 148;
    g_sms[d] = v;
  }
  return g_sms[d];
}

}  // namespace cure

using namespace cure;

extern "C" {

int32_t cure_abi_version(void) { return 105; }

const char* cure_status_string(cure_status s) {
  switch (s) {
    case CURE_OK: return "ok";
    case CURE_ERR_INVALID_ARG: return "invalid argument";
    case CURE_ERR_CAPACITY: return "workspace too small";
    case CURE_ERR_CUDA: return "CUDA error";
    case CURE_ERR_DEVICE_FAULT: return "device flagged bad data";
    case CURE_ERR_UNSUPPORTED: return "unsupported shape";
  }
  return "unknown status";
}

cure_status cure_score_draft(const void* logits, int32_t rows, int32_t vocab, int32_t topk,
                             int32_t* top_ids, float* top_vals, float* margin, float* logp1,
                             void* stream) {
  ApiRange range("cure_score_draft");
  if (rows < 0 || vocab < 2 || topk < 2 || topk > 8 || topk > vocab) return CURE_ERR_INVALID_ARG;
  if (rows > 65535) return CURE_ERR_UNSUPPORTED;
  if (rows == 0) return CURE_OK;
  if (!logits || !top_ids || !top_vals || !aligned(logits, 2)) return CURE_ERR_INVALID_ARG;
  return from_cuda(launch_score(static_cast<const uint16_t*>(logits), rows, vocab, topk, top_ids,
                                top_vals, margin, logp1, static_cast<cudaStream_t>(stream)));
}

cure_status cure_build_tree(const cure_tree_params* p, const int32_t* top_ids, const float* margin,
                            const int32_t* root_tok, const int32_t* cache_len, const int32_t* redraft,
                            int32_t* n_nodes, int32_t* tok, int32_t* pos, int32_t* parent,
                            int32_t* depth, uint64_t* anc, int32_t* ufp_pos, int32_t* n_ufp,
                            void* stream) {
  ApiRange range("cure_build_tree");
  if (!p) return CURE_ERR_INVALID_ARG;
  if (p->batch < 0 || p->block < 1 || p->block > 32 || p->topk < 2 || p->topk > 8 ||
      p->budget < 0 || p->branches < 1 || p->branches > p->topk ||
      (p->repair_depth != 1 && p->repair_depth != 2) || p->max_ufp < 0 ||
      !(p->margin_scale >= 0.f && p->margin_scale <= FLT_MAX) ||
      (p->margin_scale > 0.f && (p->branch_min < 0 || p->branch_min > p->branches - 1)) ||
      p->max_depth < 0 || p->beam < 0)
    return CURE_ERR_INVALID_ARG;
  if (1 + p->block + p->budget > kMaxNodes) return CURE_ERR_UNSUPPORTED;
  if (p->batch == 0) return CURE_OK;
  if (!top_ids || !margin || !root_tok || !cache_len || !n_nodes || !tok || !pos || !parent ||
      !depth || !anc || !ufp_pos || !n_ufp || !aligned(anc, 8))
    return CURE_ERR_INVALID_ARG;
  if (p->repair_depth == 2 && p->branches > 1 && !redraft) return CURE_ERR_INVALID_ARG;
  return from_cuda(launch_build_tree(*p, top_ids, margin, root_tok, cache_len, redraft, n_nodes,
                                     tok, pos, parent, depth, anc, ufp_pos, n_ufp,
                                     device_error_word(), static_cast<cudaStream_t>(stream)));
}

size_t cure_tree_attn_workspace_size(int32_t batch, int32_t n_max, int32_t heads_q,
                                     const cure_kv_desc* kv) {
  cure_status why;
  if (batch < 0 || n_max < 1 || n_max > kMaxNodes || heads_q < 1 || !kv_ok(kv, &why)) return 0;
  AttnPlan plan;
  if (!plan_tree_attn(batch, n_max, heads_q, *kv, &plan)) return 0;
  return plan.total();
}

cure_status cure_tree_attn(const void* q, const void* tree_k, const void* tree_v,
                           const void* k_cache, const void* v_cache, const cure_kv_desc* kv,
                           const int32_t* cache_len, const int32_t* n_nodes, const uint64_t* anc,
                           int32_t batch, int32_t n_max, int32_t heads_q, float scale, void* out,
                           void* workspace, size_t workspace_bytes, void* stream) {
  ApiRange range("cure_tree_attn");
  cure_status why;
  if (!kv_ok(kv, &why)) return why;
  if (batch < 0 || n_max < 1 || heads_q < 1 || heads_q % kv->heads_kv != 0 ||
      !(scale > 0.f && scale <= FLT_MAX))
    return CURE_ERR_INVALID_ARG;
  if (n_max > kMaxNodes || batch > kAttnBatchLimit || heads_q / kv->heads_kv > 128)
    return CURE_ERR_UNSUPPORTED;
  if (batch == 0) return CURE_OK;
  // tree_k and tree_v both NULL: the in-place layout (tree rows at cache slots L_b + j)
  if (!q || !tree_k != !tree_v || !k_cache || !v_cache || !cache_len || !n_nodes || !anc || !out ||
      !workspace)
    return CURE_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(tree_k, 16) || !aligned(tree_v, 16) || !aligned(k_cache, 16) ||
      !aligned(v_cache, 16) || !aligned(out, 16) || !aligned(workspace, 256) || !aligned(anc, 8))
    return CURE_ERR_INVALID_ARG;
  AttnPlan plan;
  if (!plan_tree_attn(batch, n_max, heads_q, *kv, &plan)) return CURE_ERR_INVALID_ARG;
  if (workspace_bytes < plan.total()) return CURE_ERR_CAPACITY;
  return from_cuda(launch_tree_attn(plan, static_cast<const uint16_t*>(q),
                                    static_cast<const uint16_t*>(tree_k),
                                    static_cast<const uint16_t*>(tree_v),
                                    static_cast<const uint16_t*>(k_cache),
                                    static_cast<const uint16_t*>(v_cache), *kv, cache_len, n_nodes,
                                    anc, batch, n_max, heads_q, scale, static_cast<uint16_t*>(out),
                                    workspace, device_error_word(),
                                    static_cast<cudaStream_t>(stream)));
}

cure_status cure_sample_target(const void* target_logits, const float* uniforms, float temperature,
                               int32_t batch, int32_t n_max, int32_t vocab, const int32_t* n_nodes,
                               int32_t* targ, void* stream) {
  ApiRange range("cure_sample_target");
  // log2(e) / T must be a finite float: T from about 4.2e-39 up
  if (batch < 0 || n_max < 1 || vocab < 1 || !(temperature > 0.f && temperature <= FLT_MAX) ||
      !(1.4426950408889634f / temperature <= FLT_MAX))
    return CURE_ERR_INVALID_ARG;
  if (n_max > kMaxNodes || (int64_t)batch * n_max > 65535) return CURE_ERR_UNSUPPORTED;
  if (batch == 0) return CURE_OK;
  if (!target_logits || !uniforms || !n_nodes || !targ || !aligned(target_logits, 2) ||
      !aligned(uniforms, 4))
    return CURE_ERR_INVALID_ARG;
  return from_cuda(launch_sample_target(static_cast<const uint16_t*>(target_logits), uniforms, temperature,
                                        batch, n_max, vocab, n_nodes, targ, device_error_word(),
                                        static_cast<cudaStream_t>(stream)));
}

size_t cure_lm_head_workspace_size(int32_t rows, int32_t vocab) {
  if (rows < 0 || vocab < 1) return 0;
  if (rows == 0) return 256;
  return plan_lm_head(rows, vocab).ws_bytes;
}

cure_status cure_lm_head_argmax(const void* hidden, const void* w_lm, int32_t rows, int32_t d_model,
                                int32_t vocab, const int32_t* out_index, int32_t* targ, void* workspace,
                                size_t workspace_bytes, void* stream) {
  ApiRange range("cure_lm_head_argmax");
  if (rows < 0 || d_model < 64 || vocab < 1) return CURE_ERR_INVALID_ARG;
  if (d_model % 64 != 0) return CURE_ERR_UNSUPPORTED;
  if (rows == 0) return CURE_OK;
  if (!hidden || !w_lm || !targ || !workspace || !aligned(hidden, 16) || !aligned(w_lm, 16) ||
      !aligned(workspace, 256) || !aligned(targ, 4) || !aligned(out_index, 4))
    return CURE_ERR_INVALID_ARG;
  const LmPlan plan = plan_lm_head(rows, vocab);
  if (workspace_bytes < plan.ws_bytes) return CURE_ERR_CAPACITY;
  return from_cuda(launch_lm_head_argmax(plan, static_cast<const uint16_t*>(hidden),
                                         static_cast<const uint16_t*>(w_lm), rows, d_model, vocab, targ,
                                         out_index, workspace, device_error_word(),
                                         static_cast<cudaStream_t>(stream)));
}

cure_status cure_accept(const void* target_logits, int32_t* targ, int32_t batch, int32_t n_max,
                        int32_t vocab, int32_t block, const int32_t* n_nodes, const int32_t* tok,
                        const int32_t* parent, const int32_t* depth, const uint64_t* anc,
                        int32_t* accept_len, int32_t* best_node, int32_t* path_nodes,
                        int32_t* out_tokens, int32_t* diverge_depth, void* stream) {
  ApiRange range("cure_accept");
  if (batch < 0 || n_max < 1 || block < 1 || block > 32 || n_max < block + 1)
    return CURE_ERR_INVALID_ARG;
  if (n_max > kMaxNodes) return CURE_ERR_UNSUPPORTED;
  if (batch == 0) return CURE_OK;
  if (!targ || !n_nodes || !tok || !parent || !depth || !anc || !accept_len || !best_node ||
      !path_nodes || !out_tokens || !diverge_depth || !aligned(anc, 8))
    return CURE_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int* err = device_error_word();
  if (target_logits) {
    if (vocab < 1 || !aligned(target_logits, 2)) return CURE_ERR_INVALID_ARG;
    if ((int64_t)batch * n_max > 65535) return CURE_ERR_UNSUPPORTED;
    const cudaError_t e = launch_target_argmax(static_cast<const uint16_t*>(target_logits), batch,
                                               n_max, vocab, n_nodes, targ, s);
    if (e != cudaSuccess) return CURE_ERR_CUDA;
  }
  return from_cuda(launch_accept_walk(batch, n_max, block, n_nodes, tok, parent, depth, anc, targ,
                                      accept_len, best_node, path_nodes, out_tokens, diverge_depth,
                                      err, s));
}

cure_status cure_resync_kv(int32_t layers, void* const* k_caches, void* const* v_caches,
                           const cure_kv_desc* kv, const void* tree_k, const void* tree_v,
                           int32_t batch, int32_t n_max, int32_t block, const int32_t* path_nodes,
                           const int32_t* accept_len, const int32_t* diverge_depth,
                           const int32_t* out_tokens, const int32_t* cache_len_in,
                           int32_t* cache_len_out, int32_t* draft_valid_len,
                           int32_t* replay_tokens, int32_t* n_replay, void* stream) {
  ApiRange range("cure_resync_kv");
  cure_status why;
  if (!kv_ok(kv, &why)) return why;
  if (layers < 0 || layers > kMaxLayers || batch < 0 || n_max < 1 || block < 1 || block > 32 ||
      n_max < block + 1)
    return CURE_ERR_INVALID_ARG;
  if (batch == 0) return CURE_OK;
  if (!path_nodes || !accept_len || !diverge_depth || !out_tokens || !cache_len_in ||
      !cache_len_out || !draft_valid_len || !replay_tokens || !n_replay)
    return CURE_ERR_INVALID_ARG;
  LayerPtrs lp;
  if (layers > 0) {
    // tree_k and tree_v both NULL: the in-place layout (tree rows at cache slots L_b + j)
    if (!k_caches || !v_caches || !tree_k != !tree_v || !aligned(tree_k, 16) ||
        !aligned(tree_v, 16))
      return CURE_ERR_INVALID_ARG;
    for (int l = 0; l < layers; ++l) {
      if (!k_caches[l] || !v_caches[l] || !aligned(k_caches[l], 16) || !aligned(v_caches[l], 16))
        return CURE_ERR_INVALID_ARG;
      lp.k[l] = k_caches[l];
      lp.v[l] = v_caches[l];
    }
  }
  return from_cuda(launch_resync(layers, lp, *kv, static_cast<const uint16_t*>(tree_k),
                                 static_cast<const uint16_t*>(tree_v), batch, n_max, block,
                                 path_nodes, accept_len, diverge_depth, out_tokens, cache_len_in,
                                 cache_len_out, draft_valid_len, replay_tokens, n_replay,
                                 device_error_word(), static_cast<cudaStream_t>(stream)));
}

cure_status cure_device_error(void* stream, int32_t* bits) {
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return CURE_ERR_CUDA;
  int v = 0;
  if (cudaMemcpyFromSymbol(&v, g_err_word, sizeof(int)) != cudaSuccess) return CURE_ERR_CUDA;
  const int zero = 0;
  if (cudaMemcpyToSymbol(g_err_word, &zero, sizeof(int)) != cudaSuccess) return CURE_ERR_CUDA;
  if (bits) *bits = v;
  return v ? CURE_ERR_DEVICE_FAULT : CURE_OK;
}

}  // extern "C"
