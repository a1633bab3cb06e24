// cure_tree_attn_noalloc: tree attention for callers that cannot allocate
// device memory.
//
// Some callers only ever receive the buffers of their own inputs and outputs:
// a plugin inside an inference server whose allocator has already reserved
// nearly all of HBM for its KV cache, or a host framework that gives an
// extension no allocator at all.  They cannot cudaMalloc the split-KV
// workspace that cure_tree_attn takes.  This entry point runs the same kernels
// with that workspace placed in a fixed array of the library's own static
// device memory instead.
//
// The array below is CURE_NOALLOC_SCRATCH_BYTES (64 MiB).  Every GPU on which
// this part of the library is loaded keeps it until the process exits.  In
// host code `g_attn_scratch` is only a host-side stand-in for the symbol, not
// a device address: its device address is looked up with
// cudaGetSymbolAddress, with the device current, the first time a call runs
// in a given CUDA context, and that address is what the kernels receive.  The
// address is cached per device and keyed by the context's id, so a context
// that is reset and created again is looked up afresh.
#include <float.h>

#include "common.cuh"

namespace {

static __device__ __align__(256) unsigned char g_attn_scratch[CURE_NOALLOC_SCRATCH_BYTES];

}  // namespace

using namespace cure;

extern "C" cure_status cure_tree_attn_noalloc(const void* q, const void* tree_k, const void* tree_v,
                                              const void* k_cache, const void* v_cache,
                                              const cure_kv_desc* kv, const int32_t* cache_len,
                                              const int32_t* n_nodes, const uint64_t* anc,
                                              int32_t batch, int32_t n_max, int32_t heads_q,
                                              float scale, void* out, void* stream) {
  ApiRange range("cure_tree_attn_noalloc");
  if (!kv) return CURE_ERR_INVALID_ARG;
  if (kv->layout != 0 && kv->layout != 1) return CURE_ERR_INVALID_ARG;
  if (kv->heads_kv < 1 || kv->max_len < 0) return CURE_ERR_INVALID_ARG;
  if (kv->head_dim != 128) return CURE_ERR_UNSUPPORTED;
  if (kv->layout == 1 &&
      (kv->page_size < 1 || kv->num_pages < 1 || !kv->block_table ||
       (int64_t)kv->max_len * kv->page_size > INT32_MAX ||
       (int64_t)kv->num_pages * kv->page_size > INT32_MAX))
    return CURE_ERR_INVALID_ARG;
  if (kv->layout == 1 && kv->page_size != 8 && kv->page_size != 16 && kv->page_size != 32 &&
      kv->page_size != 64)
    return CURE_ERR_UNSUPPORTED;
  if (batch < 0 || n_max < 1 || heads_q < 1 || heads_q % kv->heads_kv != 0 ||
      !(scale > 0.f && scale <= FLT_MAX))
    return CURE_ERR_INVALID_ARG;
  if (n_max > kMaxNodes || batch > kAttnBatchLimit || heads_q / kv->heads_kv > 128)
    return CURE_ERR_UNSUPPORTED;
  if (batch == 0) return CURE_OK;
  // tree_k and tree_v both NULL: the in-place layout, as in cure_tree_attn
  if (!q || !tree_k != !tree_v || !k_cache || !v_cache || !cache_len || !n_nodes || !anc || !out)
    return CURE_ERR_INVALID_ARG;
  const uintptr_t mis = reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(tree_k) |
                        reinterpret_cast<uintptr_t>(tree_v) | reinterpret_cast<uintptr_t>(k_cache) |
                        reinterpret_cast<uintptr_t>(v_cache) | reinterpret_cast<uintptr_t>(out);
  if ((mis & 15) != 0 || (reinterpret_cast<uintptr_t>(anc) & 7) != 0) return CURE_ERR_INVALID_ARG;
  AttnPlan plan;
  if (!plan_tree_attn(batch, n_max, heads_q, *kv, &plan)) return CURE_ERR_INVALID_ARG;
  // the shape's split-KV partials must fit in the static array
  if (plan.total() > (size_t)CURE_NOALLOC_SCRATCH_BYTES) return CURE_ERR_CAPACITY;
  static SymbolCache* cache = new_symbol_cache();
  void* scratch = nullptr;
  if (device_symbol_address(cache, g_attn_scratch, &scratch) != cudaSuccess) return CURE_ERR_CUDA;
  // Nothing in the array is cleared.  Its front holds the split units' piece
  // counters: every launch tags its counter words with a fresh launch number,
  // a word carrying another launch's tag counts as zero, and a unit whose
  // pieces have all arrived writes zero back.  Every partial result that is
  // read back was written earlier in the same launch.
  const cudaError_t e = launch_tree_attn(
      plan, static_cast<const uint16_t*>(q), static_cast<const uint16_t*>(tree_k),
      static_cast<const uint16_t*>(tree_v), static_cast<const uint16_t*>(k_cache),
      static_cast<const uint16_t*>(v_cache), *kv, cache_len, n_nodes, anc, batch, n_max, heads_q,
      scale, static_cast<uint16_t*>(out), scratch, device_error_word(),
      static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? CURE_OK : CURE_ERR_CUDA;
}
