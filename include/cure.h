/*
 * cure.h — C ABI of the CURE repair-verify step on one GB300 (sm_103a).
 *
 * CURE ("Local Uncertainty Repair for Block-Parallel Speculative Decoding")
 * repairs a block-parallel draft at its low-margin positions and verifies the
 * draft and the repairs in one tree pass.  One decoding step of the method is
 * split into five calls (a sixth replaces the greedy argmax when verifying at
 * a temperature), each one CUDA kernel (or two) on the caller's stream:
 *
 *   cure_score_draft  Sec. 3.3, Eq. (2)     top-k ids, margin, top-1 log-prob
 *   cure_build_tree   Sec. 3.1 Eq. (1),     UFP gate + budgeted selection,
 *                     Sec. 3.3, 3.4         flattened repair tree + ancestor mask
 *   cure_tree_attn    Sec. 3.2, 3.4, 3.5    tree-masked GQA attention
 *   cure_accept       Sec. 3.5 Eq. (4)      target argmax + longest accepted path
 *   cure_lm_head_argmax Sec. 3.5, 4.1       the target's argmax per node straight from
 *                                           its hidden state (LM head + argmax fused)
 *   cure_sample_target Sec. 2 (T > 0)       the target's sampled token per node, for
 *                                           stochastic verification with cure_accept
 *   cure_resync_kv    Sec. 3.5, Alg. 1      write the path into the KV cache,
 *                                           realign the draft state
 *
 * Conventions shared by every call
 *  - Every pointer argument is a DEVICE pointer unless stated otherwise; the
 *    caller owns all memory (inputs, outputs, caches, workspace).  The library
 *    never allocates device memory.
 *  - `stream` is a cudaStream_t (NULL = the legacy default stream).  Calls are
 *    asynchronous; nothing waits on the host.
 *  - Arguments the host can check (sizes, null pointers, alignment) are
 *    checked before anything is launched; a bad one returns
 *    CURE_ERR_INVALID_ARG (or CURE_ERR_UNSUPPORTED for a valid but
 *    unimplemented shape) and launches nothing.
 *  - Conditions only the device can see (a cache slot past the capacity, a
 *    missing or out-of-range page id, a node count past n_max) make the kernel
 *    skip the offending access and raise a bit in a device error word;
 *    cure_device_error() reads and clears it.
 *  - Tensors are row-major, innermost dimension last.  bf16 is IEEE bfloat16.
 *  - Tie rule everywhere: equal values rank the lower index first.
 *  - Padding: entries of per-node outputs at j >= n_nodes[b] are -1 (ints) or
 *    0 (ancestor words); output rows of cure_tree_attn at j >= n_nodes[b] are
 *    left unwritten.
 */
#ifndef CURE_H_
#define CURE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  CURE_OK = 0,
  CURE_ERR_INVALID_ARG = 1,   /* a host-checkable argument is wrong; nothing launched */
  CURE_ERR_CAPACITY = 2,      /* workspace too small for the shape; nothing launched */
  CURE_ERR_CUDA = 3,          /* a CUDA runtime call or launch failed */
  CURE_ERR_DEVICE_FAULT = 4,  /* returned by cure_device_error when a kernel flagged bad data */
  CURE_ERR_UNSUPPORTED = 5    /* valid but not implemented (e.g. head_dim != 128) */
} cure_status;

/* Bits of the device error word (cure_device_error). */
#define CURE_DEVERR_PAGE      0x1   /* block_table entry < 0 or >= num_pages */
#define CURE_DEVERR_SLOT      0x2   /* cache slot beyond the per-sequence capacity */
#define CURE_DEVERR_NODES     0x4   /* n_nodes[b] outside [1, n_max] or a bad path/parent index */
#define CURE_DEVERR_TOKEN     0x8   /* a token id outside [0, vocab) where one is required */
#define CURE_DEVERR_TIMEOUT   0x10  /* a pipeline wait inside a kernel gave up (the CTA drained and left) */
#define CURE_DEVERR_ALIGN     0x20  /* a kernel found its shared memory misaligned and did nothing */

/* Tree-construction parameters (Sec. 3.3 / 3.4 and Eq. 1). */
typedef struct {
  int32_t batch;         /* B, sequences */
  int32_t block;         /* K, draft positions per block, 1..32 */
  int32_t topk;          /* ranked candidates stored per position by cure_score_draft, 2..8 */
  float tau;             /* margin threshold: position i is a UFP iff margin_i < tau (float32 compare) */
  int32_t budget;        /* R, maximum repair nodes per sequence, >= 0; n_max = 1 + K + R <= 256 */
  int32_t branches;      /* candidates per UFP counting the draft token: ranks 2..branches are
                            the alternatives; 1..topk */
  int32_t repair_depth;  /* 1: alternative leaf; 2: alternative + its re-drafted successor */
  int32_t max_ufp;       /* 0 = no cap; else only the max_ufp lowest-margin UFPs are repaired */
  float margin_scale;    /* s of Eq. (3); 0 = fixed budget (every UFP offers branches-1
                            alternatives); > 0 and finite = dynamic budget (see cure_build_tree) */
  int32_t branch_min;    /* b_min of Eq. (3), 0..branches-1 (the paper: 1); used when
                            margin_scale > 0 */
  int32_t max_depth;     /* 0 = none; else no repair node deeper than max_depth (the paper: 15) */
  int32_t beam;          /* 0 = none; else at most `beam` nodes at any depth (the paper: 5) */
} cure_tree_params;

/* KV-cache geometry (one layer). */
typedef struct {
  int32_t layout;        /* 0: contiguous [B][max_len][heads_kv][head_dim]
                            1: paged [num_pages][page_size][heads_kv][head_dim] */
  int32_t heads_kv;      /* Hkv */
  int32_t head_dim;      /* D; 128 is implemented */
  int32_t page_size;     /* paged: tokens per page: 8, 16, 32 or 64; ignored when contiguous */
  int32_t max_len;       /* contiguous: rows per sequence; paged: entries per block_table row */
  int32_t num_pages;     /* paged: pages in the pool (bounds check); ignored when contiguous */
  const int32_t* block_table; /* paged: device int32 [B][max_len] physical page ids; else NULL */
} cure_kv_desc;

/*
 * Stage 1 — draft scores (Sec. 3.3, Eq. 2; Alg. 1 first step).
 * For each of `rows` rows (B*K draft positions) of `vocab` bf16 logits:
 *   top_ids[r][0..topk)  ids ranked by (logit desc, id asc)        int32
 *   top_vals[r][0..topk) their logits widened to float32            float
 *   margin[r]            top_vals[r][0] - top_vals[r][1] (Eq. 2; the log-softmax
 *                        normaliser cancels, so it is also the log-prob gap)
 *   logp1[r]             top_vals[r][0] - logsumexp(row)  (float32 accumulation)
 * logits: bf16 [rows][vocab], any alignment.  2 <= topk <= 8, topk <= vocab.
 * margin and logp1 may be NULL.  NaN logits are not supported (ranking undefined);
 * -inf is allowed.
 */
cure_status cure_score_draft(const void* logits, int32_t rows, int32_t vocab, int32_t topk,
                             int32_t* top_ids, float* top_vals, float* margin, float* logp1,
                             void* stream);

/*
 * Stages 2+3 — UFP selection and repair-tree construction (Sec. 3.1 Eq. 1,
 * Sec. 3.3, Sec. 3.4; Alg. 1 loop).  One warp per sequence.
 * Inputs:  top_ids int32 [B][K][topk] and margin float [B][K] (from stage 1),
 *          root_tok int32 [B] (last committed token), cache_len int32 [B] (L_b),
 *          redraft int32 [B][K][branches-1]: the successor token of each
 *          alternative (rank r at index r-2) when repair_depth == 2 (NULL
 *          otherwise).
 * Selection: positions with margin < tau, in ascending (margin, position)
 *   order; each alternative (i, r), r = 2..branches, costs min(repair_depth, K-i)
 *   nodes and is admitted while the repair nodes stay <= budget (an alternative
 *   that does not fit is skipped).
 * Dynamic branch budget (Sec. 3.3, Eq. 3), when margin_scale s > 0: UFP i
 *   offers the b_i alternatives of ranks 2..b_i+1 instead, with
 *   u_i = clip(1 - m_i / s, 0, 1) and
 *   b_i = clip(round(b_min + u_i (b_max - b_min)), b_min, b_max),
 *   b_min = branch_min, b_max = branches - 1; the quotient, the difference, the
 *   product and the sum are float32 operations rounded to nearest and round()
 *   takes halves away from zero.  The paper's (b_min, b_max) = (1, 5) is
 *   branch_min = 1, branches = 6 (topk >= 6).
 * Structural caps (Sec. 3.3, 3.4; repair branches only, branch 0 is never
 *   pruned): with max_depth > 0 an alternative at depth i+1 > max_depth is not
 *   spawned and a successor at depth i+2 > max_depth is dropped (the
 *   alternative then costs one node); with beam > 0 an alternative is admitted
 *   only while every depth it occupies holds fewer than `beam` nodes, the chain
 *   node included (one that does not fit is skipped, like the budget).
 * Tree (n_max = 1 + K + budget nodes per sequence, W = ceil(n_max/64)):
 *   node 0 root (root_tok, depth 0); nodes 1..K branch 0 (top-1 ids, chained);
 *   then repair nodes in (i, r, depth) order: the rank-r id at position i as a
 *   child of node i, and with depth-2 repairs (i < K-1) its successor.
 * Outputs: n_nodes [B]; tok, pos (= L_b + depth), parent (-1 for the root),
 *   depth: int32 [B][n_max]; anc uint64 [B][n_max][W] (bit a of node j set iff a
 *   is on the root-to-j path, j included); ufp_pos int32 [B][K] (repaired
 *   positions in selection order, then -1); n_ufp int32 [B].
 * `p` is a HOST pointer.
 */
cure_status cure_build_tree(const cure_tree_params* p, const int32_t* top_ids, const float* margin,
                            const int32_t* root_tok, const int32_t* cache_len, const int32_t* redraft,
                            int32_t* n_nodes, int32_t* tok, int32_t* pos, int32_t* parent,
                            int32_t* depth, uint64_t* anc, int32_t* ufp_pos, int32_t* n_ufp,
                            void* stream);

/*
 * Stage 4 — tree attention for one layer (Sec. 3.2 / 3.4 / 3.5: the target
 * verifies every tree path in one pass).  For sequence b, node j < n_nodes[b],
 * query head h (kv head h / (heads_q / heads_kv)):
 *   out[b][j][h] = softmax(scale * q k^T) v over the cached keys 0..L_b-1 and
 *                  the tree keys a with bit a of anc[b][j] set.
 * q, out: bf16 [B][n_max][heads_q][D]; tree_k, tree_v: bf16 [B][n_max][heads_kv][D]
 * (this step's target keys/values of the tree tokens); k_cache, v_cache: one
 * layer in the layout of `kv` (a HOST pointer).
 * In-place layout: tree_k = tree_v = NULL means the tree rows were written
 * into the cache itself, node j of sequence b at slot L_b + j (a paged cache
 * then needs block_table entries up to slot L_b + n_b - 1).  The keys are then
 * one range 0..L_b+n_b-1 of the cache, in 64-key tiles; a tile past L_b
 * masks its tree part with the ancestor bits.  L_b + n_b past the capacity
 * sets CURE_DEVERR_SLOT.  Accumulation is float32; the
 * probabilities are rounded to bf16 before the PV product.  D = 128,
 * heads_q % heads_kv == 0, scale > 0 and finite (1/sqrt(D) in the paper's
 * models; otherwise CURE_ERR_INVALID_ARG), all tensor base pointers 16-byte
 * aligned.
 * workspace: device scratch of at least cure_tree_attn_workspace_size() bytes,
 * 256-byte aligned (split-KV partial results); its contents on entry do not
 * matter.  Calls that can overlap on the GPU must not share a workspace.
 * The kernel is launched as a programmatic dependent launch: it starts its
 * set-up while the previous kernel on the stream finishes and waits for that
 * kernel before reading any argument, so stream order is kept.
 */
cure_status cure_tree_attn(const void* q, const void* tree_k, const void* tree_v,
                           const void* k_cache, const void* v_cache, const cure_kv_desc* kv,
                           const int32_t* cache_len, const int32_t* n_nodes, const uint64_t* anc,
                           int32_t batch, int32_t n_max, int32_t heads_q, float scale, void* out,
                           void* workspace, size_t workspace_bytes, void* stream);

/* Bytes of workspace cure_tree_attn needs for this shape (0 on a bad argument). */
size_t cure_tree_attn_workspace_size(int32_t batch, int32_t n_max, int32_t heads_q,
                                     const cure_kv_desc* kv);

/* Size of the static device scratch behind cure_tree_attn_noalloc (64 MiB). */
#define CURE_NOALLOC_SCRATCH_BYTES (64u * 1024u * 1024u)

/*
 * cure_tree_attn without a caller-supplied workspace.  The paper has no
 * counterpart: this entry point exists for callers that cannot allocate
 * device memory — for instance a plugin in an inference server whose
 * allocator owns (and has nearly filled) HBM, or a host framework that hands
 * an extension only its input and output buffers.  It computes exactly what
 * cure_tree_attn computes, with the same arguments minus the workspace; the
 * split-KV partial results go to a 64 MiB array in the library's own static
 * device memory, which every GPU that loads that part of the library keeps
 * until the process exits.  It allocates nothing and calls no allocator.
 *  - Shapes whose cure_tree_attn_workspace_size() is larger than
 *    CURE_NOALLOC_SCRATCH_BYTES return CURE_ERR_CAPACITY and launch nothing.
 *  - The first call on each device looks up the device address of the array
 *    (cudaGetSymbolAddress); make that first call before any stream capture.
 *  - All calls share the one array and it keeps the last call's contents.
 *    Nothing in it needs to start at zero (each call writes every partial it
 *    reads), but two calls that can overlap on the GPU — on unordered streams
 *    or from different host threads — race on it and corrupt each other's
 *    outputs: order such calls on one stream.
 */
cure_status cure_tree_attn_noalloc(const void* q, const void* tree_k, const void* tree_v,
                                   const void* k_cache, const void* v_cache,
                                   const cure_kv_desc* kv, const int32_t* cache_len,
                                   const int32_t* n_nodes, const uint64_t* anc, int32_t batch,
                                   int32_t n_max, int32_t heads_q, float scale, void* out,
                                   void* stream);

/*
 * Stage 5 — acceptance walk (Sec. 3.5 Eq. 4, greedy decoding Sec. 4.1).
 * targ[b][j] = argmax_v target_logits[b][j][v] (lowest id on ties) for
 * j < n_nodes[b] (rows beyond are not read; their targ is -1).  Pass
 * target_logits (bf16 [B][n_max][vocab]) to have the argmax computed, or
 * target_logits = NULL and targ already filled with the target's tokens.
 * A non-root node j is verified when tok[j] == targ[parent[j]]; it is accepted
 * when every non-root node on its path is verified.  pi* = the deepest accepted
 * node (lowest index on ties), a = its depth.
 * Outputs (int32): accept_len [B] = a; best_node [B];
 *   path_nodes [B][K+2]: path node at each depth 0..a, then -1;
 *   out_tokens [B][K+2]: path tokens at depths 1..a, then targ[best] (the
 *                        token after the path), then -1;
 *   diverge_depth [B]: shallowest path depth whose node is a repair node
 *                      (index > K), or -1 when branch 0 wins.
 */
/*
 * Stage 5, stochastic verification (temperature > 0).  Speculative decoding is
 * lossless sampling from the target (Sec. 2); the paper's runs are greedy
 * (Sec. 4.1), where cure_accept's argmax fills targ.  This call fills targ
 * with samples instead, and cure_accept(target_logits = NULL, targ) then walks
 * the tree unchanged: a child is accepted when its token equals its parent's
 * sample.  Each sample is drawn independently of the drafted children, so the
 * emitted tokens follow the target's distribution.
 * For j < n_nodes[b]: targ[b][j] = the first id v with
 *   sum_{w <= v} softmax(target_logits[b][j] / temperature)_w > u,
 * u = uniforms[b][j] (float [B][n_max], clamped to [0, 1)), from float32
 * partial sums: within their rounding of the exact inverse CDF, never an id
 * of probability 0.  The probabilities are formed as 2^((l - l_max) log2(e)/T),
 * which cannot overflow: at temperatures so small that every logit below the
 * maximum underflows, the draw picks among the ids that hold the maximum
 * (the limit T -> 0).  A row of -inf logits gives 0; rows j >= n_nodes[b]
 * get -1.  target_logits bf16 [B][n_max][vocab], 2-byte aligned; temperature
 * > 0 with log2(e)/temperature finite (T >= about 4.2e-39, else
 * CURE_ERR_INVALID_ARG); 1 <= n_max <= 256.  One CTA of four warps per row,
 * each warp streaming a contiguous quarter of it.
 */
cure_status cure_sample_target(const void* target_logits, const float* uniforms, float temperature,
                               int32_t batch, int32_t n_max, int32_t vocab, const int32_t* n_nodes,
                               int32_t* targ, void* stream);

/*
 * Stage 5 fused with the target's LM head (Sec. 3.5, Eq. 4: the target scores
 * every tree node in one pass; greedy decoding, Sec. 4.1).  For each of `rows`
 * final hidden states (the tree nodes of all sequences, packed):
 *   targ[out_index ? out_index[r] : r] = the first v maximising hidden[r] . w_lm[v]
 * The contraction runs on the tensor cores with float32 accumulation and the
 * argmax is taken in its epilogue: the rows x vocab logits are never written.
 * Two ids whose logits lie within float32 accumulation error of each other may
 * be ranked either way (d_model products per logit; the bound is about
 * d_model/16 roundings of 2^-23 relative to sum_k |hidden[r][k] w_lm[v][k]|).
 * Then call cure_accept(target_logits = NULL, targ).
 * hidden: bf16 [rows][d_model]; w_lm: bf16 [vocab][d_model] (row-major, the
 * layout of an LM-head weight); both 16-byte aligned.  d_model a multiple of
 * 64 (else CURE_ERR_UNSUPPORTED).  out_index: int32 [rows] (NULL: identity),
 * e.g. b * n_max + j to fill cure_accept's targ [B][n_max] from rows packed over
 * the valid nodes; entries of targ that no row maps to are left unwritten.
 * workspace: at least cure_lm_head_workspace_size(rows, vocab) bytes (computed
 * for the current device), 256-byte aligned, contents on entry do not matter;
 * calls that can overlap on the GPU must not share one.  Two kernels: the
 * persistent tcgen05 contraction (one CTA per SM) and a per-row merge.
 */
cure_status cure_lm_head_argmax(const void* hidden, const void* w_lm, int32_t rows, int32_t d_model,
                                int32_t vocab, const int32_t* out_index, int32_t* targ, void* workspace,
                                size_t workspace_bytes, void* stream);

/* Bytes of workspace cure_lm_head_argmax needs on the current device (0 on a bad argument). */
size_t cure_lm_head_workspace_size(int32_t rows, int32_t vocab);

cure_status cure_accept(const void* target_logits, int32_t* targ, int32_t batch, int32_t n_max,
                        int32_t vocab, int32_t block, const int32_t* n_nodes, const int32_t* tok,
                        const int32_t* parent, const int32_t* depth, const uint64_t* anc,
                        int32_t* accept_len, int32_t* best_node, int32_t* path_nodes,
                        int32_t* out_tokens, int32_t* diverge_depth, void* stream);

/*
 * Stage 6 — repair resynchronisation (Sec. 3.5, Alg. 1 last step).
 * For every layer l and sequence b, the K/V rows of the accepted path's nodes
 * at depths 0..a are copied from tree_k/tree_v (bf16 [layers][B][n_max][Hkv][D])
 * into cache slots L_b..L_b+a of k_caches[l]/v_caches[l] (layout `kv`).
 * In-place layout (tree_k = tree_v = NULL, see cure_tree_attn): node j's rows
 * are read from cache slot L_b + j, so the rows of branch-0 nodes (j = depth)
 * are already in place and only the repair nodes past the divergence depth
 * are copied (nothing when branch 0 wins).
 * Then cache_len_out[b] = L_b + a + 1, draft_valid_len[b] = L_b + d when a
 * repair path wins at divergence depth d (else L_b + a + 1), and
 * replay_tokens[b] (int32 [B][K+2]) = the path tokens at depths d..a followed by
 * the token after the path (only that token on branch-0 wins), then -1;
 * n_replay[b] its length.  cache_len_out may alias cache_len_in; no other
 * output may overlap an input (the copies and the replay list are written by
 * one kernel, the lengths after it only when cache_len_out aliases).
 * k_caches, v_caches: HOST arrays of `layers` device pointers (layers <= 128).
 */
cure_status cure_resync_kv(int32_t layers, void* const* k_caches, void* const* v_caches,
                           const cure_kv_desc* kv, const void* tree_k, const void* tree_v,
                           int32_t batch, int32_t n_max, int32_t block, const int32_t* path_nodes,
                           const int32_t* accept_len, const int32_t* diverge_depth,
                           const int32_t* out_tokens, const int32_t* cache_len_in,
                           int32_t* cache_len_out, int32_t* draft_valid_len,
                           int32_t* replay_tokens, int32_t* n_replay, void* stream);

/* Reads and clears the device error word of the current device after
 * synchronising `stream`.  *bits receives the CURE_DEVERR_* bits (may be NULL).
 * Returns CURE_ERR_DEVICE_FAULT when any bit was set, CURE_OK otherwise. */
cure_status cure_device_error(void* stream, int32_t* bits);

/*
 * Failure-detection self-test (no counterpart in the paper): runs the
 * library's bounded pipeline wait, the one every kernel's barrier waits go
 * through, on a barrier that nothing ever completes, with a limit of
 * `limit_cycles` SM clock cycles (1 .. 2^30, the kernels' own limit).  The
 * wait gives up, raises CURE_DEVERR_TIMEOUT in the device error word and
 * returns; cure_device_error() then reports it, and the context stays usable.
 */
cure_status cure_selftest_wait_timeout(int64_t limit_cycles, void* stream);

/* Static description of a status code. */
const char* cure_status_string(cure_status s);

/* ABI version of this header (major * 100 + minor). */
int32_t cure_abi_version(void);

#ifdef __cplusplus
}
#endif
#endif /* CURE_H_ */
