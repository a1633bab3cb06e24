"""Python binding of the C ABI (include/cure.h), one function per entry point.

Argument marshalling only: every stage runs in the CUDA kernels of
libcure.so.  Tensors must live on the current CUDA device; outputs are
allocated with torch when not given.  Calls are asynchronous on the current
torch stream (or the ``stream`` argument).
"""
from __future__ import annotations

import ctypes as C
from typing import Optional, Sequence

import torch

from . import _lib
from ._lib import KVDesc, TreeParams, check

DEVERR_PAGE, DEVERR_SLOT, DEVERR_NODES = _lib.DEVERR_PAGE, _lib.DEVERR_SLOT, _lib.DEVERR_NODES


def _stream(stream) -> C.c_void_p:
    s = torch.cuda.current_stream() if stream is None else stream
    return C.c_void_p(s.cuda_stream)


def _p(t: Optional[torch.Tensor]) -> C.c_void_p:
    if t is None:
        return C.c_void_p(0)
    if not t.is_cuda:
        raise ValueError("libcure takes CUDA tensors")
    if not t.is_contiguous():
        raise ValueError("libcure takes contiguous tensors")
    return C.c_void_p(t.data_ptr())


def _need(t: torch.Tensor, dtype, name: str) -> None:
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")


def kv_desc(heads_kv: int, head_dim: int, max_len: int, block_table: Optional[torch.Tensor] = None,
            page_size: int = 16, num_pages: int = 0) -> KVDesc:
    """Cache geometry: contiguous [B][max_len][Hkv][D], or paged [num_pages][page_size][Hkv][D]
    with block_table int32 [B][max_len] (then max_len counts pages)."""
    d = KVDesc()
    d.layout = 0 if block_table is None else 1
    d.heads_kv, d.head_dim, d.max_len = heads_kv, head_dim, max_len
    d.page_size = page_size
    d.num_pages = num_pages
    if block_table is not None:
        _need(block_table, torch.int32, "block_table")
        d.block_table = _p(block_table).value
        d._keep = block_table  # keep the table alive with the descriptor
    return d


def cure_score_draft(logits: torch.Tensor, topk: int, *, out=None, stream=None):
    """Stage 1 (Sec. 3.3, Eq. 2): (top_ids, top_vals, margin, logp1) per row."""
    _need(logits, torch.bfloat16, "logits")
    V = logits.shape[-1]
    lead = logits.shape[:-1]
    rows = logits.numel() // V if V else 0
    dev = logits.device
    if out is None:
        out = (torch.empty(*lead, topk, dtype=torch.int32, device=dev),
               torch.empty(*lead, topk, dtype=torch.float32, device=dev),
               torch.empty(*lead, dtype=torch.float32, device=dev),
               torch.empty(*lead, dtype=torch.float32, device=dev))
    ids, vals, margin, logp1 = out
    lib = _lib.load()
    check("cure_score_draft", lib.cure_score_draft(_p(logits), rows, V, topk, _p(ids), _p(vals),
                                                   _p(margin), _p(logp1), _stream(stream)))
    return ids, vals, margin, logp1


def tree_params(batch, block, topk, tau, budget, branches, repair_depth=1, max_ufp=0,
                margin_scale=0.0, branch_min=1, max_depth=0, beam=0) -> TreeParams:
    p = TreeParams()
    p.batch, p.block, p.topk, p.tau = batch, block, topk, float(tau)
    p.budget, p.branches, p.repair_depth, p.max_ufp = budget, branches, repair_depth, max_ufp
    p.margin_scale, p.branch_min = float(margin_scale), branch_min
    p.max_depth, p.beam = max_depth, beam
    return p


def cure_build_tree(top_ids: torch.Tensor, margin: torch.Tensor, root_tok: torch.Tensor,
                    cache_len: torch.Tensor, tau: float, budget: int, branches: int,
                    repair_depth: int = 1, redraft: Optional[torch.Tensor] = None,
                    max_ufp: int = 0, margin_scale: float = 0.0, branch_min: int = 1,
                    max_depth: int = 0, beam: int = 0, *, out=None, stream=None) -> dict:
    """Stages 2+3 (Sec. 3.1 Eq. 1, Sec. 3.3, Sec. 3.4): the flattened repair tree.

    margin_scale > 0 turns on the dynamic branch budget of Eq. (3): UFP i then
    offers b_i alternatives, from branch_min up to branches - 1.  max_depth and
    beam (0 = none) are the structural caps on repair branches (Sec. 3.3-3.4)."""
    _need(top_ids, torch.int32, "top_ids")
    _need(margin, torch.float32, "margin")
    B, K, k = top_ids.shape
    n_max = 1 + K + budget
    W = (n_max + 63) // 64
    dev = top_ids.device
    if out is None:
        out = dict(n_nodes=torch.empty(B, dtype=torch.int32, device=dev),
                   tok=torch.empty(B, n_max, dtype=torch.int32, device=dev),
                   pos=torch.empty(B, n_max, dtype=torch.int32, device=dev),
                   parent=torch.empty(B, n_max, dtype=torch.int32, device=dev),
                   depth=torch.empty(B, n_max, dtype=torch.int32, device=dev),
                   anc=torch.empty(B, n_max, W, dtype=torch.int64, device=dev),
                   ufp_pos=torch.empty(B, K, dtype=torch.int32, device=dev),
                   n_ufp=torch.empty(B, dtype=torch.int32, device=dev))
    p = tree_params(B, K, k, tau, budget, branches, repair_depth, max_ufp, margin_scale, branch_min,
                    max_depth, beam)
    lib = _lib.load()
    check("cure_build_tree", lib.cure_build_tree(
        C.byref(p), _p(top_ids), _p(margin), _p(root_tok), _p(cache_len), _p(redraft),
        _p(out["n_nodes"]), _p(out["tok"]), _p(out["pos"]), _p(out["parent"]), _p(out["depth"]),
        _p(out["anc"]), _p(out["ufp_pos"]), _p(out["n_ufp"]), _stream(stream)))
    return out


def cure_tree_attn_workspace_size(batch: int, n_max: int, heads_q: int, kv: KVDesc) -> int:
    return int(_lib.load().cure_tree_attn_workspace_size(batch, n_max, heads_q, C.byref(kv)))


def cure_tree_attn(q: torch.Tensor, tree_k: Optional[torch.Tensor], tree_v: Optional[torch.Tensor],
                   k_cache: torch.Tensor, v_cache: torch.Tensor, kv: KVDesc,
                   cache_len: torch.Tensor, n_nodes: torch.Tensor, anc: torch.Tensor,
                   scale: float, *, out: Optional[torch.Tensor] = None,
                   workspace: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Stage 4 (Sec. 3.2/3.4/3.5): tree-masked GQA attention for one layer.

    tree_k = tree_v = None: the in-place layout, node j's K/V rows at cache
    slot cache_len[b] + j."""
    for t, nm in ((q, "q"), (tree_k, "tree_k"), (tree_v, "tree_v"), (k_cache, "k_cache"),
                  (v_cache, "v_cache")):
        if t is not None or nm not in ("tree_k", "tree_v"):
            _need(t, torch.bfloat16, nm)
    B, n_max, Hq, D = q.shape
    if out is None:
        out = torch.empty_like(q)
    need = cure_tree_attn_workspace_size(B, n_max, Hq, kv)
    if workspace is None:
        workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=q.device)
    lib = _lib.load()
    check("cure_tree_attn", lib.cure_tree_attn(
        _p(q), _p(tree_k), _p(tree_v), _p(k_cache), _p(v_cache), C.byref(kv), _p(cache_len),
        _p(n_nodes), _p(anc), B, n_max, Hq, float(scale), _p(out), _p(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)))
    return out


def cure_accept(tree: dict, block: int, *, target_logits: Optional[torch.Tensor] = None,
                targ: Optional[torch.Tensor] = None, out=None, stream=None) -> dict:
    """Stage 5 (Sec. 3.5 Eq. 4): target argmax per node and the longest accepted path.

    Give ``target_logits`` (bf16 [B][n_max][V]) to compute the argmax, or
    ``targ`` (int32 [B][n_max]) already holding the target's tokens.
    """
    B, n_max = tree["tok"].shape
    dev = tree["tok"].device
    V = 0
    if target_logits is not None:
        _need(target_logits, torch.bfloat16, "target_logits")
        V = target_logits.shape[-1]
        if targ is None:
            targ = torch.empty(B, n_max, dtype=torch.int32, device=dev)
    elif targ is None:
        raise ValueError("cure_accept needs target_logits or targ")
    P = block + 2
    if out is None:
        out = dict(accept_len=torch.empty(B, dtype=torch.int32, device=dev),
                   best_node=torch.empty(B, dtype=torch.int32, device=dev),
                   path_nodes=torch.empty(B, P, dtype=torch.int32, device=dev),
                   out_tokens=torch.empty(B, P, dtype=torch.int32, device=dev),
                   diverge_depth=torch.empty(B, dtype=torch.int32, device=dev))
    lib = _lib.load()
    check("cure_accept", lib.cure_accept(
        _p(target_logits), _p(targ), B, n_max, V, block, _p(tree["n_nodes"]), _p(tree["tok"]),
        _p(tree["parent"]), _p(tree["depth"]), _p(tree["anc"]), _p(out["accept_len"]),
        _p(out["best_node"]), _p(out["path_nodes"]), _p(out["out_tokens"]),
        _p(out["diverge_depth"]), _stream(stream)))
    out["targ"] = targ
    return out


def cure_sample_target(target_logits: torch.Tensor, n_nodes: torch.Tensor, uniforms: torch.Tensor,
                       temperature: float, *, out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Stochastic verification (Sec. 2, T > 0): the target's token at every tree
    node sampled by inverse CDF with uniforms[b][j]; pass the result to
    cure_accept as ``targ`` (without target_logits) for the walk."""
    _need(target_logits, torch.bfloat16, "target_logits")
    _need(uniforms, torch.float32, "uniforms")
    B, n_max, V = target_logits.shape
    if out is None:
        out = torch.empty(B, n_max, dtype=torch.int32, device=target_logits.device)
    lib = _lib.load()
    check("cure_sample_target", lib.cure_sample_target(
        _p(target_logits), _p(uniforms), float(temperature), B, n_max, V, _p(n_nodes), _p(out),
        _stream(stream)))
    return out


def cure_lm_head_workspace_size(rows: int, vocab: int) -> int:
    return int(_lib.load().cure_lm_head_workspace_size(rows, vocab))


def cure_lm_head_argmax(hidden: torch.Tensor, w_lm: torch.Tensor, *, out_index: Optional[torch.Tensor] = None,
                        out: Optional[torch.Tensor] = None, workspace: Optional[torch.Tensor] = None,
                        stream=None) -> torch.Tensor:
    """Stage 5 fused with the LM head (Sec. 3.5, Sec. 4.1): the first argmax of
    hidden[r] . w_lm[v] over v for every row, without writing the logits.

    hidden bf16 [rows][d_model], w_lm bf16 [vocab][d_model].  ``out_index``
    (int32 [rows]) places row r at out.view(-1)[out_index[r]]; without it the
    result is int32 [rows].
    """
    _need(hidden, torch.bfloat16, "hidden")
    _need(w_lm, torch.bfloat16, "w_lm")
    rows, d = hidden.shape
    V = w_lm.shape[0]
    dev = hidden.device
    if out is None:
        out = torch.empty(rows, dtype=torch.int32, device=dev)
    lib = _lib.load()
    ws = int(lib.cure_lm_head_workspace_size(rows, V))
    if workspace is None or workspace.numel() < ws:
        workspace = torch.empty(max(ws, 256), dtype=torch.uint8, device=dev)
    check("cure_lm_head_argmax", lib.cure_lm_head_argmax(
        _p(hidden), _p(w_lm), rows, d, V, _p(out_index), _p(out), _p(workspace), workspace.numel(),
        _stream(stream)))
    return out


def cure_resync_kv(k_caches: Sequence[torch.Tensor], v_caches: Sequence[torch.Tensor], kv: KVDesc,
                   tree_k: Optional[torch.Tensor], tree_v: Optional[torch.Tensor], acc: dict,
                   cache_len_in: torch.Tensor, block: int, *, n_max: Optional[int] = None,
                   cache_len_out: Optional[torch.Tensor] = None, out=None, stream=None) -> dict:
    """Stage 6 (Sec. 3.5, Alg. 1): write the path into every layer's cache, realign the draft.

    tree_k/tree_v: bf16 [layers][B][n_max][Hkv][D], or None for the in-place
    layout (the path rows are then read from cache slots L + node, and only
    the rows past the divergence move; give n_max).
    """
    layers = len(k_caches)
    B = cache_len_in.shape[0]
    if n_max is None:
        if layers and tree_k is None:
            raise ValueError("cure_resync_kv: the in-place layout needs n_max")
        n_max = tree_k.shape[2] if layers else block + 1
    dev = cache_len_in.device
    P = block + 2
    if cache_len_out is None:
        cache_len_out = torch.empty_like(cache_len_in)
    if out is None:
        out = dict(draft_valid_len=torch.empty(B, dtype=torch.int32, device=dev),
                   replay_tokens=torch.empty(B, P, dtype=torch.int32, device=dev),
                   n_replay=torch.empty(B, dtype=torch.int32, device=dev))
    kp = (C.c_void_p * max(1, layers))(*[_p(t).value for t in k_caches])
    vp = (C.c_void_p * max(1, layers))(*[_p(t).value for t in v_caches])
    lib = _lib.load()
    check("cure_resync_kv", lib.cure_resync_kv(
        layers, kp, vp, C.byref(kv), _p(tree_k), _p(tree_v), B, n_max, block,
        _p(acc["path_nodes"]), _p(acc["accept_len"]), _p(acc["diverge_depth"]),
        _p(acc["out_tokens"]), _p(cache_len_in), _p(cache_len_out), _p(out["draft_valid_len"]),
        _p(out["replay_tokens"]), _p(out["n_replay"]), _stream(stream)))
    out["cache_len"] = cache_len_out
    return out


def cure_device_error(stream=None) -> int:
    """Synchronise and return (and clear) the device error word's bits."""
    bits = C.c_int32(0)
    code = _lib.load().cure_device_error(_stream(stream), C.byref(bits))
    if code not in (0, 4):
        check("cure_device_error", code)
    return int(bits.value)


def cure_selftest_wait_timeout(limit_cycles: int = 1 << 24, stream=None) -> None:
    """Runs the library's bounded wait on a barrier nothing completes (a
    failure-detection self-test); read the outcome with cure_device_error()."""
    check("cure_selftest_wait_timeout", _lib.load().cure_selftest_wait_timeout(int(limit_cycles), _stream(stream)))


def cure_status_string(code: int) -> str:
    return _lib.load().cure_status_string(code).decode()


def cure_abi_version() -> int:
    return int(_lib.load().cure_abi_version())
