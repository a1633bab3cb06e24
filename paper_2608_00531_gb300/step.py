"""One CURE repair-verify step over a batch, through the C ABI.

``RepairVerifyStep`` owns the device buffers of every stage's outputs (and the
tree-attention workspace) for a fixed shape, and runs the six stages in order
on one stream:

  score_draft -> build_tree -> tree_attn x layers -> accept -> resync_kv

Inputs of a step (``StepInputs``) are the draft logits, the tree's target
Q/K/V per layer and the target logits; the KV caches are persistent state
owned by the caller.  Nothing here computes: every stage is a libcure call.

``run_from_host`` takes the same inputs in (pinned) host memory and streams
them in on a copy stream in the order the stages consume them (draft logits,
then each layer's Q/K/V, then the target logits of the tree's nodes); each
stage waits only for its own inputs, so the copies overlap the stages before
them.
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional

import torch

from . import cure


@dataclasses.dataclass
class StepInputs:
    draft_logits: torch.Tensor      # bf16 [B][K][V]
    root_tok: torch.Tensor          # int32 [B]
    cache_len: torch.Tensor         # int32 [B]
    redraft: Optional[torch.Tensor]  # int32 [B][K][branches-1] or None
    q: torch.Tensor                 # bf16 [layers][B][n_max][Hq][D]
    tree_k: torch.Tensor            # bf16 [layers][B][n_max][Hkv][D]
    tree_v: torch.Tensor            # bf16 [layers][B][n_max][Hkv][D]
    target_logits: torch.Tensor     # bf16 [B][n_max][V]


class RepairVerifyStep:
    # target logits of at least this many bytes are copied by node rows
    NODE_ROWS_MIN_BYTES = 64 << 20

    def __init__(self, batch: int, block: int, vocab: int, topk: int, tau: float, budget: int,
                 branches: int, repair_depth: int, layers: int, heads_q: int, kv: cure.KVDesc,
                 device: torch.device, max_ufp: int = 0, layer_map: Optional[List[int]] = None):
        self.B, self.K, self.V, self.k = batch, block, vocab, topk
        self.tau, self.R, self.branches, self.depth = tau, budget, branches, repair_depth
        self.max_ufp = max_ufp
        self.layers, self.Hq, self.kv = layers, heads_q, kv
        self.n_max = 1 + block + budget
        self.D = kv.head_dim
        self.scale = 1.0 / float(self.D) ** 0.5
        # logical layer -> physical cache index (aliasing when the caches of all
        # layers do not fit in device memory)
        self.layer_map = layer_map or list(range(layers))
        dev = device
        B, K, N = batch, block, self.n_max
        W = (N + 63) // 64
        i32 = dict(dtype=torch.int32, device=dev)
        self.score = (torch.empty(B, K, topk, **i32), torch.empty(B, K, topk, dtype=torch.float32, device=dev),
                      torch.empty(B, K, dtype=torch.float32, device=dev),
                      torch.empty(B, K, dtype=torch.float32, device=dev))
        self.tree = dict(n_nodes=torch.empty(B, **i32), tok=torch.empty(B, N, **i32),
                         pos=torch.empty(B, N, **i32), parent=torch.empty(B, N, **i32),
                         depth=torch.empty(B, N, **i32),
                         anc=torch.empty(B, N, W, dtype=torch.int64, device=dev),
                         ufp_pos=torch.empty(B, K, **i32), n_ufp=torch.empty(B, **i32))
        self.attn_out = torch.empty(layers, B, N, heads_q, self.D, dtype=torch.bfloat16, device=dev)
        ws = cure.cure_tree_attn_workspace_size(B, N, heads_q, kv)
        self.workspace = torch.empty(max(ws, 256), dtype=torch.uint8, device=dev)
        self.targ = torch.empty(B, N, **i32)
        P = K + 2
        self.acc = dict(accept_len=torch.empty(B, **i32), best_node=torch.empty(B, **i32),
                        path_nodes=torch.empty(B, P, **i32), out_tokens=torch.empty(B, P, **i32),
                        diverge_depth=torch.empty(B, **i32))
        self.rs = dict(draft_valid_len=torch.empty(B, **i32), replay_tokens=torch.empty(B, P, **i32),
                       n_replay=torch.empty(B, **i32))
        self.cache_len_out = torch.empty(B, **i32)
        self._dev_inputs = None
        self._copy_stream = None
        self._n_host = None
        self.last_h2d_bytes = 0  # host-to-device bytes of the last run_from_host

    def run(self, x: StepInputs, k_caches: List[torch.Tensor], v_caches: List[torch.Tensor],
            stream=None) -> dict:
        ids, vals, margin, logp1 = cure.cure_score_draft(x.draft_logits, self.k, out=self.score,
                                                         stream=stream)
        tree = cure.cure_build_tree(ids, margin, x.root_tok, x.cache_len, self.tau, self.R,
                                    self.branches, self.depth, x.redraft, self.max_ufp,
                                    out=self.tree, stream=stream)
        for l in range(self.layers):
            p = self.layer_map[l]
            cure.cure_tree_attn(x.q[l], x.tree_k[l], x.tree_v[l], k_caches[p], v_caches[p], self.kv,
                                x.cache_len, tree["n_nodes"], tree["anc"], self.scale,
                                out=self.attn_out[l], workspace=self.workspace, stream=stream)
        acc = cure.cure_accept(tree, self.K, target_logits=x.target_logits, targ=self.targ,
                               out=self.acc, stream=stream)
        kl = [k_caches[self.layer_map[l]] for l in range(self.layers)]
        vl = [v_caches[self.layer_map[l]] for l in range(self.layers)]
        rs = cure.cure_resync_kv(kl, vl, self.kv, x.tree_k, x.tree_v, acc, x.cache_len, self.K,
                                 cache_len_out=self.cache_len_out, out=self.rs, stream=stream)
        return dict(score=self.score, tree=tree, attn=self.attn_out, acc=acc, resync=rs)

    def run_from_host(self, xh: StepInputs, k_caches: List[torch.Tensor], v_caches: List[torch.Tensor],
                      stream=None) -> dict:
        """One step with its inputs in host memory (pinned, for copies that
        overlap the stages): copies on a side stream, each stage waiting for
        the copy of its own inputs.  When the target logits are large (at
        least NODE_ROWS_MIN_BYTES), only the rows of the tree's nodes are
        copied (rows j < n_nodes[b] of each sequence, the rows stage 5 reads):
        their count is known once the tree is built, so the host reads the
        node counts back before it queues those copies, behind the layers'
        Q/K/V.  Smaller ones are copied whole, without that read-back.
        Results stay on the device, as in run()."""
        fields = ("draft_logits", "root_tok", "cache_len", "q", "tree_k", "tree_v", "target_logits")
        dev = self.attn_out.device
        if self._dev_inputs is None or any(self._dev_inputs[f].shape != getattr(xh, f).shape for f in fields):
            self._dev_inputs = {f: torch.empty(getattr(xh, f).shape, dtype=getattr(xh, f).dtype, device=dev)
                                for f in fields}
            self._copy_stream = torch.cuda.Stream(device=dev)
        if self._n_host is None:
            self._n_host = torch.empty(self.B, dtype=torch.int32).pin_memory()
        d = self._dev_inputs
        main = stream if stream is not None else torch.cuda.current_stream(dev)
        cs = self._copy_stream
        cs.wait_stream(main)  # the previous step's reads of the staging buffers come first
        ev_first = torch.cuda.Event()
        ev_layer = [torch.cuda.Event() for _ in range(self.layers)]
        ev_nodes = torch.cuda.Event()
        ev_target = torch.cuda.Event()
        h2d = 0
        with torch.cuda.stream(cs):
            for f in ("draft_logits", "root_tok", "cache_len"):
                d[f].copy_(getattr(xh, f), non_blocking=True)
                h2d += getattr(xh, f).numel() * getattr(xh, f).element_size()
            ev_first.record(cs)
            for l in range(self.layers):
                for f in ("q", "tree_k", "tree_v"):
                    d[f][l].copy_(getattr(xh, f)[l], non_blocking=True)
                    h2d += getattr(xh, f)[l].numel() * getattr(xh, f)[l].element_size()
                ev_layer[l].record(cs)
        redraft = None
        if xh.redraft is not None:
            redraft = xh.redraft.to(dev, non_blocking=True)
            h2d += xh.redraft.numel() * xh.redraft.element_size()
        x = StepInputs(d["draft_logits"], d["root_tok"], d["cache_len"], redraft, d["q"], d["tree_k"],
                       d["tree_v"], d["target_logits"])
        with torch.cuda.stream(main):
            main.wait_event(ev_first)
            ids, vals, margin, logp1 = cure.cure_score_draft(x.draft_logits, self.k, out=self.score,
                                                             stream=main)
            tree = cure.cure_build_tree(ids, margin, x.root_tok, x.cache_len, self.tau, self.R,
                                        self.branches, self.depth, x.redraft, self.max_ufp,
                                        out=self.tree, stream=main)
            node_rows = xh.target_logits.numel() * xh.target_logits.element_size() >= self.NODE_ROWS_MIN_BYTES
            if node_rows:
                self._n_host.copy_(tree["n_nodes"], non_blocking=True)
                ev_nodes.record(main)
            for l in range(self.layers):
                main.wait_event(ev_layer[l])
                p = self.layer_map[l]
                cure.cure_tree_attn(x.q[l], x.tree_k[l], x.tree_v[l], k_caches[p], v_caches[p], self.kv,
                                    x.cache_len, tree["n_nodes"], tree["anc"], self.scale,
                                    out=self.attn_out[l], workspace=self.workspace, stream=main)
        with torch.cuda.stream(cs):
            if node_rows:
                ev_nodes.synchronize()
                n_max = xh.target_logits.shape[1]
                row_bytes = xh.target_logits.shape[2] * xh.target_logits.element_size()
                for b, nb in enumerate(self._n_host.tolist()):
                    nb = max(0, min(int(nb), n_max))
                    if nb:
                        d["target_logits"][b, :nb].copy_(xh.target_logits[b, :nb], non_blocking=True)
                        h2d += nb * row_bytes
            else:
                d["target_logits"].copy_(xh.target_logits, non_blocking=True)
                h2d += xh.target_logits.numel() * xh.target_logits.element_size()
            ev_target.record(cs)
        with torch.cuda.stream(main):
            main.wait_event(ev_target)
            acc = cure.cure_accept(tree, self.K, target_logits=x.target_logits, targ=self.targ,
                                   out=self.acc, stream=main)
            kl = [k_caches[self.layer_map[l]] for l in range(self.layers)]
            vl = [v_caches[self.layer_map[l]] for l in range(self.layers)]
            rs = cure.cure_resync_kv(kl, vl, self.kv, x.tree_k, x.tree_v, acc, x.cache_len, self.K,
                                     cache_len_out=self.cache_len_out, out=self.rs, stream=main)
        self.last_h2d_bytes = h2d
        return dict(score=self.score, tree=tree, attn=self.attn_out, acc=acc, resync=rs)

    @property
    def launches_per_step(self) -> int:
        """Library kernels one step launches: scan, tree, one attention kernel per
        layer, target argmax + walk, and the resync gather (its finalize runs in
        the gather's grid, since the step's new lengths do not alias the old)."""
        return 1 + 1 + self.layers + 2 + 1
