"""Seeded synthetic workloads for the CURE repair-verify step.

This module only draws random inputs. It holds none of the method's
arithmetic (no margins, no gating, no tree building, no attention, no
acceptance): it plants draft tokens and rivals into noise logits, draws
attention tensors and cache lengths, and provides a stand-in for the target
language model (``synthetic_target_ids``) that maps each tree node to the
token the target "would" predict after it.

Both the CUDA path (through the Python binding) and the CPU oracle consume
what is drawn here; nothing here depends on either of them.

The shapes follow the workloads the paper evaluates on (block size K = 16,
greedy decoding, Sec. 4.1) and the five configurations of the build:

* ``tiny``      batch 1, block 8,  vocab 32000,  1 layer,  8/2 heads, L 512
* ``single8b``  batch 1, block 16, vocab 128256, 32 layers, 32/8 heads, L 4096
* ``serve32``   batch 32, block 16, vocab 151936, 28 layers, 28/4 heads,
                L ~ U[1024, 8192], paged 16-token blocks (the metric's workload)
* ``long64``    batch 64, block 16, vocab 128256, 80 layers, 64/8 heads,
                L 32768, depth-2 repair paths
* ``sweep16``   batch 16, block 32, vocab 151936, 28 layers, 28/4 heads, L 8192,
                budget/threshold sweep
"""
from __future__ import annotations

import dataclasses
from typing import Optional

import numpy as np
import torch

PAGE_SIZE = 16


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    batch: int
    block: int                 # K, draft positions per block
    vocab: int
    tau: float                 # margin threshold (Sec. 3.3)
    budget: int                # R, repair nodes per sequence
    branches: int              # candidates per UFP, the draft token included
    repair_depth: int          # 1: alternative leaf only; 2: alternative + re-drafted successor
    layers: int
    heads_q: int
    heads_kv: int
    head_dim: int
    len_lo: int                # cache length range (inclusive) per sequence
    len_hi: int
    paged: bool
    top_level: float           # planted draft-token logit
    gap_mean: float            # mean of the Exp() gap between draft token and rival
    first_error: str           # "uniform" (U{0..K}) or "geom9" (geometric, mean 9)
    seed: int
    qk_std: float = 1.0 / np.sqrt(128.0)
    v_std: float = 1.0 / np.sqrt(128.0)

    @property
    def topk(self) -> int:
        """Number of ranked candidates kept per draft position."""
        return max(2, self.branches)

    @property
    def n_max(self) -> int:
        """Padded node capacity of one sequence's tree: root + K chain + R repair."""
        return 1 + self.block + self.budget

    @property
    def group(self) -> int:
        return self.heads_q // self.heads_kv

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


WORKLOADS = {
    "tiny": Workload("tiny", 1, 8, 32000, 1.0, 4, 2, 1, 1, 8, 2, 128, 512, 512, False,
                     6.0, 3.0, "uniform", 1000),
    "single8b": Workload("single8b", 1, 16, 128256, 1.0, 8, 2, 1, 32, 32, 8, 128, 4096, 4096,
                         False, 6.0, 3.0, "geom9", 1001),
    "serve32": Workload("serve32", 32, 16, 151936, 0.8, 16, 3, 1, 28, 28, 4, 128, 1024, 8192,
                        True, 16.0, 2.5, "uniform", 1002),
    "long64": Workload("long64", 64, 16, 128256, 1.0, 32, 2, 2, 80, 64, 8, 128, 32768, 32768,
                       False, 6.0, 3.0, "geom9", 1003),
    "sweep16": Workload("sweep16", 16, 32, 151936, 1.0, 16, 3, 1, 28, 28, 4, 128, 8192, 8192,
                        False, 16.0, 2.5, "geom9", 1004),
}


def to_bf16(x: np.ndarray) -> torch.Tensor:
    """Round a float32 array to bfloat16 (round to nearest even) as a CPU tensor."""
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16)


def bf16_to_f64(t: torch.Tensor) -> np.ndarray:
    """Exact widening of a bf16 tensor to a float64 numpy array."""
    return t.detach().to("cpu").to(torch.float32).numpy().astype(np.float64)


@dataclasses.dataclass
class DraftBlock:
    logits: torch.Tensor        # bf16 [B][K][V]
    draft_tok: np.ndarray       # int64 [B][K]: planted draft token per position
    rival_tok: np.ndarray       # int64 [B][K]: planted second candidate per position
    root_tok: np.ndarray        # int32 [B]: last committed token (tree root)
    redraft: np.ndarray         # int32 [B][K][branches-1]: successor after each alternative


def draft_block(w: Workload, seed: Optional[int] = None, batch: Optional[int] = None) -> DraftBlock:
    """Draft logits with a planted draft token and a planted rival at each position.

    Noise N(0,1) everywhere; the draft token sits at ``top_level`` and the rival
    at ``top_level - gap`` with gap ~ Exp(``gap_mean``).  When the gap is
    larger than the noise ceiling the realised second-best is a noise entry.
    """
    rng = np.random.default_rng(w.seed if seed is None else seed)
    B = w.batch if batch is None else batch
    K, V = w.block, w.vocab
    x = rng.standard_normal((B, K, V), dtype=np.float32)
    y = rng.integers(0, V, size=(B, K))
    r = (y + rng.integers(1, V, size=(B, K))) % V
    gap = rng.exponential(w.gap_mean, size=(B, K)).astype(np.float32)
    bi, ki = np.meshgrid(np.arange(B), np.arange(K), indexing="ij")
    x[bi, ki, y] = np.float32(w.top_level)
    x[bi, ki, r] = np.float32(w.top_level) - gap
    root = rng.integers(0, V, size=B).astype(np.int32)
    nalt = max(1, w.branches - 1)
    redraft = np.full((B, K, nalt), -1, dtype=np.int32)
    # identity re-draft: the successor of a substituted token is the draft's own
    # next token (the draft model that would re-sample the suffix is not part of
    # this step).
    redraft[:, : K - 1, :] = y[:, 1:, None].astype(np.int32)
    return DraftBlock(to_bf16(x), y, r, root, redraft)


def first_errors(w: Workload, rng: np.random.Generator, B: int) -> np.ndarray:
    if w.first_error == "uniform":
        return rng.integers(0, w.block + 1, size=B)
    if w.first_error == "geom9":
        return np.minimum(rng.geometric(0.1, size=B) - 1, w.block)
    raise ValueError(w.first_error)


def target_truth(w: Workload, d: DraftBlock, seed: Optional[int] = None) -> np.ndarray:
    """The target's greedy continuation per sequence, ``truth[b][0..K]``.

    It agrees with the draft before a seeded first-error position e; at e it
    takes the planted rival with probability 1/2 (else an unrelated token);
    after e it agrees with the draft again; ``truth[K]`` is a free token.
    """
    rng = np.random.default_rng((w.seed if seed is None else seed) + 7919)
    B, K, V = d.draft_tok.shape[0], w.block, w.vocab
    e = first_errors(w, rng, B)
    truth = np.empty((B, K + 1), dtype=np.int64)
    truth[:, :K] = d.draft_tok
    truth[:, K] = rng.integers(0, V, size=B)
    coin = rng.random(B) < 0.5
    other = rng.integers(0, V, size=B)
    for b in range(B):
        if e[b] < K:
            if coin[b]:
                truth[b, e[b]] = d.rival_tok[b, e[b]]
            else:
                t = int(other[b])
                while t == d.draft_tok[b, e[b]] or t == d.rival_tok[b, e[b]]:
                    t = (t + 1) % V
                truth[b, e[b]] = t
    return truth


def synthetic_target_ids(truth: np.ndarray, n_nodes: np.ndarray, tok: np.ndarray,
                         parent: np.ndarray, depth: np.ndarray, vocab: int,
                         seed: int) -> np.ndarray:
    """Stand-in for the target model's greedy prediction at every tree node.

    A node whose root-to-node tokens equal the truth prefix predicts the next
    truth token; any other node predicts an unrelated seeded token.  Rows at or
    beyond ``n_nodes[b]`` get a seeded token too (they are never read).
    """
    rng = np.random.default_rng(seed + 104729)
    B, N = tok.shape
    out = rng.integers(0, vocab, size=(B, N)).astype(np.int64)
    for b in range(B):
        on_truth = np.zeros(N, dtype=bool)
        for j in range(int(n_nodes[b])):
            p = int(parent[b, j])
            if p < 0:
                on_truth[j] = True
            else:
                dj = int(depth[b, j])
                on_truth[j] = on_truth[p] and int(tok[b, j]) == int(truth[b, dj - 1])
            if on_truth[j]:
                out[b, j] = truth[b, int(depth[b, j])]
    return out


def target_logits(ids: np.ndarray, vocab: int, seed: int) -> torch.Tensor:
    """bf16 [B][N][V] logits: N(0,1) noise with the given id planted at +8."""
    rng = np.random.default_rng(seed + 15485863)
    B, N = ids.shape
    x = rng.standard_normal((B, N, vocab), dtype=np.float32)
    bi, ni = np.meshgrid(np.arange(B), np.arange(N), indexing="ij")
    x[bi, ni, ids] = np.float32(8.0)
    return to_bf16(x)


def cache_lengths(w: Workload, seed: Optional[int] = None, batch: Optional[int] = None) -> np.ndarray:
    rng = np.random.default_rng((w.seed if seed is None else seed) + 31337)
    B = w.batch if batch is None else batch
    return rng.integers(w.len_lo, w.len_hi + 1, size=B).astype(np.int32)


def pages_needed(cache_len: np.ndarray, block: int, page_size: int = PAGE_SIZE) -> np.ndarray:
    """Pages a sequence needs to hold its cache plus one block's worth of growth."""
    return (cache_len.astype(np.int64) + block + 1 + page_size - 1) // page_size


def block_table(cache_len: np.ndarray, block: int, seed: int,
                page_size: int = PAGE_SIZE) -> tuple[np.ndarray, int]:
    """Shuffled physical page ids per sequence; -1 marks unused slots.

    Returns (table int32 [B][max_pages], number of physical pages).
    """
    rng = np.random.default_rng(seed + 271828)
    need = pages_needed(cache_len, block, page_size)
    total = int(need.sum())
    perm = rng.permutation(total).astype(np.int32)
    maxp = int(need.max())
    table = np.full((len(cache_len), maxp), -1, dtype=np.int32)
    o = 0
    for b, n in enumerate(need):
        table[b, :n] = perm[o:o + n]
        o += n
    return table, total


def normal_bf16(shape, std: float, rng: np.random.Generator) -> torch.Tensor:
    return to_bf16(rng.standard_normal(shape, dtype=np.float32) * np.float32(std))


# ------------------------------------------------------------------ LM head
def lm_head_weight(vocab: int, d_model: int, seed: int, chunk: int = 16384) -> torch.Tensor:
    """A seeded stand-in for the target's LM-head weight, bf16 [vocab][d_model]:
    N(0, 1/d_model) entries, so each row's squared norm is about 1.  Drawn in
    slices of the vocabulary (each slice from its own seeded stream) to bound
    the float32 memory held at once."""
    out = torch.empty(vocab, d_model, dtype=torch.bfloat16)
    sd = np.float32(1.0 / np.sqrt(d_model))
    for i, v0 in enumerate(range(0, vocab, chunk)):
        rng = np.random.default_rng([seed, 7717, i])
        n = min(chunk, vocab - v0)
        out[v0:v0 + n] = to_bf16(rng.standard_normal((n, d_model), dtype=np.float32) * sd)
    return out


def lm_head_hidden(rows: int, w_lm: torch.Tensor, seed: int, planted: Optional[np.ndarray] = None,
                   strength: float = 12.0) -> torch.Tensor:
    """Seeded final hidden states bf16 [rows][d_model]: N(0, 1) entries, plus
    ``strength`` times the weight row of ``planted[r]`` where planted[r] >= 0,
    so that logit's expected value is about ``strength`` against N(0, 1) for the
    others (a stand-in target that prefers the planted token)."""
    d = w_lm.shape[1]
    rng = np.random.default_rng([seed, 4243])
    h = rng.standard_normal((rows, d), dtype=np.float32)
    if planted is not None:
        sel = np.flatnonzero(np.asarray(planted) >= 0)
        if len(sel):
            wt = w_lm[torch.from_numpy(np.asarray(planted)[sel].astype(np.int64))].to(torch.float32).numpy()
            h[sel] += np.float32(strength) * wt
    return to_bf16(h)
