"""CPU oracle for the CURE repair-verify step (test infrastructure only).

This is a plain, slow, single-threaded float64 restatement of what each stage
of the step computes, written from the paper ("CURE: Local Uncertainty Repair
for Block-Parallel Speculative Decoding"): no blocking, no fusion, no
reordering beyond the definitions.  It shares no code with the CUDA library
and imports nothing from the package.  Only the tests, the smoke check and the
benchmark's CPU-baseline leg may use it; the product path never does.

Stages and the passages they follow:

* ``score_draft``  Sec. 3.3, Eq. (2) and Alg. 1 (draft scores and margin)
* ``build_tree``   Sec. 3.1 Eq. (1) (budget), Sec. 3.3 (gate, ascending-margin
                   order, Eq. (3) dynamic branch budget), Sec. 3.4 (tree
                   construction, branch 0 anchored)
* ``tree_attn``    Sec. 3.2 / 3.4 / 3.5 (single-pass Tree Attention)
* ``accept``       Sec. 3.5 Eq. (4) with greedy decoding (Sec. 4.1)
* ``lm_head_argmax`` the target's greedy token per node from its final
                   hidden state and the LM-head weight (Sec. 3.5, Sec. 4.1)
* ``sample_target`` the target's token per node at a temperature T > 0
                   (Sec. 2: lossless speculative sampling; the paper's own
                   runs are greedy, Sec. 4.1)
* ``resync``       Sec. 3.5 and Alg. 1 (cache resynchronisation)

Readings where the paper is silent or ambiguous (each is listed in the design
notes of the repository):

* ties among equal logits rank the lower vocabulary id first;
* the gate is strict (m_i < tau) with m_i and tau compared in float32, the
  precision the kernels hold the margin in;
* UFPs are admitted in ascending margin order, ties to the lower position;
  each (position, rank) alternative costs ``min(depth, K - i)`` nodes; an
  alternative that does not fit in the remaining budget R is skipped;
* node 0 is the root (last committed token, position L), nodes 1..K are the
  draft chain, repair nodes follow in (position, rank, depth) order;
* Eq. (3), when a margin scale s > 0 is given: b_i counts the alternatives of
  UFP i (ranks 2..b_i + 1), with b_max = branches - 1 (the fixed budget's
  alternatives) and b_min = branch_min; u_i, the product and the sum are
  float32 operations, each rounded to nearest, and round() is half away from
  zero;
* the structural caps of Sec. 3.3-3.4 bound repair branches only (branch 0
  is never pruned): with a maximum depth, an alternative deeper than it is
  not spawned and a successor deeper than it is dropped (the alternative then
  costs one node, as at the last position); with a beam width, an
  alternative is admitted only if every depth it occupies still holds fewer
  nodes than the beam, the chain node included;
* stochastic verification (T > 0) draws the target's token at every tree
  node from softmax(logits / T) by inverse CDF with a given uniform u in
  [0, 1): the first id whose cumulative probability exceeds u; the walk then
  matches children against these samples as it matches them against the
  argmax when greedy.  A sample is independent of the drafted children, so
  every emitted token follows the target's distribution (lossless);
* the best path is the deepest accepted node, lowest node index on ties;
* resync writes the path's rows (root included) into cache slots L..L+a and
  realigns the draft to L + divergence depth (or L + a + 1 on branch-0 wins);
* in the in-place layout (the tree's K/V rows written by the target straight
  into the cache) node j's row is cache slot L + j; attention and resync then
  read the tree rows from there, and the result is the same as with separate
  tree tensors holding those rows.

Parity status: every function is pinned by tests that do not re-use its code
(closed forms, brute force, textbook routines, invariants); see
``tests/test_oracle_pins.py``.
"""
from __future__ import annotations

import math
from typing import Optional, Sequence

import numpy as np


# --------------------------------------------------------------------------
# S1: draft scores (Sec. 3.3, Eq. 2)
# --------------------------------------------------------------------------
def score_draft(logits: np.ndarray, k: int):
    """Per row: top-k (value desc, id asc), margin, log-sum-exp, top-1 log-prob.

    ``logits`` is float64 [rows][V] holding bf16 values widened exactly.
    Eq. (2): m_i = l_{i,1} - l_{i,2}; the log-softmax normaliser cancels in
    the difference, so the logit gap is also the log-probability gap.
    The top-1 log-probability is l_{i,1} - logsumexp_v l_{i,v}.
    Returns (ids int64 [rows][k], vals float64 [rows][k], margin float64
    [rows], lse float64 [rows], logp1 float64 [rows]).
    """
    x = np.asarray(logits, dtype=np.float64)
    R, V = x.shape
    ids = np.empty((R, k), dtype=np.int64)
    vals = np.empty((R, k), dtype=np.float64)
    margin = np.empty(R, dtype=np.float64)
    lse = np.empty(R, dtype=np.float64)
    logp1 = np.empty(R, dtype=np.float64)
    vid = np.arange(V)
    for r in range(R):
        row = x[r]
        # full sort: primary key value descending, secondary key id ascending
        order = np.lexsort((vid, -row))
        ids[r] = order[:k]
        vals[r] = row[order[:k]]
        margin[r] = vals[r, 0] - vals[r, 1] if k >= 2 else np.nan
        mx = row.max()
        lse[r] = mx + math.log(float(np.sum(np.exp(row - mx))))
        logp1[r] = vals[r, 0] - lse[r]
    return ids, vals, margin, lse, logp1


def row_argmax(logits: np.ndarray) -> np.ndarray:
    """First maximum of each row by a linear scan (greedy target, Sec. 4.1)."""
    x = np.asarray(logits, dtype=np.float64)
    out = np.empty(x.shape[0], dtype=np.int64)
    for r in range(x.shape[0]):
        out[r] = int(np.argmax(x[r]))      # numpy returns the first maximum
    return out


def lm_head_argmax(hidden: np.ndarray, w_lm: np.ndarray) -> np.ndarray:
    """The target's greedy token at each tree node from its final hidden state
    (Sec. 3.5, Eq. 4: the target scores every node in one pass; greedy
    decoding, Sec. 4.1): the first maximum over v of the logit
    hidden[r] . w_lm[v], all in float64.

    ``hidden`` is [rows][d_model] and ``w_lm`` the LM-head weight [vocab][d_model],
    both holding bf16 values widened exactly; every product of two bf16 values
    is exact in float64, so the logits are the exact dot products up to float64
    summation.  The fused kernel never writes these logits; its argmax must
    match this one wherever the float32 accumulation bound cannot reorder the
    top two.
    """
    h = np.asarray(hidden, dtype=np.float64)
    V = w_lm.shape[0]
    # the logits [rows][vocab], computed over slices of the vocabulary only to
    # bound the float64 copy of the weight held at once
    chunk = 8192
    logits = np.concatenate([h @ np.asarray(w_lm[v0:v0 + chunk], dtype=np.float64).T
                             for v0 in range(0, V, chunk)], axis=1)
    return row_argmax(logits)


# --------------------------------------------------------------------------
# S2 + S3: UFP selection and tree construction (Sec. 3.1, 3.3, 3.4)
# --------------------------------------------------------------------------
def branch_budget(margin_f32: float, scale: float, b_min: int, b_max: int) -> int:
    """Local branch budget of one UFP, Eq. (3) (Sec. 3.3, dynamic branching).

    u = clip(1 - m / s, 0, 1) and b = clip(round(b_min + u (b_max - b_min)),
    b_min, b_max): a confident position (m near s) keeps b_min alternatives,
    a tied one (m = 0) gets b_max.  Each operation is a float32 operation
    rounded to nearest (the precision the kernels hold the margin in); round()
    takes halves away from zero.
    """
    f = np.float32
    q = f(f(margin_f32) / f(scale))
    u = f(f(1.0) - q)
    u = f(min(max(u, f(0.0)), f(1.0)))
    x = f(f(b_min) + f(u * f(b_max - b_min)))
    r = math.floor(float(x) + 0.5)  # x >= 0: half away from zero
    return int(min(max(r, b_min), b_max))


def repair_cost(i: int, K: int, repair_depth: int, max_depth: int = 0) -> int:
    """Nodes one alternative at position i adds: itself (depth i + 1) and,
    with depth-2 repairs, its successor (depth i + 2), within the block and
    within the maximum depth (0 = none)."""
    c = min(repair_depth, K - i)
    if max_depth > 0:
        c = min(c, max(0, max_depth - i))
    return c


def select_ufps(margin_f32: Sequence[float], tau: float, K: int, budget: int,
                branches: int, repair_depth: int, max_ufp: int = 0,
                margin_scale: float = 0.0, branch_min: int = 1,
                max_depth: int = 0, beam: int = 0):
    """Budgeted ascending-margin selection of Uncertainty Focal Points.

    Sec. 3.3: positions with m_i < tau are UFPs, taken in ascending order of
    m_i while the tree stays within the verifier budget (Eq. 1).  UFP i offers
    the alternatives of ranks 2..branches, or, with a margin scale s > 0, the
    b_i of ranks 2..b_i + 1 that Eq. (3) gives it (b_max = branches - 1).
    A maximum depth and a beam width (Sec. 3.3-3.4, 0 = none) bound where
    alternatives may go: see ``repair_cost`` and the beam test below.
    Returns the admitted alternatives as a list of (position i, rank r), in
    admission order, and the UFP positions that received one.
    """
    t32 = np.float32(tau)
    gated = [i for i in range(K) if np.float32(margin_f32[i]) < t32]
    gated.sort(key=lambda i: (np.float32(margin_f32[i]), i))
    if max_ufp > 0:
        gated = gated[:max_ufp]
    used = 0
    admitted = []
    ufps = []
    width = [1] * (K + 2)          # nodes per depth: the root, then the chain
    for i in gated:
        cost = repair_cost(i, K, repair_depth, max_depth)
        if cost == 0:
            continue
        nalt = branches - 1
        if margin_scale > 0:
            nalt = branch_budget(margin_f32[i], margin_scale, branch_min, branches - 1)
        took = False
        for r in range(2, nalt + 2):
            depths = range(i + 1, i + 1 + cost)
            fits_beam = beam <= 0 or all(width[dd] < beam for dd in depths)
            if used + cost <= budget and fits_beam:
                admitted.append((i, r))
                used += cost
                for dd in depths:
                    width[dd] += 1
                took = True
        if took:
            ufps.append(i)
    return admitted, ufps


def build_tree(top_ids: np.ndarray, margin: np.ndarray, root_tok: np.ndarray,
               cache_len: np.ndarray, tau: float, budget: int, branches: int,
               repair_depth: int, redraft: Optional[np.ndarray] = None,
               max_ufp: int = 0, margin_scale: float = 0.0, branch_min: int = 1,
               max_depth: int = 0, beam: int = 0):
    """Flattened repair tree per sequence (Sec. 3.4, Alg. 1 loop).

    Node 0: root (the last committed token) at depth 0, position L.
    Nodes 1..K: branch 0, the block-parallel draft (top-1 ids), chained.
    Repair nodes: for each admitted (i, r), in (i, r) order, the rank-r
    candidate at position i as a child of node i (a sibling of the draft token
    it replaces); with depth-2 repairs and i < K-1 its re-drafted successor
    follows as its child.  pos = L + depth; anc[j] = anc[parent[j]] + {j}.
    """
    B, K, k = top_ids.shape
    n_max = 1 + K + budget
    W = (n_max + 63) // 64
    n_nodes = np.zeros(B, dtype=np.int64)
    tok = np.full((B, n_max), -1, dtype=np.int64)
    pos = np.full((B, n_max), -1, dtype=np.int64)
    parent = np.full((B, n_max), -1, dtype=np.int64)
    depth = np.full((B, n_max), -1, dtype=np.int64)
    anc = np.zeros((B, n_max, W), dtype=np.uint64)
    ufp_pos = np.full((B, K), -1, dtype=np.int64)
    n_ufp = np.zeros(B, dtype=np.int64)
    for b in range(B):
        admitted, ufps = select_ufps(margin[b], tau, K, budget, branches, repair_depth, max_ufp,
                                     margin_scale, branch_min, max_depth, beam)
        n_ufp[b] = len(ufps)
        ufp_pos[b, :len(ufps)] = ufps
        nodes = [(int(root_tok[b]), -1, 0)]                 # (token, parent, depth)
        for i in range(1, K + 1):
            nodes.append((int(top_ids[b, i - 1, 0]), i - 1, i))
        for (i, r) in sorted(admitted):
            nodes.append((int(top_ids[b, i, r - 1]), i, i + 1))
            if repair_cost(i, K, repair_depth, max_depth) == 2:
                nodes.append((int(redraft[b, i, r - 2]), len(nodes) - 1, i + 2))
        assert len(nodes) <= n_max
        n_nodes[b] = len(nodes)
        sets = []
        for j, (t, p, d) in enumerate(nodes):
            tok[b, j], parent[b, j], depth[b, j] = t, p, d
            pos[b, j] = int(cache_len[b]) + d
            s = ({j} | sets[p]) if p >= 0 else {j}
            sets.append(s)
            for a in s:
                anc[b, j, a // 64] |= np.uint64(1) << np.uint64(a % 64)
    return dict(n_nodes=n_nodes, tok=tok, pos=pos, parent=parent, depth=depth,
                anc=anc, ufp_pos=ufp_pos, n_ufp=n_ufp)


def anc_set(anc_row: np.ndarray) -> list:
    """Node indices whose bit is set in one node's ancestor mask."""
    out = []
    for w, word in enumerate(anc_row):
        word = int(word)
        for bit in range(64):
            if (word >> bit) & 1:
                out.append(w * 64 + bit)
    return out


# --------------------------------------------------------------------------
# S4: tree attention (Sec. 3.2, 3.4, 3.5)
# --------------------------------------------------------------------------
def cache_rows(cache: np.ndarray, b: int, length: int, block_table: Optional[np.ndarray],
               page_size: int) -> np.ndarray:
    """Rows 0..length-1 of sequence b's cache as [length][Hkv][D].

    Contiguous layout: cache[b][t].  Paged layout: cache[page][t % page_size]
    with page = block_table[b][t // page_size].
    """
    if block_table is None:
        return cache[b, :length]
    rows = []
    for t in range(length):
        rows.append(cache[int(block_table[b, t // page_size]), t % page_size])
    return np.stack(rows) if rows else np.zeros((0,) + cache.shape[2:])


def tree_rows_in_cache(cache: np.ndarray, cache_len: np.ndarray, n_nodes: np.ndarray, N: int,
                       block_table: Optional[np.ndarray], page_size: int) -> np.ndarray:
    """The in-place layout's tree rows as [B][N][Hkv][D]: node j of sequence b
    is cache slot L_b + j (rows past n_b stay zero)."""
    B = len(cache_len)
    out = np.zeros((B, N) + cache.shape[2:], dtype=cache.dtype)
    for b in range(B):
        L, n = int(cache_len[b]), int(n_nodes[b])
        out[b, :n] = cache_rows(cache, b, L + n, block_table, page_size)[L:L + n]
    return out


def tree_attn(q: np.ndarray, tree_k: Optional[np.ndarray], tree_v: Optional[np.ndarray],
              k_cache: np.ndarray, v_cache: np.ndarray, cache_len: np.ndarray,
              n_nodes: np.ndarray, anc: np.ndarray, scale: float,
              block_table: Optional[np.ndarray] = None, page_size: int = 16,
              seqs: Optional[Sequence[int]] = None) -> np.ndarray:
    """Tree-masked GQA attention of every tree query over cache + ancestors.

    Query node j of sequence b, head h (kv head h // G) attends to the cached
    keys 0..L_b-1 and to the tree keys of its ancestors (itself included),
    softmax(scale * q k^T) v, all in float64.  ``seqs`` restricts the work to
    some sequences; other rows of the result stay zero.  ``tree_k`` and
    ``tree_v`` None: the in-place layout (node j's rows at cache slot L_b + j).
    """
    B, N, Hq, D = q.shape
    if tree_k is None:
        tree_k = tree_rows_in_cache(k_cache, cache_len, n_nodes, N, block_table, page_size)
        tree_v = tree_rows_in_cache(v_cache, cache_len, n_nodes, N, block_table, page_size)
    Hkv = tree_k.shape[2]
    G = Hq // Hkv
    out = np.zeros((B, N, Hq, D), dtype=np.float64)
    for b in (range(B) if seqs is None else seqs):
        L = int(cache_len[b])
        kc = np.asarray(cache_rows(k_cache, b, L, block_table, page_size), dtype=np.float64)
        vc = np.asarray(cache_rows(v_cache, b, L, block_table, page_size), dtype=np.float64)
        for j in range(int(n_nodes[b])):
            a = anc_set(anc[b, j])
            for hk in range(Hkv):
                keys = np.concatenate([kc[:, hk, :], tree_k[b, a, hk, :]], axis=0)
                vals = np.concatenate([vc[:, hk, :], tree_v[b, a, hk, :]], axis=0)
                for g in range(G):
                    h = hk * G + g
                    s = (keys @ q[b, j, h, :].astype(np.float64)) * scale
                    p = np.exp(s - s.max())
                    out[b, j, h, :] = (p @ vals) / p.sum()
    return out


# --------------------------------------------------------------------------
# S5: acceptance walk (Sec. 3.5, Eq. 4; greedy, Sec. 4.1)
# --------------------------------------------------------------------------
def accept(targ: np.ndarray, n_nodes: np.ndarray, tok: np.ndarray, parent: np.ndarray,
           depth: np.ndarray, anc: np.ndarray, block: int):
    """Longest accepted root-to-node path per sequence.

    ``targ[b][j]`` is the target's greedy token after node j.  A non-root node
    is verified when its token equals the target token at its parent; a node is
    accepted when every non-root node on its path is verified.  pi* (Eq. 4) is
    the deepest accepted node, lowest index on ties; a(pi*) is its depth.
    Outputs the path, the emitted tokens (path tokens then the target's token
    after the last accepted node) and the divergence depth: the shallowest
    path node that is not on branch 0 (node index > K), or -1.
    """
    B, N = tok.shape
    accept_len = np.zeros(B, dtype=np.int64)
    best_node = np.zeros(B, dtype=np.int64)
    path_nodes = np.full((B, block + 2), -1, dtype=np.int64)
    out_tokens = np.full((B, block + 2), -1, dtype=np.int64)
    diverge = np.full(B, -1, dtype=np.int64)
    for b in range(B):
        n = int(n_nodes[b])
        verified = [False] * n
        for j in range(1, n):
            verified[j] = int(tok[b, j]) == int(targ[b, int(parent[b, j])])
        best = 0
        for j in range(n):
            ok = all(verified[a] for a in anc_set(anc[b, j]) if a != 0)
            if ok and (depth[b, j] > depth[b, best]):
                best = j
        a_len = int(depth[b, best])
        path = sorted(anc_set(anc[b, best]), key=lambda x: int(depth[b, x]))
        accept_len[b] = a_len
        best_node[b] = best
        path_nodes[b, :len(path)] = path
        toks = [int(tok[b, x]) for x in path[1:]] + [int(targ[b, best])]
        out_tokens[b, :len(toks)] = toks
        for t, x in enumerate(path):
            if x > block:
                diverge[b] = t
                break
    return dict(accept_len=accept_len, best_node=best_node, path_nodes=path_nodes,
                out_tokens=out_tokens, diverge_depth=diverge)


def sample_target(logits: np.ndarray, n_nodes: np.ndarray, uniforms: np.ndarray,
                  temperature: float) -> np.ndarray:
    """The target's token at each tree node, sampled at temperature T > 0.

    Sec. 2 frames speculative decoding as lossless sampling from the target;
    with T > 0 the target's token after node j is drawn from
    softmax(logits[b][j] / T), here by inverse CDF: with u = uniforms[b][j] in
    [0, 1), the first id v whose cumulative probability exceeds u.  A row of
    -inf logits gives id 0 (as the argmax's tie rule would).  Rows at
    j >= n_nodes[b] are -1.  Float64 throughout.
    """
    B, N, V = logits.shape
    out = np.full((B, N), -1, dtype=np.int64)
    for b in range(B):
        for j in range(int(n_nodes[b])):
            x = np.asarray(logits[b, j], dtype=np.float64)
            m = x.max()
            if m == -np.inf:
                out[b, j] = 0
                continue
            p = np.exp((x - m) / temperature)
            c = np.cumsum(p)
            r = float(uniforms[b, j]) * c[-1]
            y = int(np.searchsorted(c, r, side="right"))
            out[b, j] = min(y, int(np.flatnonzero(p > 0)[-1]))
    return out


# --------------------------------------------------------------------------
# S6: repair resynchronisation (Sec. 3.5, Alg. 1)
# --------------------------------------------------------------------------
def resync(k_caches: list, v_caches: list, tree_k: Optional[list], tree_v: Optional[list],
           path_nodes: np.ndarray, accept_len: np.ndarray, diverge: np.ndarray,
           out_tokens: np.ndarray, cache_len: np.ndarray, block: int,
           block_table: Optional[np.ndarray] = None, page_size: int = 16):
    """Write the verified path into the caches and realign the draft state.

    For every layer l and sequence b, the K/V rows of the path nodes at depths
    0..a go to cache slots L..L+a (through the block table when paged); the
    cache then holds L + a + 1 rows.  The draft state stays valid up to the
    divergence: L + d when a repair path wins at depth d, else L + a + 1.  The
    tokens to replay into the draft are the path tokens from depth d to a and
    the target's next token (only that token on branch-0 wins).
    ``k_caches``/``v_caches`` are per-layer arrays, modified in place;
    ``tree_k``/``tree_v`` are [layers][B][N][Hkv][D], or None for the in-place
    layout, where the path rows are read from cache slots L_b + node (all of
    them before any write).
    """
    B = len(cache_len)
    if tree_k is None:
        tree_k, tree_v = [], []
        for l in range(len(k_caches)):
            rk, rv = {}, {}
            for b in range(B):
                L = int(cache_len[b])
                for t in range(int(accept_len[b]) + 1):
                    node = int(path_nodes[b, t])
                    rk[b, node] = cache_rows(k_caches[l], b, L + node + 1, block_table, page_size)[L + node].copy()
                    rv[b, node] = cache_rows(v_caches[l], b, L + node + 1, block_table, page_size)[L + node].copy()
            tree_k.append(rk)
            tree_v.append(rv)
    new_len = np.array(cache_len, dtype=np.int64)
    draft_valid = np.zeros(B, dtype=np.int64)
    replay = np.full((B, block + 2), -1, dtype=np.int64)
    n_replay = np.zeros(B, dtype=np.int64)
    for b in range(B):
        L = int(cache_len[b])
        a = int(accept_len[b])
        for l in range(len(k_caches)):
            for t in range(a + 1):
                node = int(path_nodes[b, t])
                slot = L + t
                kr, vr = tree_k[l][b, node], tree_v[l][b, node]
                if block_table is None:
                    k_caches[l][b, slot] = kr
                    v_caches[l][b, slot] = vr
                else:
                    page = int(block_table[b, slot // page_size])
                    k_caches[l][page, slot % page_size] = kr
                    v_caches[l][page, slot % page_size] = vr
        new_len[b] = L + a + 1
        d = int(diverge[b])
        if d >= 0:
            draft_valid[b] = L + d
            toks = [int(out_tokens[b, t - 1]) for t in range(d, a + 1)] + [int(out_tokens[b, a])]
        else:
            draft_valid[b] = L + a + 1
            toks = [int(out_tokens[b, a])]
        replay[b, :len(toks)] = toks
        n_replay[b] = len(toks)
    return dict(cache_len=new_len, draft_valid_len=draft_valid, replay_tokens=replay,
                n_replay=n_replay)
