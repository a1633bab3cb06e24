"""GPU parity: every stage through the C ABI against the CPU oracle.

Bit-exact for ids, trees, accept results and resynced cache rows; margins
bit-exact (the difference of two bf16 values is exact in float32); top-1
log-probs within 1e-5 * max(1, |ref|); bf16 attention outputs within 2e-2
absolute (and 2e-2 of the output scale on flat inputs).
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2608_00531_gb300 import workload as W

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda:0")
ATTN_ABS_TOL = 2e-2
LOGP_TOL = 1e-5


@pytest.fixture(scope="module")
def cure():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_00531_gb300 import cure as c
    torch.cuda.set_device(DEV)
    return c


def _f64(t):
    return W.bf16_to_f64(t)


def _check_scores(c, logits_bf16, k, rows_sel=None):
    ids, vals, margin, logp1 = c.cure_score_draft(logits_bf16.to(DEV), k)
    torch.cuda.synchronize()
    V = logits_bf16.shape[-1]
    x = _f64(logits_bf16).reshape(-1, V)
    sel = np.arange(x.shape[0]) if rows_sel is None else np.asarray(rows_sel)
    o_ids, o_vals, o_m, _, o_lp = oracle.score_draft(x[sel], k)
    g_ids = ids.cpu().numpy().reshape(-1, k)[sel]
    g_vals = vals.cpu().numpy().reshape(-1, k)[sel]
    g_m = margin.cpu().numpy().reshape(-1)[sel]
    g_lp = logp1.cpu().numpy().reshape(-1)[sel]
    assert np.array_equal(g_ids, o_ids)
    assert np.array_equal(g_vals, o_vals.astype(np.float32))
    assert np.array_equal(g_m, o_m.astype(np.float32))
    fin = np.isfinite(o_lp)
    err = np.abs(g_lp[fin] - o_lp[fin])
    assert np.all(err <= LOGP_TOL * np.maximum(1.0, np.abs(o_lp[fin]))), err.max()
    return ids, margin, o_ids, o_m


@pytest.mark.parametrize("name", ["tiny", "single8b"])
def test_score_draft_workloads(cure, name):
    w = W.WORKLOADS[name]
    d = W.draft_block(w)
    _check_scores(cure, d.logits, w.topk)


@pytest.mark.parametrize("V,k,rows", [(1001, 2, 7), (32003, 3, 5), (77, 8, 33), (8, 2, 3), (9, 4, 4),
                                      (151936, 4, 3), (40000, 5, 2)])
def test_score_draft_ragged_and_ties(cure, V, k, rows):
    rng = np.random.default_rng(V + k)
    # a few distinct values: many exact ties, some -inf
    x = rng.integers(-3, 4, size=(rows, V)).astype(np.float32) * 0.5
    x[0, rng.integers(0, V, size=max(1, V // 10))] = -np.inf
    _check_scores(cure, W.to_bf16(x), k)


def test_score_draft_full_serve_shape_sampled(cure):
    """batch 32 x block 16 x vocab 151936 in the launch configuration the
    benchmark times; the oracle checks 64 sampled rows."""
    w = W.WORKLOADS["serve32"]
    d = W.draft_block(w)
    rows = np.random.default_rng(0).choice(w.batch * w.block, size=64, replace=False)
    _check_scores(cure, d.logits, w.topk, rows)


@pytest.mark.parametrize("rows,V,k", [(1024, 151936, 3), (960, 32003, 4), (912, 50021, 6), (1000, 4099, 8)])
def test_score_draft_one_cta_per_row(cure, rows, V, k):
    """Row counts that give every SM six CTAs take the one-CTA-per-row launch
    (no cluster merge); the top-k, margin and log-probability epilogue of that
    launch on sampled rows, half of them with many exact ties and -inf."""
    rng = np.random.default_rng(rows + V + k)
    x = rng.standard_normal((rows, V), dtype=np.float32)
    tied = rng.random(rows) < 0.5
    x[tied] = np.round(x[tied] * 2.0) * 0.5
    x[tied, : V // 7] = -np.inf
    sel = np.concatenate([np.arange(4), rng.choice(rows, size=60, replace=False)])
    _check_scores(cure, W.to_bf16(x), k, sel)


def test_score_draft_full_long_shape_sampled(cure):
    """batch 64 x block 16 x vocab 128256 with top-2: 1024 rows, one CTA per
    row, the launch the long-context configuration takes; 64 sampled rows."""
    w = W.WORKLOADS["long64"]
    d = W.draft_block(w)
    rows = np.random.default_rng(1).choice(w.batch * w.block, size=64, replace=False)
    _check_scores(cure, d.logits, w.topk, rows)


def _tree_inputs(w, seed=None):
    d = W.draft_block(w, seed=seed)
    x = _f64(d.logits).reshape(-1, w.vocab)
    o_ids, _, o_m, _, _ = oracle.score_draft(x, w.topk)
    B, K, k = w.batch, w.block, w.topk
    return d, o_ids.reshape(B, K, k), o_m.astype(np.float32).reshape(B, K)


def _gpu_tree(c, ids, margin, root, L, w, redraft=None, max_ufp=0, tau=None, budget=None):
    tau = w.tau if tau is None else tau
    budget = w.budget if budget is None else budget
    return c.cure_build_tree(torch.from_numpy(ids.astype(np.int32)).to(DEV),
                             torch.from_numpy(margin).to(DEV),
                             torch.from_numpy(root.astype(np.int32)).to(DEV),
                             torch.from_numpy(L.astype(np.int32)).to(DEV), tau, budget, w.branches,
                             w.repair_depth,
                             None if redraft is None else torch.from_numpy(redraft.astype(np.int32)).to(DEV),
                             max_ufp)


def _cmp_tree(g, t):
    for key in ("n_nodes", "tok", "pos", "parent", "depth", "ufp_pos", "n_ufp"):
        assert np.array_equal(g[key].cpu().numpy(), t[key]), key
    assert np.array_equal(g["anc"].cpu().numpy().view(np.uint64), t["anc"])


@pytest.mark.parametrize("name", ["tiny", "single8b", "serve32"])
def test_build_tree_workloads(cure, name):
    w = W.WORKLOADS[name]
    d, ids, margin = _tree_inputs(w)
    L = W.cache_lengths(w)
    g = _gpu_tree(cure, ids, margin, d.root_tok, L, w)
    t = oracle.build_tree(ids, margin, d.root_tok, L, w.tau, w.budget, w.branches, w.repair_depth)
    _cmp_tree(g, t)


def test_build_tree_depth2_long_shape(cure):
    w = W.WORKLOADS["long64"].replace(vocab=4096)   # the tree does not depend on V
    d, ids, margin = _tree_inputs(w)
    L = W.cache_lengths(w)
    g = _gpu_tree(cure, ids, margin, d.root_tok, L, w, redraft=d.redraft)
    t = oracle.build_tree(ids, margin, d.root_tok, L, w.tau, w.budget, w.branches, 2, d.redraft)
    _cmp_tree(g, t)


@pytest.mark.parametrize("budget", [0, 4, 8, 16, 32, 64])
@pytest.mark.parametrize("tau", [0.25, 0.5, 1.0, 2.0, 4.0])
def test_build_tree_sweep(cure, budget, tau):
    w = W.WORKLOADS["sweep16"].replace(vocab=4096)
    d, ids, margin = _tree_inputs(w)
    L = W.cache_lengths(w)
    g = _gpu_tree(cure, ids, margin, d.root_tok, L, w, tau=tau, budget=budget)
    t = oracle.build_tree(ids, margin, d.root_tok, L, tau, budget, w.branches, 1)
    _cmp_tree(g, t)


@pytest.mark.parametrize("seed", range(12))
def test_build_tree_random_params(cure, seed):
    rng = np.random.default_rng(seed)
    B, K = int(rng.integers(1, 9)), int(rng.integers(1, 33))
    k = int(rng.integers(2, 9))
    branches = int(rng.integers(1, k + 1))
    depth = int(rng.integers(1, 3))
    budget = int(rng.integers(0, 80))
    tau = float(rng.choice([0.0, 0.5, 1.0, 3.0]))
    max_ufp = int(rng.choice([0, 0, 1, 3]))
    margin = (rng.integers(0, 16, size=(B, K)) * 0.25).astype(np.float32)
    ids = rng.integers(0, 50000, size=(B, K, k))
    root = rng.integers(0, 50000, size=B)
    L = rng.integers(0, 1000, size=B)
    redraft = rng.integers(0, 50000, size=(B, K, max(1, branches - 1)))
    w = W.WORKLOADS["tiny"].replace(batch=B, block=K, branches=branches, repair_depth=depth)
    g = cure.cure_build_tree(torch.from_numpy(ids.astype(np.int32)).to(DEV), torch.from_numpy(margin).to(DEV),
                             torch.from_numpy(root.astype(np.int32)).to(DEV),
                             torch.from_numpy(L.astype(np.int32)).to(DEV), tau, budget, branches, depth,
                             torch.from_numpy(redraft.astype(np.int32)).to(DEV), max_ufp)
    t = oracle.build_tree(ids, margin, root, L, tau, budget, branches, depth, redraft, max_ufp)
    _cmp_tree(g, t)


@pytest.mark.parametrize("seed", range(16))
def test_build_tree_dynamic_budget_random(cure, seed):
    """Eq. (3) dynamic branch budget: bit-exact against the oracle, including
    margins on a grid where b_min + u (b_max - b_min) lands on halves."""
    rng = np.random.default_rng(100 + seed)
    B, K = int(rng.integers(1, 9)), int(rng.integers(1, 33))
    k = int(rng.integers(2, 9))
    branches = int(rng.integers(1, k + 1))
    branch_min = int(rng.integers(0, branches))
    depth = int(rng.integers(1, 3))
    budget = int(rng.integers(0, 120))
    scale = float(rng.choice([0.3, 0.8, 1.0, 2.5, 8.0]))
    tau = float(rng.choice([0.5, 1.0, 3.0, 10.0]))
    if seed % 2:
        margin = (rng.integers(0, 40, size=(B, K)) * 0.25).astype(np.float32)
    else:
        margin = rng.exponential(1.0, size=(B, K)).astype(np.float32)
    ids = rng.integers(0, 50000, size=(B, K, k))
    root = rng.integers(0, 50000, size=B)
    L = rng.integers(0, 1000, size=B)
    redraft = rng.integers(0, 50000, size=(B, K, max(1, branches - 1)))
    g = cure.cure_build_tree(torch.from_numpy(ids.astype(np.int32)).to(DEV), torch.from_numpy(margin).to(DEV),
                             torch.from_numpy(root.astype(np.int32)).to(DEV),
                             torch.from_numpy(L.astype(np.int32)).to(DEV), tau, budget, branches, depth,
                             torch.from_numpy(redraft.astype(np.int32)).to(DEV), 0,
                             margin_scale=scale, branch_min=branch_min)
    t = oracle.build_tree(ids, margin, root, L, tau, budget, branches, depth, redraft, 0,
                          margin_scale=scale, branch_min=branch_min)
    _cmp_tree(g, t)


def test_build_tree_dynamic_budget_paper_setting(cure):
    """The paper's dynamic branching, (b_min, b_max) = (1, 5), on the serving
    shape's scores (top-6 candidates), s = tau."""
    w = W.WORKLOADS["serve32"].replace(branches=6)
    d, ids, margin = _tree_inputs(w)
    L = W.cache_lengths(w)
    g = cure.cure_build_tree(torch.from_numpy(ids.astype(np.int32)).to(DEV), torch.from_numpy(margin).to(DEV),
                             torch.from_numpy(d.root_tok.astype(np.int32)).to(DEV),
                             torch.from_numpy(L.astype(np.int32)).to(DEV), w.tau, w.budget, 6, 1, None, 0,
                             margin_scale=w.tau, branch_min=1)
    t = oracle.build_tree(ids, margin, d.root_tok, L, w.tau, w.budget, 6, 1, None, 0,
                          margin_scale=w.tau, branch_min=1)
    _cmp_tree(g, t)
    # the budget varies with the margin: some UFPs take more alternatives than others
    counts = []
    for b in range(w.batch):
        par = t["parent"][b, 1 + w.block:int(t["n_nodes"][b])]
        counts += [int((par == i).sum()) for i in set(par.tolist())]
    assert len(set(counts)) > 1


@pytest.mark.parametrize("seed", range(16))
def test_build_tree_caps_random(cure, seed):
    """Maximum repair depth and beam width (with and without Eq. (3)),
    bit-exact against the oracle."""
    rng = np.random.default_rng(300 + seed)
    B, K = int(rng.integers(1, 9)), int(rng.integers(1, 33))
    k = int(rng.integers(2, 9))
    branches = int(rng.integers(1, k + 1))
    depth = int(rng.integers(1, 3))
    budget = int(rng.integers(0, 120))
    tau = float(rng.choice([0.5, 1.0, 3.0]))
    max_depth = int(rng.choice([0, 1, 2, K // 2 + 1, K]))
    beam = int(rng.choice([0, 1, 2, 3, 5]))
    scale = float(rng.choice([0.0, 1.0]))
    branch_min = int(rng.integers(0, branches)) if scale > 0 else 1
    margin = (rng.integers(0, 16, size=(B, K)) * 0.25).astype(np.float32)
    ids = rng.integers(0, 50000, size=(B, K, k))
    root = rng.integers(0, 50000, size=B)
    L = rng.integers(0, 1000, size=B)
    redraft = rng.integers(0, 50000, size=(B, K, max(1, branches - 1)))
    g = cure.cure_build_tree(torch.from_numpy(ids.astype(np.int32)).to(DEV), torch.from_numpy(margin).to(DEV),
                             torch.from_numpy(root.astype(np.int32)).to(DEV),
                             torch.from_numpy(L.astype(np.int32)).to(DEV), tau, budget, branches, depth,
                             torch.from_numpy(redraft.astype(np.int32)).to(DEV), 0,
                             margin_scale=scale, branch_min=branch_min, max_depth=max_depth, beam=beam)
    t = oracle.build_tree(ids, margin, root, L, tau, budget, branches, depth, redraft, 0,
                          margin_scale=scale, branch_min=branch_min, max_depth=max_depth, beam=beam)
    _cmp_tree(g, t)


def test_build_tree_paper_primary_configuration(cure):
    """The paper's primary configuration on the serving shape's top-6 scores:
    tau = 1.0, at most one repaired position per block, up to 5 alternatives
    (Eq. (3) with (b_min, b_max) = (1, 5), s = tau), maximum depth 15, beam 5."""
    w = W.WORKLOADS["serve32"].replace(branches=6)
    d, ids, margin = _tree_inputs(w)
    L = W.cache_lengths(w)
    kw = dict(margin_scale=1.0, branch_min=1, max_depth=15, beam=5)
    g = cure.cure_build_tree(torch.from_numpy(ids.astype(np.int32)).to(DEV), torch.from_numpy(margin).to(DEV),
                             torch.from_numpy(d.root_tok.astype(np.int32)).to(DEV),
                             torch.from_numpy(L.astype(np.int32)).to(DEV), 1.0, w.budget, 6, 1, None, 1, **kw)
    t = oracle.build_tree(ids, margin, d.root_tok, L, 1.0, w.budget, 6, 1, None, 1, **kw)
    _cmp_tree(g, t)
    assert (t["n_ufp"] <= 1).all() and (t["n_nodes"] <= 1 + w.block + 5).all()


# ------------------------------------------------------------------ attention
def _attn_case(B, K, budget, Hq, Hkv, lens, paged, qk_std, v_std, seed, tau=1.0, branches=3, ps=16):
    rng = np.random.default_rng(seed)
    k = max(2, branches)
    margin = (rng.integers(0, 8, size=(B, K)) * 0.25).astype(np.float32)
    ids = rng.integers(0, 1000, size=(B, K, k))
    root = rng.integers(0, 1000, size=B)
    L = np.asarray(lens, dtype=np.int32)
    t = oracle.build_tree(ids, margin, root, L, tau, budget, branches, 1)
    N = 1 + K + budget
    D = 128
    q = W.normal_bf16((B, N, Hq, D), qk_std, rng)
    tk = W.normal_bf16((B, N, Hkv, D), qk_std, rng)
    tv = W.normal_bf16((B, N, Hkv, D), v_std, rng)
    if paged:
        table, npages = W.block_table(L, K, seed, ps)
        kc = W.normal_bf16((npages, ps, Hkv, D), qk_std, rng)
        vc = W.normal_bf16((npages, ps, Hkv, D), v_std, rng)
    else:
        table, npages = None, 0
        cap = int(L.max()) + K + 2
        kc = W.normal_bf16((B, cap, Hkv, D), qk_std, rng)
        vc = W.normal_bf16((B, cap, Hkv, D), v_std, rng)
    return t, q, tk, tv, kc, vc, L, table, npages


def _run_attn(c, t, q, tk, tv, kc, vc, L, table, npages, Hkv):
    B = q.shape[0]
    if table is not None:
        bt = torch.from_numpy(table).to(DEV)
        kv = c.kv_desc(Hkv, 128, table.shape[1], bt, kc.shape[1], npages)
    else:
        kv = c.kv_desc(Hkv, 128, kc.shape[1])
    out = c.cure_tree_attn(q.to(DEV), tk.to(DEV), tv.to(DEV), kc.to(DEV), vc.to(DEV), kv,
                           torch.from_numpy(L).to(DEV),
                           torch.from_numpy(t["n_nodes"].astype(np.int32)).to(DEV),
                           torch.from_numpy(t["anc"].view(np.int64)).to(DEV), 1.0 / math.sqrt(128))
    torch.cuda.synchronize()
    assert c.cure_device_error() == 0
    return out.float().cpu().numpy()


def _cmp_attn(got, ref, t, seqs=None):
    B = got.shape[0]
    worst = 0.0
    for b in (range(B) if seqs is None else seqs):
        n = int(t["n_nodes"][b])
        err = np.abs(got[b, :n] - ref[b, :n])
        assert np.all(np.isfinite(got[b, :n]))
        scale = max(1e-3, float(np.abs(ref[b, :n]).max()))
        assert err.max() <= ATTN_ABS_TOL, err.max()
        assert err.max() <= 2e-2 * scale, (err.max(), scale)
        worst = max(worst, err.max())
    return worst


@pytest.mark.parametrize("paged", [False, True])
@pytest.mark.parametrize("Hq,Hkv", [(8, 2), (28, 4), (32, 8)])
@pytest.mark.parametrize("qk_std,v_std", [(1.0, 1.0), (2.0, 1.0), (1 / math.sqrt(128), 1 / math.sqrt(128))])
def test_tree_attn_small(cure, paged, Hq, Hkv, qk_std, v_std):
    # ragged lengths: empty cache, inside one tile, several tiles + tail, more than one split
    lens = [0, 37, 700, 2100]
    t, q, tk, tv, kc, vc, L, table, npages = _attn_case(4, 8, 6, Hq, Hkv, lens, paged, qk_std,
                                                         v_std, seed=Hq + int(paged))
    got = _run_attn(cure, t, q, tk, tv, kc, vc, L, table, npages, Hkv)
    ref = oracle.tree_attn(_f64(q), _f64(tk), _f64(tv), _f64(kc), _f64(vc), L, t["n_nodes"], t["anc"],
                           1.0 / math.sqrt(128), table, 16)
    _cmp_attn(got, ref, t)


@pytest.mark.parametrize("ps", [8, 32, 64])
@pytest.mark.parametrize("Hq,Hkv", [(28, 4), (32, 8)])
def test_tree_attn_page_sizes(cure, ps, Hq, Hkv):
    """Pages of 8, 32 and 64 tokens: a 64-key tile spans 8, 2 or 1 pages (the
    16-token pages of the other cases span 4); ragged lengths as above."""
    lens = [0, 37, 700, 2100, 64, 1000]
    t, q, tk, tv, kc, vc, L, table, npages = _attn_case(6, 8, 6, Hq, Hkv, lens, True, 1.0, 1.0,
                                                         seed=40 + ps, ps=ps)
    got = _run_attn(cure, t, q, tk, tv, kc, vc, L, table, npages, Hkv)
    ref = oracle.tree_attn(_f64(q), _f64(tk), _f64(tv), _f64(kc), _f64(vc), L, t["n_nodes"], t["anc"],
                           1.0 / math.sqrt(128), table, ps)
    _cmp_attn(got, ref, t)


def test_tree_attn_workspace_contents_do_not_matter(cure):
    """The split-KV workspace may hold anything on entry (old counters of
    other launches, garbage): results match those of a zeroed workspace, call
    after call."""
    t, q, tk, tv, kc, vc, L, table, npages = _attn_case(8, 16, 16, 28, 4, [3000, 5000, 40, 2500, 8000, 100,
                                                                         4100, 6100], True, 1.0, 1.0, seed=5)
    bt = torch.from_numpy(table).to(DEV)
    kv = cure.kv_desc(4, 128, table.shape[1], bt, 16, npages)
    args = (q.to(DEV), tk.to(DEV), tv.to(DEV), kc.to(DEV), vc.to(DEV), kv, torch.from_numpy(L).to(DEV),
            torch.from_numpy(t["n_nodes"].astype(np.int32)).to(DEV),
            torch.from_numpy(t["anc"].view(np.int64)).to(DEV), 1.0 / math.sqrt(128))
    nbytes = cure.cure_tree_attn_workspace_size(8, q.shape[1], 28, kv)
    ws0 = torch.zeros(nbytes, dtype=torch.uint8, device=DEV)
    ref = cure.cure_tree_attn(*args, workspace=ws0).float().cpu().numpy()
    g = torch.Generator(device=DEV).manual_seed(1)
    for fill in ("ones", "random", "random"):
        ws = torch.full((nbytes,), 255, dtype=torch.uint8, device=DEV) if fill == "ones" else \
            torch.randint(0, 256, (nbytes,), dtype=torch.uint8, device=DEV, generator=g)
        for _ in range(2):
            got = cure.cure_tree_attn(*args, workspace=ws).float().cpu().numpy()
            assert cure.cure_device_error() == 0
            for b in range(8):
                n = int(t["n_nodes"][b])
                # the last arriving piece of a split unit varies from run to
                # run, which may move a result by a bf16 rounding step
                assert np.all(np.isfinite(got[b, :n])), (fill, b)
                assert np.abs(got[b, :n] - ref[b, :n]).max() <= 1e-2, (fill, b)


def test_tree_attn_wide_tree_two_words(cure):
    """n_max = 1 + 32 + 64 = 97 nodes: two ancestor words, two tree tiles."""
    t, q, tk, tv, kc, vc, L, table, npages = _attn_case(2, 32, 64, 28, 4, [300, 1500], False, 1.0, 1.0,
                                                         seed=7, tau=4.0)
    assert t["n_nodes"].max() > 64
    got = _run_attn(cure, t, q, tk, tv, kc, vc, L, table, npages, 4)
    ref = oracle.tree_attn(_f64(q), _f64(tk), _f64(tv), _f64(kc), _f64(vc), L, t["n_nodes"], t["anc"],
                           1.0 / math.sqrt(128))
    _cmp_attn(got, ref, t)


def _in_place_case(B, K, budget, Hq, Hkv, lens, paged, seed, tau=1.0, ps=16):
    """An attention case in the in-place layout: caches with room for the
    tree, node j's K/V rows written at cache slot L_b + j."""
    t, q, tk, tv, _, _, L, _, _ = _attn_case(B, K, budget, Hq, Hkv, lens, False, 1.0, 1.0, seed, tau=tau)
    rng = np.random.default_rng(seed + 1000)
    N = 1 + K + budget
    D = 128
    if paged:
        table, npages = W.block_table(L, N - 1, seed, ps)     # pages for slots 0..L_b + N - 1
        kc = W.normal_bf16((npages, ps, Hkv, D), 1.0, rng)
        vc = W.normal_bf16((npages, ps, Hkv, D), 1.0, rng)
    else:
        table, npages = None, 0
        kc = W.normal_bf16((B, int(L.max()) + N + 3, Hkv, D), 1.0, rng)
        vc = W.normal_bf16((B, int(L.max()) + N + 3, Hkv, D), 1.0, rng)
    for b in range(B):
        for j in range(int(t["n_nodes"][b])):
            sl = int(L[b]) + j
            if paged:
                kc[table[b, sl // ps], sl % ps] = tk[b, j]
                vc[table[b, sl // ps], sl % ps] = tv[b, j]
            else:
                kc[b, sl] = tk[b, j]
                vc[b, sl] = tv[b, j]
    return t, q, kc, vc, L, table, npages


def _run_attn_in_place(c, t, q, kc, vc, L, table, npages, Hkv):
    if table is not None:
        kv = c.kv_desc(Hkv, 128, table.shape[1], torch.from_numpy(table).to(DEV), kc.shape[1], npages)
    else:
        kv = c.kv_desc(Hkv, 128, kc.shape[1])
    out = c.cure_tree_attn(q.to(DEV), None, None, kc.to(DEV), vc.to(DEV), kv, torch.from_numpy(L).to(DEV),
                           torch.from_numpy(t["n_nodes"].astype(np.int32)).to(DEV),
                           torch.from_numpy(t["anc"].view(np.int64)).to(DEV), 1.0 / math.sqrt(128))
    torch.cuda.synchronize()
    assert c.cure_device_error() == 0
    return out.float().cpu().numpy()


@pytest.mark.parametrize("paged", [False, True])
@pytest.mark.parametrize("Hq,Hkv", [(8, 2), (28, 4), (32, 8)])
def test_tree_attn_in_place(cure, paged, Hq, Hkv):
    """The in-place layout: cache lengths that put the tree at every kind of
    tile offset (L = 0, inside the first tile, L a multiple of 64, one key
    before a tile boundary, several tiles, more than one split)."""
    lens = [0, 37, 64, 127, 700, 2100]
    t, q, kc, vc, L, table, npages = _in_place_case(6, 8, 6, Hq, Hkv, lens, paged, seed=40 + Hq)
    got = _run_attn_in_place(cure, t, q, kc, vc, L, table, npages, Hkv)
    ref = oracle.tree_attn(_f64(q), None, None, _f64(kc), _f64(vc), L, t["n_nodes"], t["anc"],
                           1.0 / math.sqrt(128), table, 16)
    _cmp_attn(got, ref, t)


@pytest.mark.parametrize("paged", [False, True])
def test_tree_attn_in_place_two_words(cure, paged):
    """97-node trees in the in-place layout: the ancestor window of a tile
    straddles the two words at every bit offset."""
    lens = [300, 1500, 1, 63, 64, 65]
    t, q, kc, vc, L, table, npages = _in_place_case(6, 32, 64, 28, 4, lens, paged, seed=8, tau=4.0)
    assert t["n_nodes"].max() > 64
    got = _run_attn_in_place(cure, t, q, kc, vc, L, table, npages, 4)
    ref = oracle.tree_attn(_f64(q), None, None, _f64(kc), _f64(vc), L, t["n_nodes"], t["anc"],
                           1.0 / math.sqrt(128), table, 16)
    _cmp_attn(got, ref, t)


def test_tree_attn_full_serve_layer_sampled(cure):
    """One layer at the benchmark's serving shape (batch 32, 28/4 heads, paged
    16-token blocks, lengths U[1024, 8192]); the oracle checks 3 sequences."""
    w = W.WORKLOADS["serve32"]
    d, ids, margin = _tree_inputs(w)
    L = W.cache_lengths(w)
    t = oracle.build_tree(ids, margin, d.root_tok, L, w.tau, w.budget, w.branches, 1)
    table, npages = W.block_table(L, w.block, w.seed)
    rng = np.random.default_rng(3)
    N, D = w.n_max, 128
    q = W.normal_bf16((w.batch, N, w.heads_q, D), 1.0, rng)
    tk = W.normal_bf16((w.batch, N, w.heads_kv, D), 1.0, rng)
    tv = W.normal_bf16((w.batch, N, w.heads_kv, D), 1.0, rng)
    g = torch.Generator(device=DEV).manual_seed(11)
    kc = torch.randn(npages, 16, w.heads_kv, D, generator=g, device=DEV, dtype=torch.float32).to(torch.bfloat16)
    vc = torch.randn(npages, 16, w.heads_kv, D, generator=g, device=DEV, dtype=torch.float32).to(torch.bfloat16)
    bt = torch.from_numpy(table).to(DEV)
    kv = cure.kv_desc(w.heads_kv, D, table.shape[1], bt, 16, npages)
    out = cure.cure_tree_attn(q.to(DEV), tk.to(DEV), tv.to(DEV), kc, vc, kv, torch.from_numpy(L).to(DEV),
                              torch.from_numpy(t["n_nodes"].astype(np.int32)).to(DEV),
                              torch.from_numpy(t["anc"].view(np.int64)).to(DEV), 1.0 / math.sqrt(D))
    torch.cuda.synchronize()
    assert cure.cure_device_error() == 0
    got = out.float().cpu().numpy()
    seqs = [int(np.argmax(t["n_nodes"])), int(np.argmax(L)), int(np.argmin(L))]
    ref = oracle.tree_attn(_f64(q), _f64(tk), _f64(tv), _f64(kc.cpu()), _f64(vc.cpu()), L, t["n_nodes"],
                           t["anc"], 1.0 / math.sqrt(D), table, 16, seqs=seqs)
    _cmp_attn(got, ref, t, seqs)


def test_tree_attn_maximum_batch(cure):
    """256 sequences, the most one call takes: the per-sequence prefix sums
    span eight warp-wide passes and the schedule holds 1024 units over the
    CTAs; short ragged caches (0 to 300 keys, paged) and trees of up to 9
    nodes, every sequence checked against the oracle."""
    B, K, budget = 256, 4, 4
    rng = np.random.default_rng(256)
    lens = rng.integers(0, 301, size=B)
    lens[:4] = [0, 1, 64, 300]
    t, q, tk, tv, kc, vc, L, table, npages = _attn_case(B, K, budget, 32, 8, lens, True, 1.0, 1.0, seed=256)
    got = _run_attn(cure, t, q, tk, tv, kc, vc, L, table, npages, 8)
    ref = oracle.tree_attn(_f64(q), _f64(tk), _f64(tv), _f64(kc), _f64(vc), L, t["n_nodes"], t["anc"],
                           1.0 / math.sqrt(128), table, 16)
    _cmp_attn(got, ref, t)


@pytest.mark.parametrize("name,budget", [("single8b", None), ("long64", None), ("sweep16", 64)])
def test_tree_attn_config_layer_sampled(cure, name, budget):
    """One layer at the other configurations' full shapes, contiguous caches:
    single8b (1 x 4096, 32/8 heads), long64 (64 x 32768, 64/8 heads, depth-2
    repairs, 49 nodes: two row groups per kv head) and sweep16 at R = 64 (16 x
    8192, up to 97 nodes: two ancestor words).  The oracle checks two
    sequences, on their own."""
    w = W.WORKLOADS[name]
    budget = w.budget if budget is None else budget
    wt = w.replace(vocab=4096)  # the tree does not depend on the vocabulary
    d, ids, margin = _tree_inputs(wt)
    L = W.cache_lengths(w)
    t = oracle.build_tree(ids, margin, d.root_tok, L, w.tau, budget, w.branches, w.repair_depth,
                          d.redraft if w.repair_depth > 1 else None)
    rng = np.random.default_rng(17)
    N, D = 1 + w.block + budget, 128
    q = W.normal_bf16((w.batch, N, w.heads_q, D), 1.0, rng)
    tk = W.normal_bf16((w.batch, N, w.heads_kv, D), 1.0, rng)
    tv = W.normal_bf16((w.batch, N, w.heads_kv, D), 1.0, rng)
    cap = int(L.max())
    g = torch.Generator(device=DEV).manual_seed(19)
    kc = torch.randn(w.batch, cap, w.heads_kv, D, generator=g, device=DEV, dtype=torch.bfloat16)
    vc = torch.randn(w.batch, cap, w.heads_kv, D, generator=g, device=DEV, dtype=torch.bfloat16)
    kv = cure.kv_desc(w.heads_kv, D, cap)
    out = cure.cure_tree_attn(q.to(DEV), tk.to(DEV), tv.to(DEV), kc, vc, kv, torch.from_numpy(L).to(DEV),
                              torch.from_numpy(t["n_nodes"].astype(np.int32)).to(DEV),
                              torch.from_numpy(t["anc"].view(np.int64)).to(DEV), 1.0 / math.sqrt(D))
    torch.cuda.synchronize()
    assert cure.cure_device_error() == 0
    got = out.float().cpu().numpy()
    seqs = sorted({int(np.argmax(t["n_nodes"])), int(np.argmin(L))})
    sub = {k_: v[seqs] for k_, v in t.items()}
    ref = oracle.tree_attn(_f64(q)[seqs], _f64(tk)[seqs], _f64(tv)[seqs], _f64(kc[seqs].cpu()),
                           _f64(vc[seqs].cpu()), L[seqs], sub["n_nodes"], sub["anc"], 1.0 / math.sqrt(D))
    _cmp_attn(got[seqs], ref, sub)


# ------------------------------------------------------------------ accept
def _target_for(w, d, t, seed):
    truth = W.target_truth(w, d, seed)
    ids = W.synthetic_target_ids(truth, t["n_nodes"], t["tok"], t["parent"], t["depth"], w.vocab, seed)
    return W.target_logits(ids, w.vocab, seed)


def _gpu_tree_dict(t):
    return {k: torch.from_numpy((v.view(np.int64) if k == "anc" else v.astype(np.int32))).to(DEV)
            for k, v in t.items()}


@pytest.mark.parametrize("name", ["tiny", "single8b", "serve32"])
def test_accept_workloads(cure, name):
    w = W.WORKLOADS[name]
    d, ids, margin = _tree_inputs(w)
    L = W.cache_lengths(w)
    t = oracle.build_tree(ids, margin, d.root_tok, L, w.tau, w.budget, w.branches, 1)
    tl = _target_for(w, d, t, w.seed)
    acc = cure.cure_accept(_gpu_tree_dict(t), w.block, target_logits=tl.to(DEV))
    targ_rows = _f64(tl).reshape(-1, w.vocab)
    o_targ = oracle.row_argmax(targ_rows).reshape(w.batch, w.n_max)
    o_acc = oracle.accept(o_targ, t["n_nodes"], t["tok"], t["parent"], t["depth"], t["anc"], w.block)
    g_targ = acc["targ"].cpu().numpy()
    for b in range(w.batch):
        n = int(t["n_nodes"][b])
        assert np.array_equal(g_targ[b, :n], o_targ[b, :n])
        assert (g_targ[b, n:] == -1).all()
    for key in ("accept_len", "best_node", "path_nodes", "out_tokens", "diverge_depth"):
        assert np.array_equal(acc[key].cpu().numpy(), o_acc[key]), key


def test_accept_full_long_shape_sampled(cure):
    """The long-context shape's target argmax (64 x 49 rows of 128256 logits,
    one CTA per row) and walk with depth-2 repairs.  The oracle recomputes 8
    sampled sequences (the largest tree among them); every other valid row
    must give the planted id, which lies 8 above N(0, 1) noise."""
    w = W.WORKLOADS["long64"]
    wt = w.replace(vocab=4096)          # the tree does not depend on V
    d, ids, margin = _tree_inputs(wt)
    L = W.cache_lengths(w)
    t = oracle.build_tree(ids, margin, d.root_tok, L, w.tau, w.budget, w.branches, 2, d.redraft)
    truth = W.target_truth(wt, d, w.seed)
    planted = W.synthetic_target_ids(truth, t["n_nodes"], t["tok"], t["parent"], t["depth"], w.vocab, w.seed)
    B, N, V = w.batch, w.n_max, w.vocab
    g = torch.Generator(device=DEV).manual_seed(w.seed)
    x = torch.randn(B, N, V, generator=g, device=DEV).to(torch.bfloat16)
    pid = torch.from_numpy(planted).to(DEV)
    x.scatter_(2, pid[:, :, None], 8.0)
    acc = cure.cure_accept(_gpu_tree_dict(t), w.block, target_logits=x)
    g_targ = acc["targ"].cpu().numpy()
    n = t["n_nodes"]
    for b in range(B):
        assert np.array_equal(g_targ[b, :n[b]], planted[b, :n[b]]), b
        assert (g_targ[b, n[b]:] == -1).all()
    rng = np.random.default_rng(2)
    S = np.unique(np.concatenate([[int(np.argmax(n))], rng.choice(B, size=7, replace=False)]))
    o_targ = np.full((len(S), N), -1, dtype=np.int64)
    for i, b in enumerate(S):
        o_targ[i, :n[b]] = oracle.row_argmax(_f64(x[b, :n[b]]))
        assert np.array_equal(g_targ[b, :n[b]], o_targ[i, :n[b]]), b
    o_acc = oracle.accept(o_targ, n[S], t["tok"][S], t["parent"][S], t["depth"][S], t["anc"][S], w.block)
    for key in ("accept_len", "best_node", "path_nodes", "out_tokens", "diverge_depth"):
        assert np.array_equal(acc[key].cpu().numpy()[S], o_acc[key]), key
    assert cure.cure_device_error() == 0


@pytest.mark.parametrize("B,N,V", [(3, 9, 4099), (2, 5, 1001), (1, 4, 8), (2, 3, 9), (4, 33, 151937),
                                   (40, 33, 32003)])
def test_target_argmax_ragged_rows_and_ties(cure, B, N, V):
    """The ring-fed target argmax on rows that start off a 16-byte boundary
    (odd vocabularies), vocabularies smaller than one vector, few rows (rows
    split over a cluster) and many, with exact ties and -inf: the ids must be
    the oracle's first maximum, and rows past n_nodes -1."""
    rng = np.random.default_rng(B * 1000 + V)
    x = (rng.integers(-4, 5, size=(B, N, V)) * 0.5).astype(np.float32)   # many exact ties
    x[0, 0, :] = -np.inf
    x[0, 0, V - 1] = 1.0                              # the maximum in the last id
    if N > 1:
        x[0, 1, :] = -np.inf                          # no finite logit: id 0
    logits = W.to_bf16(x)
    n = rng.integers(1, N + 1, size=B).astype(np.int32)
    n[0] = N
    tree = {"n_nodes": torch.from_numpy(n).to(DEV),
            "tok": torch.zeros(B, N, dtype=torch.int32, device=DEV),
            "parent": torch.zeros(B, N, dtype=torch.int32, device=DEV),
            "depth": torch.zeros(B, N, dtype=torch.int32, device=DEV),
            "anc": torch.ones(B, N, (N + 63) // 64, dtype=torch.int64, device=DEV)}
    tree["parent"][:, 0] = -1
    acc = cure.cure_accept(tree, 1 if N < 3 else 2, target_logits=logits.to(DEV))
    got = acc["targ"].cpu().numpy()
    want = oracle.row_argmax(_f64(logits).reshape(-1, V)).reshape(B, N)
    for b in range(B):
        assert np.array_equal(got[b, :n[b]], want[b, :n[b]]), b
        assert (got[b, n[b]:] == -1).all()
    assert got[0, 0] == V - 1


@pytest.mark.parametrize("name", ["sweep16", "serve32", "single8b"])
def test_budget_zero_is_prefix_verification_on_the_gpu(cure, name):
    """R = 0 (Sec. 3.1, Eq. 1 with no repair nodes): the tree is the draft
    chain alone, and the walk must accept exactly the longest prefix of the
    chain that the target's tokens confirm, i.e. plain block-parallel prefix
    verification, computed here by a direct scan."""
    w = W.WORKLOADS[name].replace(vocab=4096, budget=0)
    d, ids, margin = _tree_inputs(w)
    L = W.cache_lengths(w)
    t = oracle.build_tree(ids, margin, d.root_tok, L, w.tau, 0, w.branches, 1)
    assert (t["n_nodes"] == w.block + 1).all()
    truth = W.target_truth(w, d, w.seed)
    targ = W.synthetic_target_ids(truth, t["n_nodes"], t["tok"], t["parent"], t["depth"], w.vocab, w.seed)
    acc = cure.cure_accept(_gpu_tree_dict(t), w.block, targ=torch.from_numpy(targ.astype(np.int32)).to(DEV))
    a = acc["accept_len"].cpu().numpy()
    dv = acc["diverge_depth"].cpu().numpy()
    out = acc["out_tokens"].cpu().numpy()
    for b in range(w.batch):
        e = 0
        while e < w.block and t["tok"][b, e + 1] == targ[b, e]:
            e += 1
        assert a[b] == e, (b, a[b], e)
        assert dv[b] == -1
        assert list(out[b, :e + 1]) == list(t["tok"][b, 1:e + 1]) + [targ[b, e]]


@pytest.mark.parametrize("seed", range(8))
def test_accept_random_trees_with_ids(cure, seed):
    """Random trees (depth-2 repairs included) with small-alphabet targets so
    that many paths verify, through the precomputed-ids entry."""
    rng = np.random.default_rng(seed)
    B, K = 6, int(rng.integers(2, 20))
    k, branches, depth = 4, 4, 1 + seed % 2
    budget = int(rng.integers(0, 40))
    margin = (rng.integers(0, 8, size=(B, K)) * 0.25).astype(np.float32)
    ids = np.tile(np.arange(k), (B, K, 1))
    redraft = rng.integers(0, 3, size=(B, K, branches - 1))
    t = oracle.build_tree(ids, margin, rng.integers(0, 3, size=B), rng.integers(0, 99, size=B), 1.5,
                          budget, branches, depth, redraft)
    targ = rng.integers(0, 3, size=t["tok"].shape)
    o_acc = oracle.accept(targ, t["n_nodes"], t["tok"], t["parent"], t["depth"], t["anc"], K)
    acc = cure.cure_accept(_gpu_tree_dict(t), K, targ=torch.from_numpy(targ.astype(np.int32)).to(DEV))
    for key in ("accept_len", "best_node", "path_nodes", "out_tokens", "diverge_depth"):
        assert np.array_equal(acc[key].cpu().numpy(), o_acc[key]), key


# ------------------------------------------------------ stochastic verification
def _sum_tol(V):
    """Relative bound on the kernel's float32 cumulative sums for a row of V
    ids: each lane adds 8 * ceil(V / 1024) terms in sequence (four warp
    segments of 32 lanes, eight ids per group), the walk adds up to
    ceil(V / 1024) chunk totals, and the warp and segment reductions, the
    rescales and the chunk scan add fewer than 64 more roundings; each
    rounding contributes at most 2^-24 of the sum, and ex2.approx a further
    2^-20 (its relative error, with room)."""
    c = -(-V // 1024)
    return (9 * c + 64) * 2.0 ** -24 + 2.0 ** -20


def _valid_sample(x, T, u, y, tol=None):
    """y is a valid inverse-CDF draw for u: an id of nonzero probability whose
    cumulative range (float64) contains u Z, up to the kernel's float32
    summation bound (tol Z)."""
    tol = _sum_tol(len(x)) if tol is None else tol
    m = x.max()
    if m == -np.inf:
        return y == 0
    p = np.exp((x - m) / T)
    c = np.cumsum(p)
    Z = c[-1]
    r = min(max(u, 0.0), float(np.nextafter(np.float32(1), np.float32(0)))) * Z
    if not (0 <= y < len(x)) or p[y] <= 0:
        return False
    lo = c[y - 1] if y > 0 else 0.0
    return lo - tol * Z <= r <= c[y] + tol * Z


@pytest.mark.parametrize("V", [1000, 4099, 151936])
@pytest.mark.parametrize("T", [0.5, 1.0, 2.0])
def test_sample_target_inverse_cdf(cure, V, T):
    rng = np.random.default_rng(V + int(10 * T))
    B, N = 4, 9
    n = np.array([1, 5, 9, 3], dtype=np.int32)
    x = (rng.standard_normal((B, N, V)) * 2.0).astype(np.float32)
    x[2, 1, :] = -np.inf
    x[2, 1, 17] = 3.0                 # one finite logit
    x[2, 2, :] = -np.inf              # none: id 0
    x[3, 0, : V // 2] = -np.inf       # the first half impossible
    logits = W.to_bf16(x)
    u = rng.random((B, N)).astype(np.float32)
    u[1, 0], u[1, 1], u[3, 0] = 0.0, np.float32(0.9999999), 0.0
    got = cure.cure_sample_target(logits.to(DEV), torch.from_numpy(n).to(DEV), torch.from_numpy(u).to(DEV),
                                  T).cpu().numpy()
    assert cure.cure_device_error() == 0
    xf = _f64(logits)
    for b in range(B):
        for j in range(N):
            if j >= n[b]:
                assert got[b, j] == -1
            else:
                assert _valid_sample(xf[b, j], T, float(u[b, j]), int(got[b, j])), (b, j, got[b, j])
    assert got[2, 1] == 17 and got[2, 2] == 0 and got[3, 0] >= V // 2


@pytest.mark.parametrize("T", [1e-30, 1e-38])
def test_sample_target_tiny_temperature_and_huge_logits(cure, T):
    """Temperatures so small that every logit below the maximum has
    probability 0 pick among the ids holding the maximum by the uniform (the
    T -> 0 limit), and logits near the bf16 limit do not overflow: the draws
    equal the oracle's exact inverse CDF (no u near a step boundary)."""
    rng = np.random.default_rng(7)
    B, N, V = 3, 6, 5000
    x = rng.standard_normal((B, N, V)).astype(np.float32)
    ties = rng.choice(V, size=3, replace=False)
    x[0, :, ties] = 9.0                               # three ids share the maximum
    x[1, :, :] = rng.uniform(-3e38, 1e38, size=(N, V)).astype(np.float32)
    x[1, :, 4321] = 3.0e38                            # a maximum near the bf16 limit
    x[2, :, :] = -np.inf
    x[2, :, [5, 17]] = -3.0e38                        # the maximum is very negative
    logits = W.to_bf16(x)
    u = np.tile(np.array([0.05, 0.2, 0.4, 0.6, 0.8, 0.95], np.float32), (B, 1))
    n = np.full(B, N, dtype=np.int32)
    got = cure.cure_sample_target(logits.to(DEV), torch.from_numpy(n).to(DEV), torch.from_numpy(u).to(DEV),
                                  T).cpu().numpy()
    assert cure.cure_device_error() == 0
    want = oracle.sample_target(_f64(logits), n, u.astype(np.float64), T)
    assert np.array_equal(got, want)
    assert set(got[0].tolist()) == set(ties.tolist()) and (got[1] == 4321).all()
    assert set(got[2].tolist()) <= {5, 17}


def test_sample_target_frequencies_follow_softmax(cure):
    """2000 rows of the same 7 logits with u on a grid: the ids drawn match
    the oracle's exact inverse CDF (but for u within rounding of a boundary),
    so their frequencies are the softmax probabilities to one grid step."""
    rng = np.random.default_rng(5)
    B, N, V, T = 250, 8, 7, 0.7
    x = np.broadcast_to(rng.standard_normal(V).astype(np.float32) * 2.0, (B, N, V)).copy()
    logits = W.to_bf16(x)
    M = B * N
    u = ((np.arange(M) + 0.5) / M).astype(np.float32).reshape(B, N)
    n = np.full(B, N, dtype=np.int32)
    got = cure.cure_sample_target(logits.to(DEV), torch.from_numpy(n).to(DEV), torch.from_numpy(u).to(DEV),
                                  T).cpu().numpy()
    want = oracle.sample_target(_f64(logits), n, u.astype(np.float64), T)
    assert (got != want).sum() <= 2
    p = np.exp(_f64(logits)[0, 0] / T)
    p /= p.sum()
    assert np.abs(np.bincount(got.ravel(), minlength=V) / M - p).max() <= 2.0 / M


def test_sample_target_then_accept(cure):
    """Stochastic verification end to end: sampled target tokens, then the
    unchanged acceptance walk, against the oracle walk on the same samples."""
    w = W.WORKLOADS["tiny"].replace(batch=8, vocab=512)
    rng = np.random.default_rng(9)
    d, ids, margin = _tree_inputs(w)
    L = W.cache_lengths(w)
    t = oracle.build_tree(ids, margin, d.root_tok, L, w.tau, w.budget, w.branches, 1)
    N = w.n_max
    # target logits that favour the draft's tokens, so that paths get accepted
    x = rng.standard_normal((w.batch, N, w.vocab)).astype(np.float32)
    for b in range(w.batch):
        for j in range(int(t["n_nodes"][b])):
            kids = [c for c in range(int(t["n_nodes"][b])) if t["parent"][b, c] == j]
            for c in kids:
                x[b, j, int(t["tok"][b, c])] += 9.0
    logits = W.to_bf16(x)
    u = rng.random((w.batch, N)).astype(np.float32)
    tree_d = _gpu_tree_dict(t)
    targ = cure.cure_sample_target(logits.to(DEV), tree_d["n_nodes"], torch.from_numpy(u).to(DEV), 1.0)
    acc = cure.cure_accept(tree_d, w.block, targ=targ)
    g = targ.cpu().numpy()
    xf = _f64(logits)
    for b in range(w.batch):
        for j in range(int(t["n_nodes"][b])):
            assert _valid_sample(xf[b, j], 1.0, float(u[b, j]), int(g[b, j]))
    o = oracle.accept(g, t["n_nodes"], t["tok"], t["parent"], t["depth"], t["anc"], w.block)
    for key in ("accept_len", "best_node", "path_nodes", "out_tokens", "diverge_depth"):
        assert np.array_equal(acc[key].cpu().numpy(), o[key]), key
    assert o["accept_len"].max() > 0


def test_sample_target_serving_shape_sampled(cure):
    """The serving shape (32 x 33 rows of 151936 logits), rows checked on a sample."""
    B, N, V = 32, 33, 151936
    g = torch.Generator(device=DEV).manual_seed(11)
    logits = (torch.randn(B, N, V, generator=g, device=DEV) * 3).to(torch.bfloat16)
    n = torch.randint(17, N + 1, (B,), generator=g, device=DEV, dtype=torch.int32)
    u = torch.rand(B, N, generator=g, device=DEV)
    got = cure.cure_sample_target(logits, n, u, 0.8).cpu().numpy()
    nh, uh = n.cpu().numpy(), u.cpu().numpy()
    rng = np.random.default_rng(3)
    for _ in range(24):
        b, j = int(rng.integers(0, B)), int(rng.integers(0, N))
        if j >= nh[b]:
            assert got[b, j] == -1
        else:
            xr = logits[b, j].float().cpu().numpy().astype(np.float64)
            assert _valid_sample(xr, 0.8, float(uh[b, j]), int(got[b, j])), (b, j)


# ------------------------------------------------------------------ resync
@pytest.mark.parametrize("paged", [0, 8, 16, 32, 64])
def test_resync(cure, paged):
    """paged: the page size in tokens, 0 for the contiguous layout."""
    rng = np.random.default_rng(21 + int(paged))
    B, K, budget, Hkv, D, layers = 5, 8, 6, 4, 128, 3
    margin = (rng.integers(0, 8, size=(B, K)) * 0.25).astype(np.float32)
    ids = np.tile(np.arange(3), (B, K, 1))
    t = oracle.build_tree(ids, margin, rng.integers(0, 3, size=B), rng.integers(0, 99, size=B), 1.5,
                          budget, 3, 1)
    targ = rng.integers(0, 3, size=t["tok"].shape)
    o_acc = oracle.accept(targ, t["n_nodes"], t["tok"], t["parent"], t["depth"], t["anc"], K)
    L = rng.integers(0, 200, size=B).astype(np.int32)
    N = 1 + K + budget
    tk = W.normal_bf16((layers, B, N, Hkv, D), 1.0, rng)
    tv = W.normal_bf16((layers, B, N, Hkv, D), 1.0, rng)
    if paged:
        table, npages = W.block_table(L, K, 5, paged)
        shape = (npages, paged, Hkv, D)
        kv = cure.kv_desc(Hkv, D, table.shape[1], torch.from_numpy(table).to(DEV), paged, npages)
    else:
        table = None
        shape = (B, int(L.max()) + K + 1, Hkv, D)
        kv = cure.kv_desc(Hkv, D, shape[1])
    kcs = [W.normal_bf16(shape, 1.0, rng) for _ in range(layers)]
    vcs = [W.normal_bf16(shape, 1.0, rng) for _ in range(layers)]
    kd = [x.to(DEV) for x in kcs]
    vd = [x.to(DEV) for x in vcs]
    acc = {k_: torch.from_numpy(v.astype(np.int32)).to(DEV) for k_, v in o_acc.items()}
    rs = cure.cure_resync_kv(kd, vd, kv, tk.to(DEV), tv.to(DEV), acc, torch.from_numpy(L).to(DEV), K)
    torch.cuda.synchronize()
    assert cure.cure_device_error() == 0
    ko = [_f64(x) for x in kcs]
    vo = [_f64(x) for x in vcs]
    o_rs = oracle.resync(ko, vo, _f64(tk), _f64(tv), o_acc["path_nodes"], o_acc["accept_len"],
                         o_acc["diverge_depth"], o_acc["out_tokens"], L, K, table, paged or 16)
    for key in ("cache_len", "draft_valid_len", "replay_tokens", "n_replay"):
        assert np.array_equal(rs[key].cpu().numpy(), o_rs[key]), key
    for l in range(layers):
        assert np.array_equal(_f64(kd[l].cpu()), ko[l])
        assert np.array_equal(_f64(vd[l].cpu()), vo[l])


@pytest.mark.parametrize("paged", [0, 16])
def test_resync_in_place_layout(cure, paged):
    """The in-place layout: the path rows come from cache slots L + node and
    only the repair rows move; the whole cache must match the oracle."""
    rng = np.random.default_rng(31 + int(paged))
    B, K, budget, Hkv, D, layers = 6, 8, 6, 4, 128, 3
    margin = (rng.integers(0, 8, size=(B, K)) * 0.25).astype(np.float32)
    ids = np.tile(np.arange(3), (B, K, 1))
    t = oracle.build_tree(ids, margin, rng.integers(0, 3, size=B), rng.integers(0, 99, size=B), 1.5,
                          budget, 3, 1)
    targ = rng.integers(0, 3, size=t["tok"].shape)
    o_acc = oracle.accept(targ, t["n_nodes"], t["tok"], t["parent"], t["depth"], t["anc"], K)
    assert (o_acc["diverge_depth"] >= 0).any() and (o_acc["diverge_depth"] < 0).any()
    L = rng.integers(0, 200, size=B).astype(np.int32)
    N = 1 + K + budget
    if paged:
        table, npages = W.block_table(L, N - 1, 5, paged)
        shape = (npages, paged, Hkv, D)
        kv = cure.kv_desc(Hkv, D, table.shape[1], torch.from_numpy(table).to(DEV), paged, npages)
    else:
        table = None
        shape = (B, int(L.max()) + N + 1, Hkv, D)
        kv = cure.kv_desc(Hkv, D, shape[1])
    kcs = [W.normal_bf16(shape, 1.0, rng) for _ in range(layers)]
    vcs = [W.normal_bf16(shape, 1.0, rng) for _ in range(layers)]
    kd = [x.to(DEV) for x in kcs]
    vd = [x.to(DEV) for x in vcs]
    acc = {k_: torch.from_numpy(v.astype(np.int32)).to(DEV) for k_, v in o_acc.items()}
    rs = cure.cure_resync_kv(kd, vd, kv, None, None, acc, torch.from_numpy(L).to(DEV), K, n_max=N)
    torch.cuda.synchronize()
    assert cure.cure_device_error() == 0
    ko = [_f64(x) for x in kcs]
    vo = [_f64(x) for x in vcs]
    o_rs = oracle.resync(ko, vo, None, None, o_acc["path_nodes"], o_acc["accept_len"],
                         o_acc["diverge_depth"], o_acc["out_tokens"], L, K, table, paged or 16)
    for key in ("cache_len", "draft_valid_len", "replay_tokens", "n_replay"):
        assert np.array_equal(rs[key].cpu().numpy(), o_rs[key]), key
    for l in range(layers):
        assert np.array_equal(_f64(kd[l].cpu()), ko[l])
        assert np.array_equal(_f64(vd[l].cpu()), vo[l])


def test_resync_in_place_lengths(cure):
    """cache_len_out may alias cache_len_in."""
    B, K = 3, 4
    acc = dict(accept_len=torch.tensor([0, 2, 4], dtype=torch.int32, device=DEV),
               path_nodes=torch.tensor([[0, -1, -1, -1, -1, -1], [0, 1, 5, -1, -1, -1], [0, 1, 2, 3, 4, -1]],
                                       dtype=torch.int32, device=DEV),
               diverge_depth=torch.tensor([-1, 2, -1], dtype=torch.int32, device=DEV),
               out_tokens=torch.tensor([[7, -1, -1, -1, -1, -1], [3, 9, 8, -1, -1, -1], [1, 2, 3, 4, 5, -1]],
                                       dtype=torch.int32, device=DEV))
    lens = torch.tensor([10, 20, 30], dtype=torch.int32, device=DEV)
    kv = cure.kv_desc(4, 128, 64)
    rs = cure.cure_resync_kv([], [], kv, None, None, acc, lens, K, cache_len_out=lens)
    torch.cuda.synchronize()
    assert lens.tolist() == [11, 23, 35]
    assert rs["draft_valid_len"].tolist() == [11, 22, 35]
    assert rs["n_replay"].tolist() == [1, 2, 1]
    assert rs["replay_tokens"].cpu().numpy()[1, :2].tolist() == [9, 8]


# ------------------------------------------------------------------ device-side checks
def test_device_error_word_reports_bad_pages_and_slots(cure):
    """Bad data the host cannot see: a missing page and a slot past the capacity.
    The kernels skip the access and raise bits; the context stays usable."""
    B, K, Hkv, D = 2, 4, 2, 128
    acc = dict(accept_len=torch.tensor([1, 1], dtype=torch.int32, device=DEV),
               path_nodes=torch.tensor([[0, 1, -1, -1, -1, -1]] * 2, dtype=torch.int32, device=DEV),
               diverge_depth=torch.tensor([-1, -1], dtype=torch.int32, device=DEV),
               out_tokens=torch.tensor([[1, 2, -1, -1, -1, -1]] * 2, dtype=torch.int32, device=DEV))
    tk = torch.zeros(1, B, 1 + K, Hkv, D, dtype=torch.bfloat16, device=DEV)
    table = torch.tensor([[0, -1], [1, 2]], dtype=torch.int32, device=DEV)
    pages = torch.zeros(3, 16, Hkv, D, dtype=torch.bfloat16, device=DEV)
    kv = cure.kv_desc(Hkv, D, 2, table, 16, 3)
    assert cure.cure_device_error() == 0
    # sequence 0 writes slots 16..17 (page entry -1); sequence 1 writes slots 40..41 (past 2 pages)
    lens = torch.tensor([16, 40], dtype=torch.int32, device=DEV)
    cure.cure_resync_kv([pages], [pages.clone()], kv, tk, tk.clone(), acc, lens, K)
    bits = cure.cure_device_error()
    assert bits & cure.DEVERR_PAGE and bits & cure.DEVERR_SLOT
    assert cure.cure_device_error() == 0
    # the context is still usable
    x = torch.ones(4, device=DEV)
    assert float(x.sum()) == 4.0


# ------------------------------------------------------------------ whole step
def test_full_step_serve_shape(cure):
    """The six stages chained through RepairVerifyStep at the benchmark's shape
    (2 layers); integers compared in full, attention on sampled sequences."""
    from paper_2608_00531_gb300.step import RepairVerifyStep, StepInputs
    w = W.WORKLOADS["serve32"]
    layers = 2
    d = W.draft_block(w)
    L = W.cache_lengths(w)
    x64 = _f64(d.logits).reshape(-1, w.vocab)
    o_ids, _, o_m, _, _ = oracle.score_draft(x64, w.topk)
    B, K, k, N = w.batch, w.block, w.topk, w.n_max
    t = oracle.build_tree(o_ids.reshape(B, K, k), o_m.astype(np.float32).reshape(B, K), d.root_tok, L,
                          w.tau, w.budget, w.branches, 1)
    tl = _target_for(w, d, t, w.seed)
    table, npages = W.block_table(L, K, w.seed)
    rng = np.random.default_rng(9)
    q = W.normal_bf16((layers, B, N, w.heads_q, 128), 1.0, rng)
    tk = W.normal_bf16((layers, B, N, w.heads_kv, 128), 1.0, rng)
    tv = W.normal_bf16((layers, B, N, w.heads_kv, 128), 1.0, rng)
    g = torch.Generator(device=DEV).manual_seed(5)
    kcs = [torch.randn(npages, 16, w.heads_kv, 128, generator=g, device=DEV).to(torch.bfloat16) for _ in range(layers)]
    vcs = [torch.randn(npages, 16, w.heads_kv, 128, generator=g, device=DEV).to(torch.bfloat16) for _ in range(layers)]
    seqs = [int(np.argmax(t["n_nodes"])), 5]
    kc_host = [_f64(c.cpu()) for c in kcs]
    vc_host = [_f64(c.cpu()) for c in vcs]
    bt = torch.from_numpy(table).to(DEV)
    kv = cure.kv_desc(w.heads_kv, 128, table.shape[1], bt, 16, npages)
    st = RepairVerifyStep(B, K, w.vocab, k, w.tau, w.budget, w.branches, 1, layers, w.heads_q, kv, DEV)
    xin = StepInputs(d.logits.to(DEV), torch.from_numpy(d.root_tok).to(DEV), torch.from_numpy(L).to(DEV),
                     None, q.to(DEV), tk.to(DEV), tv.to(DEV), tl.to(DEV))
    r = st.run(xin, kcs, vcs)
    torch.cuda.synchronize()
    assert cure.cure_device_error() == 0
    _cmp_tree(r["tree"], t)
    for l in range(layers):
        ref = oracle.tree_attn(_f64(q[l]), _f64(tk[l]), _f64(tv[l]), kc_host[l], vc_host[l], L, t["n_nodes"],
                               t["anc"], 1.0 / math.sqrt(128), table, 16, seqs=seqs)
        _cmp_attn(r["attn"][l].float().cpu().numpy(), ref, t, seqs)
    o_targ = oracle.row_argmax(_f64(tl).reshape(-1, w.vocab)).reshape(B, N)
    o_acc = oracle.accept(o_targ, t["n_nodes"], t["tok"], t["parent"], t["depth"], t["anc"], K)
    for key in ("accept_len", "best_node", "path_nodes", "out_tokens", "diverge_depth"):
        assert np.array_equal(r["acc"][key].cpu().numpy(), o_acc[key]), key
    o_rs = oracle.resync(kc_host, vc_host, _f64(tk), _f64(tv), o_acc["path_nodes"], o_acc["accept_len"],
                         o_acc["diverge_depth"], o_acc["out_tokens"], L, K, table, 16)
    for key in ("cache_len", "draft_valid_len", "replay_tokens", "n_replay"):
        assert np.array_equal(r["resync"][key].cpu().numpy(), o_rs[key]), key
    for l in range(layers):
        assert np.array_equal(_f64(kcs[l].cpu()), kc_host[l])
        assert np.array_equal(_f64(vcs[l].cpu()), vc_host[l])
    # the same step with its inputs in pinned host memory, streamed in on a
    # copy stream: the same results (the step's buffers are reused, so the
    # first results are copied out first)
    ints = {("tree", k_): v.clone() for k_, v in r["tree"].items()}
    ints.update({("acc", k_): v.clone() for k_, v in r["acc"].items()})
    ints.update({("resync", k_): v.clone() for k_, v in r["resync"].items()})
    attn = r["attn"].float().clone()
    xh = StepInputs(d.logits.pin_memory(), torch.from_numpy(d.root_tok).pin_memory(),
                    torch.from_numpy(L).pin_memory(), None, q.pin_memory(), tk.pin_memory(), tv.pin_memory(),
                    tl.pin_memory())
    # first with the target logits copied by node rows, then whole (a
    # threshold above their size): the same results, fewer bytes the first way
    h2d = []
    for thr in (RepairVerifyStep.NODE_ROWS_MIN_BYTES, 1 << 62):
        st.NODE_ROWS_MIN_BYTES = thr
        r2 = st.run_from_host(xh, kcs, vcs)
        torch.cuda.synchronize()
        assert cure.cure_device_error() == 0
        h2d.append(st.last_h2d_bytes)
        for (grp, key), v in ints.items():
            assert torch.equal(r2[grp][key], v), (grp, key)
        for b in range(B):
            nb = int(t["n_nodes"][b])
            assert float((r2["attn"][:, b, :nb].float() - attn[:, b, :nb]).abs().max()) <= 1e-2, b
    row_bytes = w.vocab * 2
    assert h2d[1] - h2d[0] == int((N - t["n_nodes"]).sum()) * row_bytes
