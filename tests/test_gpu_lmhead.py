"""GPU parity of the fused LM head + argmax (cure_lm_head_argmax) against the oracle.

The kernel accumulates hidden[r] . w_lm[v] in float32 on the tensor cores, the
oracle in float64.  Where the oracle's top two logits of a row are further
apart than twice the float32 accumulation bound, the ids must be equal;
otherwise the kernel's id must be one whose exact logit lies within twice the
bound of the row maximum.  The bound for (r, v) is
    (d_model / 16 + 16) * 2^-22 * sum_k |hidden[r][k] w_lm[v][k]|:
every product of two bf16 values is exact in float32, each K = 16 product
step adds one rounding (allowing truncation, 2^-23, and a factor 2 of room)
to the running sum, and the step itself adds fewer than 16 more.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_00531_gb300 import workload as W

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda:0")


@pytest.fixture(scope="module")
def cure():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_00531_gb300 import cure as c
    torch.cuda.set_device(DEV)
    return c


def _bound(h64, w, d):
    """Per row: the accumulation bound at the largest sum_k |h w| over v."""
    gamma = (d / 16 + 16) * 2.0 ** -22
    ha = np.abs(h64)
    worst = np.zeros(h64.shape[0])
    for v0 in range(0, w.shape[0], 8192):
        wa = np.abs(np.asarray(w[v0:v0 + 8192], dtype=np.float64))
        worst = np.maximum(worst, (ha @ wa.T).max(axis=1))
    return gamma * worst


def _logits(h64, w):
    return np.concatenate([h64 @ np.asarray(w[v0:v0 + 8192], dtype=np.float64).T
                           for v0 in range(0, w.shape[0], 8192)], axis=1)


def _check(got, h64, w, d, want=None):
    """got: the kernel's ids for the rows of h64; returns the rows checked exactly."""
    want = oracle.lm_head_argmax(h64, w) if want is None else want
    lg = _logits(h64, w)
    bnd = _bound(h64, w, d)
    exact = 0
    for r in range(h64.shape[0]):
        row = lg[r]
        top = np.sort(row)[-2:]
        gap = top[1] - top[0]
        y = int(got[r])
        assert 0 <= y < w.shape[0], (r, y)
        if gap > 2 * bnd[r]:
            assert y == int(want[r]), (r, y, int(want[r]), gap, bnd[r])
            exact += 1
        else:
            assert row[y] >= row.max() - 2 * bnd[r], (r, y, row[y], row.max(), bnd[r])
    return exact


@pytest.mark.parametrize("rows,d,V", [(1, 64, 256), (37, 128, 1000), (130, 256, 4099), (300, 192, 20000),
                                      (129, 4096, 3001), (64, 8192, 20011)])
def test_lm_head_argmax_small_shapes(cure, rows, d, V):
    """Ragged rows (M tails), vocabularies ending inside an N tile, several
    K slices (up to d_model 8192, the 70B-class width: 128 of them); unplanted
    rows, so the argmax is decided by noise."""
    rng = np.random.default_rng(rows * 7 + V)
    h = W.to_bf16(rng.standard_normal((rows, d)).astype(np.float32))
    w = W.to_bf16((rng.standard_normal((V, d)) / np.sqrt(d)).astype(np.float32))
    got = cure.cure_lm_head_argmax(h.to(DEV), w.to(DEV)).cpu().numpy()
    assert cure.cure_device_error() == 0
    exact = _check(got, W.bf16_to_f64(h), W.bf16_to_f64(w), d)
    assert exact >= 0.8 * rows


def test_lm_head_argmax_more_m_tiles_than_sms(cure):
    """More 128-row tiles than SMs: one vocab range per tile and a grid of
    more than one wave."""
    rng = np.random.default_rng(8)
    rows, d, V = 160 * 128 + 37, 64, 700
    h = W.to_bf16(rng.standard_normal((rows, d)).astype(np.float32))
    w = W.to_bf16((rng.standard_normal((V, d)) / np.sqrt(d)).astype(np.float32))
    got = cure.cure_lm_head_argmax(h.to(DEV), w.to(DEV)).cpu().numpy()
    assert cure.cure_device_error() == 0
    sel = np.concatenate([np.arange(64), rows - 64 + np.arange(64), rng.choice(rows, 128, replace=False)])
    exact = _check(got[sel], W.bf16_to_f64(h)[sel], W.bf16_to_f64(w), d)
    assert exact >= 0.8 * len(sel)


def test_lm_head_argmax_ties_take_the_lowest_id(cure):
    """Identical weight rows give bit-identical logits; the lowest id must win
    within a tile, across N tiles and across the CTAs' vocab ranges."""
    rng = np.random.default_rng(3)
    rows, d, V = 40, 128, 151936
    w = (rng.standard_normal((V, d)) / np.sqrt(d)).astype(np.float32)
    pairs = [(5, 17), (300, 70000), (1000, 151935), (151000, 151001)]
    for a, b in pairs:
        w[b] = w[a]
    wb = W.to_bf16(w)
    h = rng.standard_normal((rows, d)).astype(np.float32)
    wf = wb.to(torch.float32).numpy()
    for r in range(rows):
        a, _ = pairs[r % len(pairs)]
        h[r] += 30.0 * wf[a]
    hb = W.to_bf16(h)
    got = cure.cure_lm_head_argmax(hb.to(DEV), wb.to(DEV)).cpu().numpy()
    want = oracle.lm_head_argmax(W.bf16_to_f64(hb), wf)
    for r in range(rows):
        assert got[r] == want[r] == pairs[r % len(pairs)][0], (r, got[r], want[r])


def test_lm_head_argmax_out_index_scatter(cure):
    """out_index places each packed row at its [B][n_max] slot; the slots no
    row maps to keep their contents."""
    rng = np.random.default_rng(4)
    B, N, d, V = 5, 9, 128, 3000
    n = np.array([1, 9, 4, 7, 2])
    idx = np.concatenate([b * N + np.arange(n[b]) for b in range(B)]).astype(np.int32)
    rows = len(idx)
    h = W.to_bf16(rng.standard_normal((rows, d)).astype(np.float32))
    w = W.to_bf16((rng.standard_normal((V, d)) / np.sqrt(d)).astype(np.float32))
    targ = torch.full((B, N), -7, dtype=torch.int32, device=DEV)
    cure.cure_lm_head_argmax(h.to(DEV), w.to(DEV), out_index=torch.from_numpy(idx).to(DEV), out=targ)
    flat = cure.cure_lm_head_argmax(h.to(DEV), w.to(DEV)).cpu().numpy()
    t = targ.cpu().numpy().reshape(-1)
    assert np.array_equal(t[idx], flat)
    mask = np.ones(B * N, bool)
    mask[idx] = False
    assert (t[mask] == -7).all()


def test_lm_head_argmax_full_serve_shape_then_accept(cure):
    """The serving shape: the realised tree nodes of batch 32 (block 16, budget
    16) packed, d_model 4096, vocab 151936, with hidden states that plant the
    stand-in target's tokens; every row must give its planted id (8 to 12
    above the noise), 24 sampled rows are recomputed by the oracle, and the
    acceptance walk on the fused path's tokens equals the oracle's walk."""
    w = W.WORKLOADS["serve32"]
    d_model = 4096
    d = W.draft_block(w)
    x = W.bf16_to_f64(d.logits).reshape(-1, w.vocab)
    rows_sel = slice(None)
    o_ids, _, o_m, _, _ = oracle.score_draft(x[rows_sel], w.topk)
    B, K, N = w.batch, w.block, w.n_max
    L = W.cache_lengths(w)
    t = oracle.build_tree(o_ids.reshape(B, K, w.topk), o_m.astype(np.float32).reshape(B, K), d.root_tok, L,
                          w.tau, w.budget, w.branches, 1)
    truth = W.target_truth(w, d, w.seed)
    planted = W.synthetic_target_ids(truth, t["n_nodes"], t["tok"], t["parent"], t["depth"], w.vocab, w.seed)
    n = t["n_nodes"]
    idx = np.concatenate([b * N + np.arange(n[b]) for b in range(B)]).astype(np.int32)
    pl_rows = planted.reshape(-1)[idx]
    wl = W.lm_head_weight(w.vocab, d_model, w.seed)
    h = W.lm_head_hidden(len(idx), wl, w.seed, pl_rows)
    targ = torch.full((B, N), -1, dtype=torch.int32, device=DEV)
    wl_d = wl.to(DEV)
    cure.cure_lm_head_argmax(h.to(DEV), wl_d, out_index=torch.from_numpy(idx).to(DEV), out=targ)
    tree_d = {k: torch.from_numpy((v.view(np.int64) if k == "anc" else v.astype(np.int32))).to(DEV)
              for k, v in t.items()}
    acc = cure.cure_accept(tree_d, K, targ=targ)
    assert cure.cure_device_error() == 0
    g_rows = targ.cpu().numpy().reshape(-1)[idx]
    assert np.array_equal(g_rows, pl_rows)
    rng = np.random.default_rng(0)
    sel = rng.choice(len(idx), size=24, replace=False)
    wf = wl.to(torch.float32).numpy()
    _check(g_rows[sel], W.bf16_to_f64(h)[sel], wf, d_model)
    o_targ = np.full((B, N), -1, dtype=np.int64)
    o_targ.reshape(-1)[idx] = pl_rows
    o_acc = oracle.accept(o_targ, n, t["tok"], t["parent"], t["depth"], t["anc"], K)
    for key in ("accept_len", "best_node", "path_nodes", "out_tokens", "diverge_depth"):
        assert np.array_equal(acc[key].cpu().numpy(), o_acc[key]), key


def test_lm_head_argmax_full_shape_unplanted_rows(cure):
    """d_model 4096, vocab 151936, 300 rows of noise: the argmax is decided by
    small gaps, checked on 16 sampled rows against the float64 oracle within
    the accumulation bound (most of them exactly)."""
    V, d_model, rows = 151936, 4096, 300
    wl = W.lm_head_weight(V, d_model, 77)
    rng = np.random.default_rng(5)
    h = W.to_bf16(rng.standard_normal((rows, d_model)).astype(np.float32))
    got = cure.cure_lm_head_argmax(h.to(DEV), wl.to(DEV)).cpu().numpy()
    assert cure.cure_device_error() == 0
    sel = rng.choice(rows, size=16, replace=False)
    exact = _check(got[sel], W.bf16_to_f64(h)[sel], wl.to(torch.float32).numpy(), d_model)
    assert exact >= 12
