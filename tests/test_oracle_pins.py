"""Pins for the CPU oracle against what the paper and mathematics fix.

Nothing here re-uses the oracle's code to compute an expectation: the checks
are hand-derived fixtures, closed forms, brute force over tiny inputs,
textbook routines (sorting, logsumexp, scaled-dot-product attention) and
invariants.  Each check is chosen so that a plausible mistake in the oracle
(a dropped term, a wrong sign or index, a transposed operand, a flipped tie
rule) fails at least one of them; ``test_pins_catch_planted_mistakes`` plants
such mistakes in oracle outputs and confirms the checkers flag them.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2608_00531_gb300 import workload as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _num(v):
    return float(v) if not isinstance(v, str) else float(v)


# ---------------------------------------------------------------- S1 pins
def test_score_hand_ties():
    g = _load("score_ties.json")
    for row in g["rows"]:
        x = np.array([_num(v) for v in row["x"]], dtype=np.float64)[None, :]
        ids, vals, margin, lse, logp1 = oracle.score_draft(x, g["k"])
        assert ids[0].tolist() == row["ids"]
        assert vals[0].tolist() == [_num(v) for v in row["vals"]]
        assert margin[0] == _num(row["margin"])


def test_lse_closed_forms():
    # all-equal row: lse = c + ln V, logp1 = -ln V
    for V, c in [(7, 0.0), (32000, 3.25), (151936, -11.5)]:
        x = np.full((1, V), c)
        _, _, m, lse, lp = oracle.score_draft(x, 2)
        assert m[0] == 0.0
        assert abs(lse[0] - (c + math.log(V))) < 1e-12 * max(1, abs(c) + math.log(V))
        assert abs(lp[0] + math.log(V)) < 1e-12 * math.log(V)
    # the hand-tie row: log(e^1 + 3 e^3 + e^2)
    x = np.array([[1, 3, 3, 2, -np.inf, 3]], dtype=np.float64)
    _, _, _, lse, lp = oracle.score_draft(x, 3)
    want = math.log(math.e + 3 * math.e ** 3 + math.e ** 2)
    assert abs(lse[0] - want) < 1e-13
    assert abs(lp[0] - (3 - want)) < 1e-13
    # a single finite entry: probability one
    x = np.array([[-np.inf, 7, -np.inf, -np.inf]])
    _, _, _, lse, lp = oracle.score_draft(x, 2)
    assert lse[0] == 7.0 and lp[0] == 0.0


@pytest.mark.parametrize("seed", range(6))
def test_score_bruteforce_and_textbook(seed):
    from scipy.special import logsumexp
    rng = np.random.default_rng(seed)
    V = int(rng.integers(2, 40))
    k = int(rng.integers(1, min(8, V) + 1))
    # few distinct values so ties are common
    x = rng.integers(-4, 5, size=(5, V)).astype(np.float64) * 0.5
    ids, vals, margin, lse, logp1 = oracle.score_draft(x, k)
    for r in range(5):
        ranked = sorted(range(V), key=lambda i: (-x[r, i], i))
        assert ids[r].tolist() == ranked[:k]
        assert vals[r].tolist() == [x[r, i] for i in ranked[:k]]
        s = math.fsum(math.exp(v) for v in x[r])
        assert abs(lse[r] - math.log(s)) < 1e-13 * max(1.0, abs(math.log(s)))
        assert abs(lse[r] - logsumexp(x[r])) < 1e-12
        if k >= 2:
            # Eq. (2): the logit gap equals the log-probability gap
            lp = x[r] - math.log(s)
            assert abs(margin[r] - (lp[ranked[0]] - lp[ranked[1]])) < 1e-12
        assert abs(logp1[r] - (x[r, ranked[0]] - math.log(s))) < 1e-12
    # np.argsort(kind="stable") on the negated values is the same ranking
    order = np.argsort(-x, axis=1, kind="stable")[:, :k]
    assert np.array_equal(order, ids)


def test_row_argmax_first_max():
    x = np.array([[0, 5, 5, 1], [-1, -1, -1, -1], [3, 2, 1, 3]], dtype=np.float64)
    assert oracle.row_argmax(x).tolist() == [1, 0, 0]
    rng = np.random.default_rng(3)
    x = rng.integers(0, 4, size=(50, 30)).astype(np.float64)
    want = [min(i for i in range(30) if x[r, i] == x[r].max()) for r in range(50)]
    assert oracle.row_argmax(x).tolist() == want


# ---------------------------------------------------------------- S2/S3 pins
def _tree_hand():
    g = _load("tree_hand.json")
    K = g["K"]
    top = np.array(g["top_ids"])[None]
    margin = np.array(g["margin"], dtype=np.float32)[None]
    t = oracle.build_tree(top, margin, np.array([g["root_tok"]]), np.array([g["cache_len"]]),
                          g["tau"], g["budget"], g["branches"], g["repair_depth"])
    return g, t


def test_tree_hand():
    g, t = _tree_hand()
    e = g["expect_tree"]
    n = e["n_nodes"]
    assert t["n_nodes"][0] == n
    for key in ("tok", "parent", "depth", "pos"):
        assert t[key][0, :n].tolist() == e[key], key
        assert (t[key][0, n:] == -1).all()
    assert [int(v) for v in t["anc"][0, :n, 0]] == e["anc"]
    assert t["ufp_pos"][0].tolist() == e["ufp_pos"]
    assert t["n_ufp"][0] == e["n_ufp"]


def ancestors_by_parent_walk(parent_row, j):
    s = set()
    while j >= 0 and j not in s:          # a cycle (a corrupt tree) ends the walk
        s.add(j)
        j = int(parent_row[j])
    return s


def check_tree(t, top_ids, margin, tau, budget, branches, depth_rep, cache_len, redraft=None):
    """Invariants of a built tree; returns a list of violations."""
    bad = []
    B, K, k = top_ids.shape
    for b in range(B):
        n = int(t["n_nodes"][b])
        if n > 1 + K + budget:
            bad.append(("budget", b))
        if t["parent"][b, 0] != -1 or t["depth"][b, 0] != 0:
            bad.append(("root", b))
        for i in range(1, K + 1):        # branch 0 is the draft chain
            if (t["tok"][b, i] != top_ids[b, i - 1, 0] or t["parent"][b, i] != i - 1
                    or t["depth"][b, i] != i):
                bad.append(("chain", b, i))
        for j in range(n):
            p = int(t["parent"][b, j])
            if j > 0 and not (0 <= p < j):
                bad.append(("parent-order", b, j))
            if j > 0 and t["depth"][b, j] != t["depth"][b, p] + 1:
                bad.append(("depth", b, j))
            if t["pos"][b, j] != cache_len[b] + t["depth"][b, j]:
                bad.append(("pos", b, j))
            if set(oracle.anc_set(t["anc"][b, j])) != ancestors_by_parent_walk(t["parent"][b], j):
                bad.append(("anc", b, j))
        for j in range(n, t["tok"].shape[1]):
            if t["tok"][b, j] != -1 or t["anc"][b, j].any():
                bad.append(("padding", b, j))
        # every repair node hangs under a gated position with a ranked alternative
        repair_pos = []
        for j in range(K + 1, n):
            p = int(t["parent"][b, j])
            if p <= K:                        # an alternative: child of chain node i
                i = p
                if not (np.float32(margin[b, i]) < np.float32(tau)):
                    bad.append(("gate", b, j))
                if int(t["tok"][b, j]) not in [int(v) for v in top_ids[b, i, 1:branches]]:
                    bad.append(("alt-token", b, j))
                repair_pos.append(i)
            else:                             # a successor of an alternative
                if depth_rep < 2:
                    bad.append(("depth1-successor", b, j))
                else:
                    i = int(t["parent"][b, p])
                    r = [int(v) for v in top_ids[b, i, :]].index(int(t["tok"][b, p])) + 1
                    if t["tok"][b, j] != redraft[b, i, r - 2]:
                        bad.append(("successor-token", b, j))
        # ascending-margin priority: an eligible position left without any
        # alternative never has a smaller (margin, position) than a taken one
        # whose alternatives could have been swapped for it
        eligible = [i for i in range(K) if np.float32(margin[b, i]) < np.float32(tau)]
        taken = set(repair_pos)
        for i in eligible:
            if i in taken:
                continue
            cost = min(depth_rep, K - i)
            if n - (1 + K) + cost <= budget:
                bad.append(("fits-but-skipped", b, i))
            for jpos in taken:
                if (np.float32(margin[b, jpos]), jpos) > (np.float32(margin[b, i]), i) and \
                        min(depth_rep, K - jpos) >= cost:
                    bad.append(("priority", b, i, jpos))
        if len(taken) != int(t["n_ufp"][b]) or set(t["ufp_pos"][b, :len(taken)].tolist()) != taken:
            bad.append(("ufp-list", b))
    return bad


def _random_case(seed, K=None, budget=None, branches=None, depth_rep=1, tau=None):
    rng = np.random.default_rng(seed)
    B = 3
    K = K or int(rng.integers(2, 12))
    k = 4
    branches = branches or int(rng.integers(2, 5))
    budget = int(rng.integers(0, 3 * K)) if budget is None else budget
    tau = float(rng.choice([0.0, 0.5, 1.0, 2.0])) if tau is None else tau
    # margins on a coarse grid so that ties happen
    margin = (rng.integers(0, 12, size=(B, K)) * 0.25).astype(np.float32)
    top = np.stack([rng.permutation(1000)[:k] for _ in range(B * K)]).reshape(B, K, k)
    root = rng.integers(0, 1000, size=B)
    L = rng.integers(10, 50, size=B)
    redraft = rng.integers(0, 1000, size=(B, K, max(1, branches - 1)))
    return top, margin, root, L, tau, budget, branches, depth_rep, redraft


@pytest.mark.parametrize("seed", range(40))
def test_tree_invariants(seed):
    depth_rep = 2 if seed % 3 == 0 else 1
    top, margin, root, L, tau, budget, branches, d, redraft = _random_case(seed, depth_rep=depth_rep)
    t = oracle.build_tree(top, margin, root, L, tau, budget, branches, d, redraft)
    assert check_tree(t, top, margin, tau, budget, branches, d, L, redraft) == []


def test_tree_special_cases():
    top, margin, root, L, _, _, branches, _, redraft = _random_case(7, K=8, branches=3)
    K = 8
    # tau <= 0: margins are >= 0, so no position is gated: the tree is branch 0
    t = oracle.build_tree(top, margin, root, L, 0.0, 20, branches, 1, redraft)
    assert (t["n_nodes"] == K + 1).all() and (t["n_ufp"] == 0).all()
    # budget 0: branch 0 only, whatever the gate says
    t = oracle.build_tree(top, margin, root, L, 100.0, 0, branches, 1, redraft)
    assert (t["n_nodes"] == K + 1).all()
    # a budget that covers everything admits every gated position, every rank
    for d in (1, 2):
        t = oracle.build_tree(top, margin, root, L, 1.0, K * (branches - 1) * d, branches, d, redraft)
        for b in range(3):
            eligible = [i for i in range(K) if margin[b, i] < 1.0]
            want = sum((branches - 1) * min(d, K - i) for i in eligible)
            assert t["n_nodes"][b] == 1 + K + want
    # a margin exactly at tau is not a UFP (strict gate)
    m = np.full((1, 4), 1.0, dtype=np.float32)
    t = oracle.build_tree(top[:1, :4], m, root[:1], L[:1], 1.0, 8, 2, 1, None)
    assert t["n_nodes"][0] == 5
    m[0, 2] = np.nextafter(np.float32(1.0), np.float32(0.0))
    t = oracle.build_tree(top[:1, :4], m, root[:1], L[:1], 1.0, 8, 2, 1, None)
    assert t["n_nodes"][0] == 6 and t["ufp_pos"][0, 0] == 2


def test_tree_depth2_last_position_costs_one():
    # Depth-2 repairs: the last position has no successor, so it costs one node
    # and can still fit when the remaining budget is odd.
    K = 4
    top = np.array([[[10, 20], [11, 21], [12, 22], [13, 23]]])
    margin = np.array([[0.1, 5, 5, 0.2]], dtype=np.float32)
    redraft = np.array([[[50], [51], [52], [-1]]])
    t = oracle.build_tree(top, margin, np.array([1]), np.array([30]), 1.0, 3, 2, 2, redraft)
    assert t["n_nodes"][0] == 1 + K + 3
    assert t["tok"][0, 5:8].tolist() == [20, 50, 23]
    assert t["parent"][0, 5:8].tolist() == [0, 5, 3]
    assert t["depth"][0, 5:8].tolist() == [1, 2, 4]


# ------------------------------------------------- Eq. (3) branch budget pins
def test_branch_budget_closed_forms():
    """Eq. (3) by hand at the paper's (b_min, b_max) = (1, 5).

    With s = 8 every quotient m / s, every u = 1 - m / s and every
    x = 1 + 4u below is exact in float32, so the expected b is the rounded
    hand value; x = 1.5, 2.5, 3.5 and 4.5 pin the halves (away from zero:
    half to even would give 2, 2, 4, 4).
    """
    assert _branch_budget_closed_forms_hold(oracle.branch_budget)


def _branch_budget_closed_forms_hold(bb):
    cases = [(0.0, 5),    # u = 1: a tied position gets b_max
             (2.0, 4),    # u = 3/4: x = 4
             (3.0, 4),    # u = 5/8: x = 3.5
             (4.0, 3),    # u = 1/2: x = 3
             (5.0, 3),    # u = 3/8: x = 2.5
             (6.0, 2),    # u = 1/4: x = 2
             (7.0, 2),    # u = 1/8: x = 1.5
             (1.0, 5),    # u = 7/8: x = 4.5
             (8.0, 1),    # u = 0: b_min
             (12.0, 1)]   # m > s: u clipped to 0
    ok = all(bb(np.float32(m), 8.0, 1, 5) == want for m, want in cases)
    ok = ok and all(bb(np.float32(m), 1.0, 3, 3) == 3 for m in (0.0, 0.3, 7.9, 100.0))  # b_min = b_max
    ok = ok and bb(np.float32(1.0), 1.0, 0, 4) == 0 and bb(np.float32(0.0), 1.0, 0, 4) == 4
    ok = ok and bb(np.float32(np.inf), 1.0, 1, 5) == 1   # rival at -inf: margin +inf
    return ok


@pytest.mark.parametrize("seed", range(6))
def test_branch_budget_bounded_monotone_nearest(seed):
    rng = np.random.default_rng(seed)
    s = float(rng.choice([0.25, 0.8, 1.0, 2.5]))
    b_min = int(rng.integers(0, 3))
    b_max = b_min + int(rng.integers(0, 5))
    ms = np.sort(rng.uniform(0.0, 2.0 * s, 400).astype(np.float32))
    bs = [oracle.branch_budget(m, s, b_min, b_max) for m in ms]
    assert all(b_min <= b <= b_max for b in bs)
    assert all(x >= y for x, y in zip(bs, bs[1:]))      # more margin, fewer branches
    for m, b in zip(ms, bs):                             # the nearest integer (exact arithmetic)
        x = b_min + max(0.0, 1.0 - float(m) / s) * (b_max - b_min)
        assert abs(b - x) <= 0.5 + 1e-5, (m, b, x)


def _tree_dynamic_hand(budget):
    K = 4
    top = np.array([[[10 * i + r for r in range(6)] for i in range(K)]])
    margin = np.array([[0.0, 0.5, 2.0, 0.75]], dtype=np.float32)
    return oracle.build_tree(top, margin, np.array([7]), np.array([40]), 1.0, budget, 6, 1,
                             margin_scale=1.0, branch_min=1)


def test_tree_dynamic_budget_hand():
    # tau = 1, s = 1, (b_min, b_max) = (1, 5): position 0 (m = 0) gets 5
    # alternatives, position 1 (m = 0.5, x = 3) 3, position 3 (m = 0.75, x = 2)
    # 2; position 2 (m = 2) is no UFP.  Nodes in (position, rank) order.
    t = _tree_dynamic_hand(20)
    assert t["n_nodes"][0] == 1 + 4 + 10
    assert t["tok"][0, 5:15].tolist() == [1, 2, 3, 4, 5, 11, 12, 13, 31, 32]
    assert t["parent"][0, 5:15].tolist() == [0] * 5 + [1] * 3 + [3] * 2
    assert t["depth"][0, 5:15].tolist() == [1] * 5 + [2] * 3 + [4] * 2
    assert t["ufp_pos"][0].tolist() == [0, 1, 3, -1] and t["n_ufp"][0] == 3
    # budget 6: ascending margin admits position 0's five, then one of
    # position 1's; position 3 no longer fits
    t = _tree_dynamic_hand(6)
    assert t["n_nodes"][0] == 1 + 4 + 6
    assert t["tok"][0, 5:11].tolist() == [1, 2, 3, 4, 5, 11]
    assert t["ufp_pos"][0].tolist() == [0, 1, -1, -1] and t["n_ufp"][0] == 2


@pytest.mark.parametrize("seed", range(12))
def test_tree_dynamic_budget_special_cases(seed):
    top, margin, root, L, tau, budget, branches, d, redraft = _random_case(
        seed, depth_rep=2 if seed % 2 else 1)
    fixed = oracle.build_tree(top, margin, root, L, tau, budget, branches, d, redraft)
    # b_min = b_max = branches - 1: every UFP keeps the fixed budget's alternatives
    same = oracle.build_tree(top, margin, root, L, tau, budget, branches, d, redraft,
                             margin_scale=float(1 + seed % 3), branch_min=branches - 1)
    for key in fixed:
        assert np.array_equal(fixed[key], same[key]), key
    # m_i >= s for every position: Eq. (3) gives b_min everywhere (here 1)
    one = oracle.build_tree(top, margin, root, L, tau, budget, branches, d, redraft,
                            margin_scale=1e-6, branch_min=1)
    ref1 = oracle.build_tree(top, margin, root, L, tau, budget, 2, d, redraft)
    for b in range(top.shape[0]):
        if (margin[b] > 0).all():
            for key in ("n_nodes", "tok", "parent", "depth"):
                assert np.array_equal(one[key][b], ref1[key][b]), key
    # every tree with a dynamic budget keeps the invariants of a repair tree
    dyn = oracle.build_tree(top, margin, root, L, tau, budget, branches, d, redraft,
                            margin_scale=1.5, branch_min=1)
    assert check_tree(dyn, top, margin, tau, budget, branches, d, L, redraft) == []


# --------------------------------------- structural caps (depth, beam) pins
def _caps_hand(**kw):
    K = 4
    top = np.array([[[100 * i + r for r in range(3)] for i in range(K)]])
    margin = np.full((1, K), 0.1, dtype=np.float32)       # every position a UFP, ties by position
    redraft = np.array([[[900 + 10 * i + a for a in range(2)] for i in range(K)]])
    d = kw.pop("d", 1)
    return oracle.build_tree(top, margin, np.array([5]), np.array([60]), 1.0, 40, 3, d, redraft, **kw)


def test_tree_caps_hand():
    # no caps: two alternatives at each of the four positions
    assert _caps_hand()["n_nodes"][0] == 5 + 8
    # beam 1: the chain fills every depth, so nothing is added
    t = _caps_hand(beam=1)
    assert t["n_nodes"][0] == 5 and t["n_ufp"][0] == 0
    # beam 2: one alternative per depth, the rank-2 one (ranks are tried in order)
    t = _caps_hand(beam=2)
    assert t["n_nodes"][0] == 5 + 4
    assert t["tok"][0, 5:9].tolist() == [1, 101, 201, 301]
    # beam 3: everything fits again
    assert _caps_hand(beam=3)["n_nodes"][0] == 5 + 8
    # maximum depth 2: alternatives only at positions 0 and 1 (depths 1 and 2)
    t = _caps_hand(max_depth=2)
    assert t["n_nodes"][0] == 5 + 4
    assert t["parent"][0, 5:9].tolist() == [0, 0, 1, 1]
    assert t["ufp_pos"][0].tolist() == [0, 1, -1, -1]
    # depth-2 repairs under maximum depth 2: position 0 keeps its successors
    # (depths 1, 2); position 1's successors (depth 3) are dropped
    t = _caps_hand(d=2, max_depth=2)
    assert t["n_nodes"][0] == 5 + 6
    assert t["tok"][0, 5:11].tolist() == [1, 900, 2, 901, 101, 102]
    assert t["parent"][0, 5:11].tolist() == [0, 5, 0, 7, 1, 1]
    assert t["depth"][0, 5:11].tolist() == [1, 2, 1, 2, 2, 2]
    # depth-2 repairs under beam 2: position 0's first alternative and its
    # successor take depths 1 and 2, so position 1 (depth 2) finds no room;
    # position 2 fits (depths 3, 4); position 3 (depth 4) does not
    t = _caps_hand(d=2, beam=2)
    assert t["tok"][0, 5:].tolist()[:4] == [1, 900, 201, 920]
    assert t["n_nodes"][0] == 5 + 4
    assert t["ufp_pos"][0].tolist() == [0, 2, -1, -1]


@pytest.mark.parametrize("seed", range(16))
def test_tree_caps_invariants_and_no_op_values(seed):
    depth_rep = 2 if seed % 2 else 1
    top, margin, root, L, tau, budget, branches, d, redraft = _random_case(seed, depth_rep=depth_rep)
    K = top.shape[1]
    base = oracle.build_tree(top, margin, root, L, tau, budget, branches, d, redraft)
    # caps that cannot bind change nothing
    wide = oracle.build_tree(top, margin, root, L, tau, budget, branches, d, redraft,
                             max_depth=K, beam=1 + 2 * branches)
    for key in base:
        assert np.array_equal(base[key], wide[key]), key
    # binding caps: no repair node past the maximum depth, no depth wider
    # than the beam, branch 0 intact
    rng = np.random.default_rng(seed)
    md, bw = int(rng.integers(1, K + 1)), int(rng.integers(1, 4))
    t = oracle.build_tree(top, margin, root, L, tau, budget, branches, d, redraft, max_depth=md, beam=bw)
    for b in range(top.shape[0]):
        n = int(t["n_nodes"][b])
        dep = t["depth"][b, :n]
        assert (dep[1 + K:] <= md).all()
        assert np.bincount(dep, minlength=K + 2).max() <= max(bw, 1)
        assert t["tok"][b, 1:K + 1].tolist() == top[b, :, 0].tolist()
        assert n <= 1 + K + budget


# ---------------------------------------------------------------- S4 pins
def _attn_case(seed, paged=False):
    rng = np.random.default_rng(seed)
    B, K, Hkv, G, D = 2, 4, 2, 3, 16
    Hq = Hkv * G
    top, margin, root, _, _, _, _, _, redraft = _random_case(seed, K=K, branches=3, budget=4, tau=1.0)
    top, margin, root = top[:B], margin[:B], root[:B]
    L = rng.integers(5, 40, size=B)
    t = oracle.build_tree(top, margin, root, L, 1.0, 4, 3, 1)
    N = 1 + K + 4
    q = rng.standard_normal((B, N, Hq, D))
    tk = rng.standard_normal((B, N, Hkv, D))
    tv = rng.standard_normal((B, N, Hkv, D))
    Lmax = int(L.max())
    kc = rng.standard_normal((B, Lmax, Hkv, D))
    vc = rng.standard_normal((B, Lmax, Hkv, D))
    return q, tk, tv, kc, vc, L, t, D


@pytest.mark.parametrize("seed", range(4))
def test_tree_attn_equals_per_path_causal_sdpa(seed):
    """Sec. 3.4: one tree pass equals separate causal attention per path."""
    q, tk, tv, kc, vc, L, t, D = _attn_case(seed)
    scale = 1.0 / math.sqrt(D)
    out = oracle.tree_attn(q, tk, tv, kc, vc, L, t["n_nodes"], t["anc"], scale)
    B, N, Hq, _ = q.shape
    Hkv = tk.shape[2]
    G = Hq // Hkv
    for b in range(B):
        for j in range(int(t["n_nodes"][b])):
            # the path root..j as an explicit token sequence after the cache
            path = []
            x = j
            while x >= 0:
                path.append(x)
                x = int(t["parent"][b, x])
            path = path[::-1]
            for h in range(Hq):
                hk = h // G
                ks = np.concatenate([kc[b, :L[b], hk], tk[b, path, hk]])
                vs = np.concatenate([vc[b, :L[b], hk], tv[b, path, hk]])
                # causal attention of the whole sequence; the last row is node j
                Tq = torch.from_numpy(np.concatenate([np.zeros((len(ks) - 1, D)), q[b, j, h][None]]))
                o = torch.nn.functional.scaled_dot_product_attention(
                    Tq[None, None], torch.from_numpy(ks)[None, None], torch.from_numpy(vs)[None, None],
                    is_causal=True, scale=scale)[0, 0, -1].numpy()
                assert np.allclose(out[b, j, h], o, rtol=1e-11, atol=1e-12)


def _in_place_caches(kc, vc, tk, tv, L, n, paged, ps=4):
    """Caches holding each sequence's cache rows at slots 0..L_b-1 and its
    tree rows at slots L_b + j (the in-place layout); paged through a
    shuffled block table when asked."""
    B, _, Hkv, D = kc.shape
    cap = int(max(L[b] + n[b] for b in range(B)))
    ck = np.zeros((B, cap, Hkv, D))
    cv = np.zeros((B, cap, Hkv, D))
    for b in range(B):
        ck[b, :L[b]], cv[b, :L[b]] = kc[b, :L[b]], vc[b, :L[b]]
        ck[b, L[b]:L[b] + n[b]], cv[b, L[b]:L[b] + n[b]] = tk[b, :n[b]], tv[b, :n[b]]
    if not paged:
        return ck, cv, None
    per = (cap + ps - 1) // ps
    table = np.random.default_rng(5).permutation(B * per).reshape(B, per)
    pk = np.zeros((B * per, ps, Hkv, D))
    pv = np.zeros((B * per, ps, Hkv, D))
    for b in range(B):
        for sl in range(cap):
            pk[table[b, sl // ps], sl % ps] = ck[b, sl]
            pv[table[b, sl // ps], sl % ps] = cv[b, sl]
    return pk, pv, table


@pytest.mark.parametrize("paged", [False, True])
@pytest.mark.parametrize("seed", range(3))
def test_tree_attn_in_place_equals_per_path_causal_sdpa(seed, paged):
    """The in-place layout (tree rows at cache slots L_b + j): the same
    attention as per-path causal SDPA over the explicit path."""
    q, tk, tv, kc, vc, L, t, D = _attn_case(seed)
    n = t["n_nodes"]
    ck, cv, table = _in_place_caches(kc, vc, tk, tv, L, n, paged)
    scale = 1.0 / math.sqrt(D)
    out = oracle.tree_attn(q, None, None, ck, cv, L, n, t["anc"], scale, block_table=table, page_size=4)
    B, N, Hq, _ = q.shape
    G = Hq // tk.shape[2]
    for b in range(B):
        for j in range(int(n[b])):
            path = []
            x = j
            while x >= 0:
                path.append(x)
                x = int(t["parent"][b, x])
            path = path[::-1]
            for h in range(Hq):
                hk = h // G
                ks = np.concatenate([kc[b, :L[b], hk], tk[b, path, hk]])
                vs = np.concatenate([vc[b, :L[b], hk], tv[b, path, hk]])
                Tq = torch.from_numpy(np.concatenate([np.zeros((len(ks) - 1, D)), q[b, j, h][None]]))
                o = torch.nn.functional.scaled_dot_product_attention(
                    Tq[None, None], torch.from_numpy(ks)[None, None], torch.from_numpy(vs)[None, None],
                    is_causal=True, scale=scale)[0, 0, -1].numpy()
                assert np.allclose(out[b, j, h], o, rtol=1e-11, atol=1e-12)


def test_tree_attn_constant_keys_give_mean_of_values():
    q, tk, tv, kc, vc, L, t, D = _attn_case(11)
    kc[:] = 0.3
    tk[:] = 0.3
    out = oracle.tree_attn(q, tk, tv, kc, vc, L, t["n_nodes"], t["anc"], 0.25)
    G = q.shape[2] // tk.shape[2]
    for b in range(q.shape[0]):
        for j in range(int(t["n_nodes"][b])):
            vis = ancestors_by_parent_walk(t["parent"][b], j)
            for h in range(q.shape[2]):
                rows = [vc[b, i, h // G] for i in range(L[b])] + [tv[b, i, h // G] for i in sorted(vis)]
                assert np.allclose(out[b, j, h], np.mean(rows, axis=0), rtol=1e-12, atol=1e-12)


def test_tree_attn_paged_equals_contiguous():
    q, tk, tv, kc, vc, L, t, D = _attn_case(5)
    B, Lmax, Hkv, _ = kc.shape
    ps = 4
    npg = (Lmax + ps - 1) // ps
    rng = np.random.default_rng(0)
    perm = rng.permutation(B * npg)
    table = perm.reshape(B, npg)
    kp = np.zeros((B * npg, ps, Hkv, D))
    vp = np.zeros((B * npg, ps, Hkv, D))
    for b in range(B):
        for s in range(Lmax):
            kp[table[b, s // ps], s % ps] = kc[b, s]
            vp[table[b, s // ps], s % ps] = vc[b, s]
    a = oracle.tree_attn(q, tk, tv, kc, vc, L, t["n_nodes"], t["anc"], 0.25)
    p = oracle.tree_attn(q, tk, tv, kp, vp, L, t["n_nodes"], t["anc"], 0.25, table, ps)
    assert np.array_equal(a, p)


# ---------------------------------------------------------------- S5 pins
def _hand_accept(case):
    g, t = _tree_hand()
    c = g[case]
    targ = np.array(c["targ"])[None]
    r = oracle.accept(targ, t["n_nodes"], t["tok"], t["parent"], t["depth"], t["anc"], g["K"])
    return g, t, c, r


@pytest.mark.parametrize("case", ["repair_win", "branch0_win"])
def test_accept_hand(case):
    g, t, c, r = _hand_accept(case)
    for key in ("accept_len", "best_node", "diverge_depth"):
        assert int(r[key][0]) == c[key], key
    assert r["path_nodes"][0].tolist() == c["path_nodes"]
    assert r["out_tokens"][0].tolist() == c["out_tokens"]


def brute_force_accept(targ, n, tok, parent, depth):
    """a(pi) for every root-to-leaf path, the maximum, and its first best leaf."""
    children = {j: [] for j in range(n)}
    for j in range(1, n):
        children[int(parent[j])].append(j)
    leaves = [j for j in range(n) if not children[j]]
    best_a, best_nodes = -1, None
    for leaf in leaves:
        path = []
        x = leaf
        while x >= 0:
            path.append(x)
            x = int(parent[x])
        path = path[::-1]
        a = 0
        for t in range(1, len(path)):
            if tok[path[t]] == targ[path[t - 1]]:
                a = t
            else:
                break
        if a > best_a:
            best_a = a
    return best_a


@pytest.mark.parametrize("seed", range(30))
def test_accept_bruteforce_all_paths(seed):
    top, margin, root, L, tau, budget, branches, d, redraft = _random_case(
        seed, depth_rep=2 if seed % 2 else 1)
    # a tiny token alphabet so that many nodes verify
    top = top % 5
    redraft = redraft % 5
    for b in range(top.shape[0]):
        for i in range(top.shape[1]):
            top[b, i] = np.array([0, 1, 2, 3])   # distinct ranked ids per position
    t = oracle.build_tree(top, margin, root, L, tau, budget, branches, d, redraft)
    rng = np.random.default_rng(seed + 99)
    targ = rng.integers(0, 3, size=t["tok"].shape)
    r = oracle.accept(targ, t["n_nodes"], t["tok"], t["parent"], t["depth"], t["anc"], top.shape[1])
    for b in range(top.shape[0]):
        n = int(t["n_nodes"][b])
        a = brute_force_accept(targ[b], n, t["tok"][b], t["parent"][b], t["depth"][b])
        assert r["accept_len"][b] == a
        best = int(r["best_node"][b])
        assert t["depth"][b, best] == a
        # best is the lowest-index node at depth a whose path verifies
        path = r["path_nodes"][b, :a + 1].tolist()
        assert path[0] == 0 and path[-1] == best
        for s in range(1, a + 1):
            assert t["parent"][b, path[s]] == path[s - 1]
            assert t["tok"][b, path[s]] == targ[b, path[s - 1]]
        assert r["out_tokens"][b, :a + 1].tolist() == [int(t["tok"][b, x]) for x in path[1:]] + [int(targ[b, best])]
        off = [s for s in range(a + 1) if path[s] > top.shape[1]]
        assert r["diverge_depth"][b] == (off[0] if off else -1)


@pytest.mark.parametrize("seed", range(10))
def test_budget_zero_is_prefix_verification(seed):
    """R = 0 leaves branch 0 alone: the result is plain prefix verification."""
    w = W.WORKLOADS["tiny"].replace(vocab=64, budget=0, top_level=3.0)
    d = W.draft_block(w, seed=seed)
    x = W.bf16_to_f64(d.logits).reshape(-1, w.vocab)
    ids, _, margin, _, _ = oracle.score_draft(x, w.topk)
    K = w.block
    t = oracle.build_tree(ids.reshape(1, K, -1), margin.astype(np.float32).reshape(1, K), d.root_tok,
                          np.array([100]), w.tau, 0, w.branches, 1)
    rng = np.random.default_rng(seed)
    # the target agrees with the draft on a random prefix
    e = int(rng.integers(0, K + 1))
    targ = np.full((1, K + 1), -5)
    targ[0, :e] = ids.reshape(K, -1)[:e, 0]
    r = oracle.accept(targ, t["n_nodes"], t["tok"], t["parent"], t["depth"], t["anc"], K)
    # plain prefix verification written out: count leading draft tokens that
    # equal the target's token at the previous position
    draft = ids.reshape(K, -1)[:, 0]
    a = 0
    while a < K and draft[a] == targ[0, a]:
        a += 1
    assert r["accept_len"][0] == a == e
    assert r["diverge_depth"][0] == -1
    assert r["out_tokens"][0, :a + 1].tolist() == list(draft[:a]) + [int(targ[0, a])]


# ---------------------------------------------------------------- S6 pins
@pytest.mark.parametrize("case", ["repair_win", "branch0_win"])
def test_resync_hand(case):
    g, t, c, r = _hand_accept(case)
    rng = np.random.default_rng(1)
    N, Hkv, D, layers = 8, 2, 4, 3
    tk = rng.standard_normal((layers, 1, N, Hkv, D))
    tv = rng.standard_normal((layers, 1, N, Hkv, D))
    kc = [rng.standard_normal((1, 120, Hkv, D)) for _ in range(layers)]
    vc = [rng.standard_normal((1, 120, Hkv, D)) for _ in range(layers)]
    k0 = [x.copy() for x in kc]
    v0 = [x.copy() for x in vc]
    s = oracle.resync(kc, vc, tk, tv, r["path_nodes"], r["accept_len"], r["diverge_depth"],
                      r["out_tokens"], np.array([g["cache_len"]]), g["K"])
    assert s["cache_len"][0] == c["cache_len"]
    assert s["draft_valid_len"][0] == c["draft_valid_len"]
    assert s["replay_tokens"][0].tolist() == c["replay_tokens"]
    assert s["n_replay"][0] == c["n_replay"]
    L, a = g["cache_len"], c["accept_len"]
    for l in range(layers):
        assert np.array_equal(kc[l][0, :L], k0[l][0, :L])            # older rows untouched
        assert np.array_equal(kc[l][0, L + a + 1:], k0[l][0, L + a + 1:])
        for tdep, node in enumerate(c["path_nodes"][:a + 1]):
            assert np.array_equal(kc[l][0, L + tdep], tk[l, 0, node])
            assert np.array_equal(vc[l][0, L + tdep], tv[l, 0, node])


def test_resync_paged_matches_contiguous():
    g, t, c, r = _hand_accept("repair_win")
    rng = np.random.default_rng(2)
    N, Hkv, D, ps = 8, 2, 4, 16
    tk = rng.standard_normal((2, 1, N, Hkv, D))
    tv = rng.standard_normal((2, 1, N, Hkv, D))
    cont_k = [np.zeros((1, 128, Hkv, D)) for _ in range(2)]
    cont_v = [np.zeros((1, 128, Hkv, D)) for _ in range(2)]
    table = np.array([[5, 3, 7, 0, 6, 1, 2, 4]])
    pag_k = [np.zeros((8, ps, Hkv, D)) for _ in range(2)]
    pag_v = [np.zeros((8, ps, Hkv, D)) for _ in range(2)]
    args = (tk, tv, r["path_nodes"], r["accept_len"], r["diverge_depth"], r["out_tokens"],
            np.array([g["cache_len"]]), g["K"])
    oracle.resync(cont_k, cont_v, *args)
    oracle.resync(pag_k, pag_v, *args, block_table=table, page_size=ps)
    for l in range(2):
        for s in range(128):
            assert np.array_equal(cont_k[l][0, s], pag_k[l][table[0, s // ps], s % ps])
            assert np.array_equal(cont_v[l][0, s], pag_v[l][table[0, s // ps], s % ps])


@pytest.mark.parametrize("case", ["repair_win", "branch0_win"])
def test_resync_in_place_hand(case):
    """In-place resync: the path rows come from cache slots L + node.  The
    result at slots L..L+a is the path's rows by depth; rows of chain nodes
    are already in place, so only the repair nodes' rows change slots."""
    g, t, c, r = _hand_accept(case)
    L, K = g["cache_len"], g["K"]
    n = int(t["n_nodes"][0])
    rng = np.random.default_rng(3)
    Hkv, D = 2, 4
    ck = [rng.standard_normal((1, L + n + 4, Hkv, D)) for _ in range(2)]
    cv = [rng.standard_normal((1, L + n + 4, Hkv, D)) for _ in range(2)]
    before_k = [x.copy() for x in ck]
    oracle.resync(ck, cv, None, None, r["path_nodes"], r["accept_len"], r["diverge_depth"],
                  r["out_tokens"], np.array([L]), K)
    a = int(r["accept_len"][0])
    path = [int(x) for x in r["path_nodes"][0, :a + 1]]
    for l in range(2):
        for d, node in enumerate(path):
            assert np.array_equal(ck[l][0, L + d], before_k[l][0, L + node])
        assert np.array_equal(ck[l][0, :L], before_k[l][0, :L])   # the old cache is untouched
        moved = [d for d, node in enumerate(path) if node != d]
        assert all(node > K for d, node in enumerate(path) if node != d)
        if case == "branch0_win":
            assert moved == [] and np.array_equal(ck[l], before_k[l])


# ------------------------------------------- stochastic verification pins
def test_sample_target_closed_forms():
    """Inverse-CDF sampling by hand: equal logits give floor(u V); two finite
    logits a, b give the first id while u < e^(a/T) / (e^(a/T) + e^(b/T))."""
    assert _sample_closed_forms_hold(oracle.sample_target)


def _sample_closed_forms_hold(sample):
    V = 10
    x = np.zeros((1, 1, V))
    ok = True
    for u in (0.0, 0.05, 0.31, 0.5, 0.99):
        ok = ok and sample(x, np.array([1]), np.array([[u]]), 1.0)[0, 0] == math.floor(u * V)
    x = np.full((1, 1, V), -np.inf)
    x[0, 0, 3], x[0, 0, 7] = 1.0, 2.0
    for T in (0.5, 1.0, 3.0):
        p3 = math.exp(1.0 / T) / (math.exp(1.0 / T) + math.exp(2.0 / T))
        for u in (0.0, p3 - 1e-9, p3 + 1e-9, 0.999):
            ok = ok and sample(x, np.array([1]), np.array([[u]]), T)[0, 0] == (3 if u < p3 else 7)
    # one finite logit: always that id; only -inf: id 0; rows past n_nodes: -1
    x = np.full((1, 3, V), -np.inf)
    x[0, 0, 6] = -4.0
    y = sample(x, np.array([2]), np.array([[0.7, 0.2, 0.5]]), 1.0)
    return bool(ok and y[0].tolist() == [6, 0, -1])


@pytest.mark.parametrize("seed", range(4))
def test_sample_target_frequencies_follow_softmax(seed):
    """Over a fine grid of u, each id is drawn a share of the grid equal to
    its softmax probability at T (to one grid step), and the draw never
    decreases as u grows."""
    rng = np.random.default_rng(seed)
    V, M = 7, 20000
    T = float(rng.choice([0.5, 1.0, 2.0]))
    x = rng.standard_normal(V) * 2.0
    us = (np.arange(M) + 0.5) / M
    logits = np.broadcast_to(x, (1, M, V))
    y = oracle.sample_target(logits, np.array([M]), us[None], T)[0]
    assert (np.diff(y) >= 0).all()
    want = np.exp(x / T - (x / T).max())
    want /= want.sum()
    got = np.bincount(y, minlength=V) / M
    assert np.abs(got - want).max() <= 1.0 / M + 1e-12


# ---------------------------------------------------------------- pin power
def test_new_pins_catch_planted_mistakes():
    """Mutants of Eq. (3) and of the inverse-CDF sampler, each a plausible
    slip; the closed-form checkers must reject every one."""
    f = np.float32

    def bb_half_even(m, s, lo, hi):          # round() half to even
        u = f(min(max(f(f(1) - f(f(m) / f(s))), f(0)), f(1)))
        x = f(f(lo) + f(u * f(hi - lo)))
        return int(min(max(int(np.rint(x)), lo), hi))

    def bb_swapped(m, s, lo, hi):            # b_min and b_max exchanged
        return oracle.branch_budget(m, s, hi, lo) if hi >= lo else lo

    def bb_no_complement(m, s, lo, hi):      # u = m / s instead of 1 - m / s
        u = f(min(max(f(f(m) / f(s)), f(0)), f(1)))
        x = f(f(lo) + f(u * f(hi - lo)))
        return int(min(max(math.floor(float(x) + 0.5), lo), hi))

    def bb_branches_not_alternatives(m, s, lo, hi):   # b_i counting the draft token too
        return max(lo, oracle.branch_budget(m, s, lo, hi) - 1)

    assert _branch_budget_closed_forms_hold(oracle.branch_budget)
    for mutant in (bb_half_even, bb_swapped, bb_no_complement, bb_branches_not_alternatives):
        assert not _branch_budget_closed_forms_hold(mutant), mutant.__name__

    def sample_left(logits, n_nodes, uniforms, T):     # first id with cumulative >= r
        out = np.full(logits.shape[:2], -1, dtype=np.int64)
        for b in range(logits.shape[0]):
            for j in range(int(n_nodes[b])):
                x = logits[b, j]
                if x.max() == -np.inf:
                    out[b, j] = 0
                    continue
                c = np.cumsum(np.exp((x - x.max()) / T))
                out[b, j] = int(np.searchsorted(c, uniforms[b, j] * c[-1], side="left"))
        return out

    def sample_times_T(logits, n_nodes, uniforms, T):  # logits scaled by T, not by 1/T
        return oracle.sample_target(logits, n_nodes, uniforms, 1.0 / T)

    def sample_no_mask(logits, n_nodes, uniforms, T):  # -inf rows not special-cased, tail not -1
        y = oracle.sample_target(np.where(np.isinf(logits), -30.0, logits), np.full_like(n_nodes, logits.shape[1]),
                                 uniforms, T)
        return y

    assert _sample_closed_forms_hold(oracle.sample_target)
    for mutant in (sample_left, sample_times_T, sample_no_mask):
        assert not _sample_closed_forms_hold(mutant), mutant.__name__


def test_cap_and_in_place_pins_catch_planted_mistakes(monkeypatch):
    """A depth cap that drops the whole alternative (not only its successor)
    and an in-place layout read one slot late must fail their pins."""
    import oracle.cure_oracle as oc
    real_cost = oc.repair_cost

    def cost_drops_alternative(i, K, repair_depth, max_depth=0):
        c = min(repair_depth, K - i)
        return 0 if (max_depth > 0 and i + c > max_depth) else c

    monkeypatch.setattr(oc, "repair_cost", cost_drops_alternative)
    t = _caps_hand(d=2, max_depth=2)
    assert t["n_nodes"][0] != 5 + 6            # the hand pin expects six repair nodes
    monkeypatch.setattr(oc, "repair_cost", real_cost)
    assert _caps_hand(d=2, max_depth=2)["n_nodes"][0] == 5 + 6

    real_rows = oc.tree_rows_in_cache

    def rows_one_late(cache, cache_len, n_nodes, N, block_table, page_size):
        return real_rows(cache, np.asarray(cache_len) + 1, n_nodes, N, block_table, page_size)

    q, tk, tv, kc, vc, L, t, D = _attn_case(0)
    ck, cv, _ = _in_place_caches(kc, vc, tk, tv, L, t["n_nodes"], False)
    ck = np.concatenate([ck, np.zeros_like(ck[:, :1])], axis=1)   # room for the late read
    cv = np.concatenate([cv, np.zeros_like(cv[:, :1])], axis=1)
    good = oracle.tree_attn(q, None, None, ck, cv, L, t["n_nodes"], t["anc"], 1.0 / math.sqrt(D))
    sep = oracle.tree_attn(q, tk, tv, kc, vc, L, t["n_nodes"], t["anc"], 1.0 / math.sqrt(D))
    monkeypatch.setattr(oc, "tree_rows_in_cache", rows_one_late)
    bad = oracle.tree_attn(q, None, None, ck, cv, L, t["n_nodes"], t["anc"], 1.0 / math.sqrt(D))
    assert np.allclose(good, sep, rtol=1e-12, atol=1e-13)
    assert not np.allclose(bad, sep, rtol=1e-6, atol=1e-6)


def test_pins_catch_planted_mistakes():
    """Plant typical mistakes in oracle outputs; the checkers must object."""
    top, margin, root, L, tau, budget, branches, d, redraft = _random_case(4, K=8, budget=5, tau=2.0,
                                                                            branches=3)
    t = oracle.build_tree(top, margin, root, L, tau, budget, branches, d, redraft)
    assert check_tree(t, top, margin, tau, budget, branches, d, L, redraft) == []
    mutants = []
    m = {k: v.copy() for k, v in t.items()}
    m["parent"][0, 5] = m["parent"][0, 5] + 1         # wrong parent index
    mutants.append(m)
    m = {k: v.copy() for k, v in t.items()}
    m["anc"][0, 3, 0] ^= np.uint64(1 << 1)             # dropped ancestor bit
    mutants.append(m)
    m = {k: v.copy() for k, v in t.items()}
    m["tok"][0, 2] = top[0, 1, 1]                      # chain takes the rank-2 token
    mutants.append(m)
    m = {k: v.copy() for k, v in t.items()}
    m["pos"][0, 4] += 1                                # off-by-one position
    mutants.append(m)
    for mt in mutants:
        assert check_tree(mt, top, margin, tau, budget, branches, d, L, redraft) != []
    # ascending order flipped (descending-margin admission) breaks the priority pin
    flipped = oracle.build_tree(top, -margin + 3.0, root, L, tau, budget, branches, d, redraft)
    assert check_tree(flipped, top, margin, tau, budget, branches, d, L, redraft) != []
    # a non-strict gate (<=) admits margin == tau
    m32 = np.full((1, 4), 1.0, dtype=np.float32)
    t_le = oracle.build_tree(top[:1, :4], m32 - np.float32(1e-7), root[:1], L[:1], 1.0, 8, 2, 1)
    assert check_tree(t_le, top[:1, :4], m32, 1.0, 8, 2, 1, L[:1]) != []


# ---------------------------------------------------------------- LM-head argmax pins
def _lm_bruteforce(h, w):
    """Every logit as an exactly rounded sum (math.fsum) of its products, then
    the first maximum by a scan: the definition with no library matmul."""
    out = []
    for r in range(h.shape[0]):
        best, bi = None, -1
        for v in range(w.shape[0]):
            s = math.fsum(float(h[r, k]) * float(w[v, k]) for k in range(h.shape[1]))
            if best is None or s > best:
                best, bi = s, v
        out.append(bi)
    return np.array(out)


def _lm_case(seed, rows=6, V=41, d=12):
    rng = np.random.default_rng(seed)
    h = W.bf16_to_f64(W.to_bf16(rng.standard_normal((rows, d)).astype(np.float32)))
    w = W.bf16_to_f64(W.to_bf16(rng.standard_normal((V, d)).astype(np.float32)))
    w[7] = w[3]                        # two identical rows: ties between ids 3 and 7
    h[0] = w[3] * 4.0                  # row 0 prefers that direction
    return h, w


@pytest.mark.parametrize("seed", range(4))
def test_lm_head_argmax_bruteforce(seed):
    h, w = _lm_case(seed)
    got = oracle.lm_head_argmax(h, w)
    assert np.array_equal(got, _lm_bruteforce(h, w))
    assert got[0] == 3                 # the tie between 3 and 7 goes to the lower id


def test_lm_head_argmax_basis_rows_and_square_shape():
    """hidden = c e_k picks the first maximum (c > 0) or first minimum (c < 0)
    of the weight's column k; a square weight, whose transpose has the same
    shape, tells w from w^T."""
    rng = np.random.default_rng(3)
    d = 9
    w = W.bf16_to_f64(W.to_bf16(rng.standard_normal((d, d)).astype(np.float32)))
    for k in range(d):
        for c in (1.0, -2.0):
            h = np.zeros((1, d))
            h[0, k] = c
            col = w[:, k] * c
            assert oracle.lm_head_argmax(h, w)[0] == int(np.flatnonzero(col == col.max())[0])
    h = W.bf16_to_f64(W.to_bf16(rng.standard_normal((5, d)).astype(np.float32)))
    assert np.array_equal(oracle.lm_head_argmax(h, w), _lm_bruteforce(h, w))
    assert not np.array_equal(_lm_bruteforce(h, w.T), _lm_bruteforce(h, w))


def test_lm_head_argmax_planted_stand_in_target():
    """The synthetic hidden states built from a planted token give that token,
    at the serving vocabulary with a small model width (the construction's
    logit margin is about 12 against N(0, 1) noise)."""
    w = W.lm_head_weight(151936, 128, 11)
    planted = np.array([0, 151935, 5, -1, 77777, 5])
    h = W.lm_head_hidden(6, w, 11, planted, strength=40.0)
    got = oracle.lm_head_argmax(W.bf16_to_f64(h), w.to(torch.float32).numpy())
    sel = planted >= 0
    assert np.array_equal(got[sel], planted[sel])


def test_lm_head_pins_catch_planted_mistakes():
    """A transposed weight, a last-maximum tie rule and a dropped feature must
    each fail the brute-force or tie pins."""
    h, w = _lm_case(0, rows=5, V=12, d=12)
    good = _lm_bruteforce(h, w)

    def transposed(h, w):
        return oracle.lm_head_argmax(h, w.T)

    def last_max(h, w):
        lg = h @ w.T
        return np.array([len(r) - 1 - int(np.argmax(r[::-1])) for r in lg])

    def dropped_feature(h, w):
        return oracle.lm_head_argmax(h[:, :-1], w[:, :-1])

    h2 = h.copy()
    h2[1:, -1] *= 64.0                  # the last feature decides rows 1..4
    good2 = _lm_bruteforce(h2, w)
    assert np.array_equal(oracle.lm_head_argmax(h, w), good)
    assert not np.array_equal(transposed(h, w), good)
    assert last_max(h, w)[0] == 7 and good[0] == 3
    assert not np.array_equal(dropped_feature(h2, w), good2)
