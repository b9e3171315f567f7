"""Pins of the oracle's draft-tree verification (ancestor-masked attention
and the greedy walk of the tree).

Attention is pinned against torch's scaled_dot_product_attention in float64
with a mask built from the transitive closure of the tree's adjacency matrix
(reachability by repeated boolean matrix products, not by walking parents),
against the chain oracle on the gathered root-to-node path, and by mask and
relabelling invariances. The walk is pinned by hand-worked trees, by brute
force over all root-to-node paths, and by the chain acceptance rule.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_08721_gb300 import workloads


def _bf16(shape, rng, scale=1.0):
    return torch.from_numpy((rng.standard_normal(shape) * scale).astype(np.float32)).to(torch.bfloat16)


def _closure(parent_row, n):
    """visible[t, a]: a is t or an ancestor of t, by boolean matrix powers."""
    A = np.zeros((n + 1, n + 1), bool)
    for t in range(1, n + 1):
        A[t, parent_row[t]] = True
    R = np.eye(n + 1, dtype=bool)
    P = np.eye(n + 1, dtype=bool)
    for _ in range(n):
        P = (P.astype(np.int64) @ A.astype(np.int64)) > 0
        R |= P
    return R


def _inputs(rng, B, K, Hq, Hkv, d, kv_len, S):
    return (_bf16((B, K + 1, Hq, d), rng), _bf16((B, Hkv, S, d), rng, 2.0), _bf16((B, Hkv, S, d), rng))


@pytest.mark.parametrize("shape,K", [("random", 9), ("topk", 9), ("star", 9), ("ddtree", 9), ("ddtree", 130),
                                     ("random", 130)])
@pytest.mark.parametrize("Hq,Hkv,d", [(4, 2, 16), (3, 1, 8)])
def test_tree_attn_matches_sdpa_with_closure_mask(shape, K, Hq, Hkv, d):
    rng = np.random.default_rng(5 + Hq * 10 + d)
    B = 3
    kv_len = np.array([0, 5, 21], np.int32)
    L = np.array([K, K // 2, K - 2], np.int32)
    S = (21 + K + 1 + 63) // 64 * 64
    Q, Kc, Vc = _inputs(rng, B, K, Hq, Hkv, d, kv_len, S)
    par = workloads.draft_tree(B, K, L, seed=3, shape=shape)
    scale = 1.0 / np.sqrt(d)
    O, lse = oracle.verify_attn_tree(Q, Kc, Vc, kv_len, L, par, scale)
    g = Hq // Hkv
    for b in range(B):
        n, kv = int(L[b]), int(kv_len[b])
        vis = _closure(par[b], n)
        mask = np.zeros((n + 1, kv + n + 1), bool)
        mask[:, :kv] = True
        mask[:, kv:] = vis
        for h in range(Hq):
            q = Q[b, :n + 1, h].double()[None, None]
            k = Kc[b, h // g, :kv + n + 1].double()[None, None]
            v = Vc[b, h // g, :kv + n + 1].double()[None, None]
            ref = torch.nn.functional.scaled_dot_product_attention(
                q, k, v, attn_mask=torch.from_numpy(mask), scale=scale)[0, 0].numpy()
            np.testing.assert_allclose(O[b, :n + 1, h], ref, rtol=1e-11, atol=1e-12)
            s = (q[0, 0] @ k[0, 0].T).numpy() * scale
            s[~mask] = -np.inf
            m = s.max(axis=1)
            np.testing.assert_allclose(lse[b, :n + 1, h], m + np.log(np.exp(s - m[:, None]).sum(1)), rtol=1e-12)
        assert np.all(np.isnan(O[b, n + 1:]))


@pytest.mark.parametrize("budget", [64, 512])
def test_ddtree_generator_shape(budget):
    """Node numbers are a topological order, depth stays within the block
    length, and every node but the budget's last is a candidate's best-first
    expansion (siblings appear in rank order: a node's children are
    numbered after it)."""
    L = np.full(8, budget)
    par = workloads.draft_tree(8, budget, L, seed=1, shape="ddtree", depth=16)
    assert par.shape == (8, budget + 1)
    for b in range(8):
        dep = np.zeros(budget + 1, int)
        for t in range(1, budget + 1):
            assert 0 <= par[b, t] < t
            dep[t] = dep[par[b, t]] + 1
        assert dep.max() <= 16
    # the same seed gives the same trees
    np.testing.assert_array_equal(par, workloads.draft_tree(8, budget, L, seed=1, shape="ddtree", depth=16))


def test_chain_tree_is_the_chain_verify():
    rng = np.random.default_rng(11)
    B, K, Hq, Hkv, d = 4, 12, 4, 1, 16
    kv_len = np.array([3, 0, 64, 17], np.int32)
    L = np.array([12, 0, 5, 9], np.int32)
    S = 80
    Q, Kc, Vc = _inputs(rng, B, K, Hq, Hkv, d, kv_len, S)
    par = workloads.draft_tree(B, K, L, seed=0, shape="chain")
    O1, l1 = oracle.verify_attn(Q, Kc, Vc, kv_len, L)
    O2, l2 = oracle.verify_attn_tree(Q, Kc, Vc, kv_len, L, par)
    np.testing.assert_array_equal(O1, O2)
    np.testing.assert_array_equal(l1, l2)


def test_node_equals_chain_verify_of_its_gathered_path():
    """Node t of a tree attends exactly as row 0 of a chain whose cache is the
    prefix followed by the keys of t's root path (ancestors in depth order)."""
    rng = np.random.default_rng(12)
    B, K, Hq, Hkv, d = 2, 14, 2, 2, 8
    kv_len = np.array([6, 30], np.int32)
    L = np.array([14, 10], np.int32)
    S = 48
    Q, Kc, Vc = _inputs(rng, B, K, Hq, Hkv, d, kv_len, S)
    par = workloads.draft_tree(B, K, L, seed=9, shape="random")
    O, lse = oracle.verify_attn_tree(Q, Kc, Vc, kv_len, L, par)
    for b in range(B):
        kv = int(kv_len[b])
        for t in range(int(L[b]) + 1):
            path = [t]
            while path[-1] != 0:
                path.append(int(par[b, path[-1]]))
            path = path[::-1]                              # root .. t
            keys = list(range(kv)) + [kv + a for a in path]
            Kg = Kc[b:b + 1, :, keys]
            Vg = Vc[b:b + 1, :, keys]
            Qg = torch.zeros((1, 1, Hq, d), dtype=torch.bfloat16)
            Qg[0, 0] = Q[b, t]
            # chain row 0 sees keys 0 .. kv' with kv' = len(keys) - 1
            Oc, lc = oracle.verify_attn(Qg, Kg.contiguous(), Vg.contiguous(),
                                        np.array([len(keys) - 1], np.int32), np.array([0], np.int32))
            np.testing.assert_array_equal(O[b, t], Oc[0, 0])
            np.testing.assert_array_equal(lse[b, t], lc[0, 0])


def test_non_ancestor_keys_do_not_matter_and_ancestors_do():
    rng = np.random.default_rng(13)
    B, K, Hq, Hkv, d = 1, 10, 2, 1, 16
    kv_len = np.array([9], np.int32)
    L = np.array([10], np.int32)
    S = 24
    Q, Kc, Vc = _inputs(rng, B, K, Hq, Hkv, d, kv_len, S)
    par = workloads.draft_tree(B, K, L, seed=4, shape="topk")
    O, _ = oracle.verify_attn_tree(Q, Kc, Vc, kv_len, L, par)
    vis = _closure(par[0], 10)
    for t in range(11):
        others = [a for a in range(11) if not vis[t, a]]
        anc = [a for a in range(11) if vis[t, a]]
        K2, V2 = Kc.clone(), Vc.clone()
        for a in others:
            K2[0, :, 9 + a] = _bf16((Hkv, d), rng, 5.0)
            V2[0, :, 9 + a] = _bf16((Hkv, d), rng, 5.0)
        O2, _ = oracle.verify_attn_tree(Q, K2, V2, kv_len, L, par)
        np.testing.assert_array_equal(O[0, t], O2[0, t])
        a = anc[-1]
        V3 = Vc.clone()
        V3[0, :, 9 + a] += 1.0
        O3, _ = oracle.verify_attn_tree(Q, Kc, V3, kv_len, L, par)
        assert np.all(np.abs(O3[0, t] - O[0, t]) > 0)


def test_relabelling_the_tree_permutes_the_rows():
    """Another topological numbering of the same tree (block keys, queries and
    parents permuted alike) gives the same output per node."""
    rng = np.random.default_rng(14)
    B, K, Hq, Hkv, d = 1, 8, 2, 1, 16
    kv_len = np.array([5], np.int32)
    L = np.array([8], np.int32)
    S = 16
    Q, Kc, Vc = _inputs(rng, B, K, Hq, Hkv, d, kv_len, S)
    # a tree with two branches; number branch B before branch A
    par = np.array([[0, 0, 1, 2, 0, 4, 5, 3, 6]], np.int32)
    #                  node: 1  2  3  4  5  6  7  8
    # relabel: keep 0, branch {4,5,6,8} first, then {1,2,3,7}
    new_of_old = {0: 0, 4: 1, 5: 2, 6: 3, 8: 4, 1: 5, 2: 6, 3: 7, 7: 8}
    old_of_new = {v: k for k, v in new_of_old.items()}
    par2 = np.zeros_like(par)
    for t in range(1, 9):
        par2[0, t] = new_of_old[int(par[0, old_of_new[t]])]
        assert par2[0, t] < t
    Q2, K2, V2 = Q.clone(), Kc.clone(), Vc.clone()
    for t in range(9):
        Q2[0, t] = Q[0, old_of_new[t]]
        K2[0, :, 5 + t] = Kc[0, :, 5 + old_of_new[t]]
        V2[0, :, 5 + t] = Vc[0, :, 5 + old_of_new[t]]
    O, l1 = oracle.verify_attn_tree(Q, Kc, Vc, kv_len, L, par)
    O2, l2 = oracle.verify_attn_tree(Q2, K2, V2, kv_len, L, par2)
    for t in range(9):
        np.testing.assert_array_equal(O[0, old_of_new[t]], O2[0, t])
        np.testing.assert_array_equal(l1[0, old_of_new[t]], l2[0, t])


@pytest.mark.parametrize("bad", [[0, 0, 2], [0, -1, 0], [0, 0, 5]])
def test_tree_attn_rejects_bad_parents(bad):
    rng = np.random.default_rng(15)
    Q, Kc, Vc = _inputs(rng, 1, 2, 2, 1, 8, None, 8)
    with pytest.raises(oracle.OracleError):
        oracle.verify_attn_tree(Q, Kc, Vc, np.array([1], np.int32), np.array([2], np.int32),
                                np.array([bad], np.int32))


# ---------------------------------------------------------------------------
# greedy walk
# ---------------------------------------------------------------------------
def _onehot_rows(args, V, K1):
    """Target rows whose argmax at node i is args[i] (logit 3, others ~N(0,.1))."""
    rng = np.random.default_rng(99)
    x = (rng.standard_normal((K1, V)) * 0.1).astype(np.float32)
    for i, a in enumerate(args):
        x[i, a] = 3.0
    return x


# Hand-worked tree, V = 6, K = 6:
#   node:   1  2  3  4  5  6
#   parent: 0  0  1  1  2  4
#   token:  2  4  1  5  0  3
_PAR = [0, 0, 0, 1, 1, 2, 4]
_TOK = [2, 4, 1, 5, 0, 3]


@pytest.mark.parametrize("args,L,expect", [
    # row 0 picks 2 -> node 1; row 1 picks 5 -> node 4; row 4 picks 3 -> node 6; row 6 -> bonus 1
    ([2, 5, 0, 0, 3, 0, 1], 6, (3, 6, 1)),
    # row 0 picks 4 -> node 2; row 2 picks 0 -> node 5 (a leaf); bonus = argmax of row 5 = 2
    ([4, 0, 0, 0, 0, 2, 0], 6, (2, 5, 2)),
    # row 0 picks 3: no child carries 3
    ([3, 5, 0, 0, 3, 0, 1], 6, (0, 0, 3)),
    # L = 5 drops node 6: the walk stops at node 4 and emits row 4's argmax 3
    ([2, 5, 0, 0, 3, 0, 1], 5, (2, 4, 3)),
    # L = 0: only the root's row
    ([2, 5, 0, 0, 3, 0, 1], 0, (0, 0, 2)),
])
def test_tree_walk_hand_worked(args, L, expect):
    V, K = 6, 6
    x = _onehot_rows(args, V, K + 1)[None]
    n, last, bonus = oracle.accept_tree_greedy(x, np.array([_TOK], np.int32), np.array([_PAR], np.int32),
                                               np.array([L], np.int32))
    assert (int(n[0]), int(last[0]), int(bonus[0])) == expect


def _brute_force_walk(x, tok, par, L):
    """Deepest node whose every edge on the root path matches the parent row's
    argmax (unique when siblings carry distinct tokens)."""
    best, depth_best = 0, 0
    for t in range(1, L + 1):
        ok, depth, a = True, 0, t
        while a != 0:
            p = par[a]
            if tok[a - 1] != int(np.argmax(x[p])):
                ok = False
                break
            depth += 1
            a = p
        if ok and depth > depth_best:
            best, depth_best = t, depth
    return depth_best, best, int(np.argmax(x[best]))


@pytest.mark.parametrize("shape", ["random", "topk", "star", "chain"])
def test_tree_walk_matches_brute_force(shape):
    rng = np.random.default_rng({"random": 1, "topk": 2, "star": 3, "chain": 4}[shape])
    B, K, V = 64, 20, 24
    L = rng.integers(0, K + 1, size=B).astype(np.int32)
    par = workloads.draft_tree(B, K, L, seed=5, shape=shape)
    tok = np.zeros((B, K), np.int32)
    for b in range(B):
        # distinct tokens among siblings
        for p in range(K + 1):
            kids = [t for t in range(1, int(L[b]) + 1) if par[b, t] == p]
            vals = rng.permutation(V)[:len(kids)]
            for t, v in zip(kids, vals):
                tok[b, t - 1] = v
    # rows make a match likely: argmax = one of the node's children's tokens
    x = (rng.standard_normal((B, K + 1, V)) * 0.1).astype(np.float32)
    for b in range(B):
        for p in range(K + 1):
            kids = [t for t in range(1, int(L[b]) + 1) if par[b, t] == p]
            if kids and rng.random() < 0.8:
                x[b, p, tok[b, kids[rng.integers(len(kids))] - 1]] = 2.0
    n, last, bonus = oracle.accept_tree_greedy(x, tok, par, L)
    deep = 0
    for b in range(B):
        exp = _brute_force_walk(x[b], tok[b], par[b], int(L[b]))
        assert (int(n[b]), int(last[b]), int(bonus[b])) == exp, b
        deep = max(deep, exp[0])
    assert deep >= (1 if shape == "star" else 3)


def test_chain_tree_walk_is_greedy_acceptance():
    rng = np.random.default_rng(21)
    B, K, V = 32, 16, 50
    L = rng.integers(0, K + 1, size=B).astype(np.int32)
    x = rng.standard_normal((B, K + 1, V)).astype(np.float32)
    tok = np.argmax(x[:, :K], axis=2).astype(np.int32)
    # break the chain at random places
    for b in range(B):
        j = rng.integers(0, K + 4)
        if j < K:
            tok[b, j] = (tok[b, j] + 1) % V
    par = workloads.draft_tree(B, K, L, seed=0, shape="chain")
    n, last, bonus = oracle.accept_tree_greedy(x, tok, par, L)
    n2, bonus2, _ = oracle.accept(x, np.zeros((B, K, V), np.float32), tok, L, np.zeros(B, np.float32), seed=0)
    np.testing.assert_array_equal(n, n2)
    np.testing.assert_array_equal(bonus, bonus2)
    np.testing.assert_array_equal(last, n)


@pytest.mark.parametrize("case", ["parent", "token", "length"])
def test_tree_walk_rejects_bad_input(case):
    x = np.zeros((1, 3, 4), np.float32)
    tok = np.array([[1, 2]], np.int32)
    par = np.array([[0, 0, 1]], np.int32)
    L = np.array([2], np.int32)
    if case == "parent":
        par = np.array([[0, 0, 2]], np.int32)
    elif case == "token":
        tok = np.array([[1, 4]], np.int32)
    else:
        L = np.array([3], np.int32)
    with pytest.raises(oracle.OracleError):
        oracle.accept_tree_greedy(x, tok, par, L)


# ---------------------------------------------------------------------------
# sampling walk (temperature > 0)
# ---------------------------------------------------------------------------
def _softmax(y, T):
    z = np.asarray(y, np.float64) / T
    e = np.exp(z - z.max())
    return e / e.sum()


def _chi2_ok(counts, probs, n):
    """Pearson chi-square against expected counts, cells with >= 5 expected;
    accept unless the statistic is beyond the 1e-4 upper tail."""
    from scipy.stats import chi2

    exp = probs * n
    keep = exp >= 5
    stat = float(((counts[keep] - exp[keep]) ** 2 / exp[keep]).sum()) + 0.0
    rest_o, rest_e = counts[~keep].sum(), exp[~keep].sum()
    dof = int(keep.sum()) - 1
    if rest_e >= 5:
        stat += (rest_o - rest_e) ** 2 / rest_e
        dof += 1
    return stat < chi2.ppf(1 - 1e-4, max(dof, 1)), stat


def test_tree_sampling_at_zero_temperature_is_the_greedy_walk():
    rng = np.random.default_rng(40)
    B, K, V = 40, 12, 30
    L = rng.integers(0, K + 1, size=B).astype(np.int32)
    par = workloads.draft_tree(B, K, L, seed=3, shape="random")
    x = rng.standard_normal((B, K + 1, V)).astype(np.float32)
    tok = rng.integers(0, V, size=(B, K)).astype(np.int32)
    for b in range(B):   # make some matches
        for t in range(1, int(L[b]) + 1):
            if rng.random() < 0.7:
                tok[b, t - 1] = int(np.argmax(x[b, par[b, t]]))
    n, last, bonus, flag = oracle.accept_tree(x, tok, par, L, np.zeros(B, np.float32), seed=7)
    n2, last2, bonus2 = oracle.accept_tree_greedy(x, tok, par, L)
    np.testing.assert_array_equal(n, n2)
    np.testing.assert_array_equal(last, last2)
    np.testing.assert_array_equal(bonus, bonus2)
    assert not flag.any()


def test_tree_sampling_root_draw_follows_the_target():
    """With no children the round emits one draw from softmax(row / T)."""
    V, T, B = 7, 0.8, 40000
    y = np.array([1.0, -0.5, 2.0, 0.3, 0.3, -2.0, 1.5], np.float32)
    x = np.broadcast_to(y, (B, 1, V)).copy()
    n, last, bonus, flag = oracle.accept_tree(x, np.zeros((B, 0), np.int32), np.zeros((B, 1), np.int32),
                                              np.zeros(B, np.int32), np.full(B, T, np.float32), seed=123)
    assert not n.any() and not last.any()
    ok, stat = _chi2_ok(np.bincount(bonus, minlength=V).astype(float), _softmax(y, T), B)
    assert ok, stat


def test_tree_sampling_is_lossless_on_a_small_tree():
    """The emitted token sequence follows the target's own sampling along the
    tree, P(x1, x2, ...) = p_0(x1) p_{node(x1)}(x2) ..., enumerated exactly.

    Tree (V = 4): node 1 (token 0) and node 2 (token 2) under the root, node 3
    (token 1) under node 1, node 4 (token 3) under node 2."""
    V, T, B = 4, 0.7, 60000
    par = np.array([0, 0, 0, 1, 2], np.int32)
    tok = np.array([0, 2, 1, 3], np.int32)
    rows = np.array([[0.5, -1.0, 0.2, 0.0],     # root
                     [-0.3, 0.9, 0.1, -1.2],    # node 1
                     [0.0, 0.4, -0.6, 0.7],     # node 2
                     [1.1, -0.2, 0.3, 0.0],     # node 3 (leaf)
                     [-0.5, 0.5, 0.2, 0.8]],    # node 4 (leaf)
                    np.float32)
    p = [_softmax(r, T) for r in rows]
    child = {(0, 0): 1, (0, 2): 2, (1, 1): 3, (2, 3): 4}
    probs = {}

    def walk(node, prefix, pr):
        for v in range(V):
            q = pr * p[node][v]
            if (node, v) in child:
                walk(child[(node, v)], prefix + (v,), q)
            else:
                probs[prefix + (v,)] = q
    walk(0, (), 1.0)
    assert abs(sum(probs.values()) - 1.0) < 1e-12
    x = np.broadcast_to(rows, (B, 5, V)).copy()
    n, last, bonus, flag = oracle.accept_tree(x, np.broadcast_to(tok, (B, 4)).copy(),
                                              np.broadcast_to(par, (B, 5)).copy(), np.full(B, 4, np.int32),
                                              np.full(B, T, np.float32), seed=2024, round_offset=3)
    keys = sorted(probs)
    index = {k: i for i, k in enumerate(keys)}
    counts = np.zeros(len(keys))
    node_token = {1: 0, 2: 2, 3: 1, 4: 3}
    for b in range(B):
        path, t = [], int(last[b])
        while t != 0:
            path.append(node_token[t])
            t = int(par[t])
        assert len(path) == n[b]
        counts[index[tuple(path[::-1]) + (int(bonus[b]),)]] += 1
    ok, stat = _chi2_ok(counts, np.array([probs[k] for k in keys]), B)
    assert ok, stat
    # the root's children are accepted with the target's probability of their tokens
    acc = float((n >= 1).mean())
    assert abs(acc - (p[0][0] + p[0][2])) < 4 * np.sqrt(acc * (1 - acc) / B)


def test_tree_sampling_sequence_offset_and_rounds():
    """Draws depend on the global sequence index and the round: a batch split
    with seq_offset reproduces the unsplit batch; another round differs."""
    rng = np.random.default_rng(41)
    B, K, V = 24, 10, 50
    L = np.full(B, K, np.int32)
    par = workloads.draft_tree(B, K, L, seed=8, shape="topk")
    x = (rng.standard_normal((B, K + 1, V)) * 2).astype(np.float32)
    tok = rng.integers(0, V, size=(B, K)).astype(np.int32)
    T = np.full(B, 1.0, np.float32)
    full = oracle.accept_tree(x, tok, par, L, T, seed=5, round_offset=2)
    part = oracle.accept_tree(x[10:], tok[10:], par[10:], L[10:], T[10:], seed=5, round_offset=2, seq_offset=10)
    for a, b in zip(full, part):
        np.testing.assert_array_equal(a[10:], b)
    other = oracle.accept_tree(x, tok, par, L, T, seed=5, round_offset=3)
    assert (other[2] != full[2]).any()


def test_tree_sampling_rejects_bad_temperature():
    x = np.zeros((1, 2, 4), np.float32)
    with pytest.raises(oracle.OracleError):
        oracle.accept_tree(x, np.array([[1]], np.int32), np.array([[0, 0]], np.int32), np.array([1], np.int32),
                           np.array([-1.0], np.float32), seed=0)
