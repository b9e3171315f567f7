"""GPU parity: draft-tree verification (ancestor-masked verify attention and
the greedy walk of the tree) vs. the oracle, bit-for-bit vs. the chain
kernels on a chain tree, and the paged tree kernel vs. the dense one."""
import numpy as np
import pytest
import torch

from helpers import check_attn, cuda
from paper_2608_08721_gb300 import binding as lr
from paper_2608_08721_gb300 import workloads

pytestmark = pytest.mark.gpu


def _layers(B, K, Hq, Hkv, d, S, seed, n_layers=1):
    g = torch.Generator(device="cuda").manual_seed(seed)
    out = []
    for _ in range(n_layers):
        Q = torch.randn((B, K + 1, Hq, d), generator=g, device=cuda()).to(torch.bfloat16)
        Kc = (torch.randn((B, Hkv, S, d), generator=g, device=cuda()) * 2.0).to(torch.bfloat16)
        Vc = torch.randn((B, Hkv, S, d), generator=g, device=cuda()).to(torch.bfloat16)
        out.append({"Q": Q, "Kc": Kc, "Vc": Vc})
    return out


def _i32(x):
    return torch.as_tensor(np.asarray(x), dtype=torch.int32).to(cuda())


def _run_tree(layers, parent, kv, L, K):
    B, _, Hq, d = layers[0]["Q"].shape
    _, Hkv, S, _ = layers[0]["Kc"].shape
    ws = lr.Workspace(B, K, 1, Hq, Hkv, d, S, device=cuda())
    outs, lses = lr.libraspec_verify_attn_tree_layers(layers, _i32(parent), _i32(kv), _i32(L), ws, want_lse=True)
    torch.cuda.synchronize()
    return outs, lses, lr.libraspec_get_status(ws)


@pytest.mark.parametrize("shape", ["topk", "random", "star"])
@pytest.mark.parametrize("d,Hq,Hkv", [(128, 32, 8), (64, 8, 2), (128, 28, 4)])
def test_tree_attn_matches_oracle(orc, shape, d, Hq, Hkv):
    K = 20
    # block keys straddling a tile edge (kv % 64 near 63), at a tile start, a
    # fresh sequence, a long prefix split over CTAs
    kv = [0, 62, 64, 700, 2900, 127]
    L = [20, 20, 5, 1, 17, 11]
    B = len(kv)
    S = (max(k + l + 1 for k, l in zip(kv, L)) + 63) // 64 * 64
    parent = workloads.draft_tree(B, K, L, seed=d + Hq, shape=shape)
    layers = _layers(B, K, Hq, Hkv, d, S, seed=d + Hq + len(shape))
    outs, lses, status = _run_tree(layers, parent, kv, L, K)
    assert status == 0
    O_ref, lse_ref = orc.verify_attn_tree(layers[0]["Q"], layers[0]["Kc"], layers[0]["Vc"], np.array(kv),
                                          np.array(L), parent)
    check_attn(outs[0], lses[0], O_ref, lse_ref, L)


def test_tree_attn_full_depth_and_width(orc):
    """K = 64 (the mask's last bit): a depth-64 chain, a 64-leaf star and a
    random tree, with the block at every offset within a tile."""
    K, Hq, Hkv, d = 64, 8, 2, 128
    kv = [0, 1, 63, 64, 65, 191]
    L = [64] * 6
    B = len(kv)
    S = (max(kv) + K + 1 + 63) // 64 * 64
    layers = _layers(B, K, Hq, Hkv, d, S, seed=64)
    for shape in ("chain", "star", "random"):
        parent = workloads.draft_tree(B, K, L, seed=7, shape=shape)
        outs, lses, status = _run_tree(layers, parent, kv, L, K)
        assert status == 0
        O_ref, lse_ref = orc.verify_attn_tree(layers[0]["Q"], layers[0]["Kc"], layers[0]["Vc"], np.array(kv),
                                              np.array(L), parent)
        check_attn(outs[0], lses[0], O_ref, lse_ref, L)


@pytest.mark.parametrize("d,Hq,Hkv", [(128, 32, 8), (64, 8, 2)])
def test_chain_tree_is_bit_identical_to_chain_call(d, Hq, Hkv):
    K = 16
    kv = [5, 63, 1000, 4096, 0]
    L = [16, 3, 16, 9, 0]
    B = len(kv)
    S = (max(k + l + 1 for k, l in zip(kv, L)) + 63) // 64 * 64
    layers = _layers(B, K, Hq, Hkv, d, S, seed=3, n_layers=2)
    parent = workloads.draft_tree(B, K, L, seed=0, shape="chain")
    outs, lses, status = _run_tree(layers, parent, kv, L, K)
    assert status == 0
    ws = lr.Workspace(B, K, 1, Hq, Hkv, d, S, device=cuda())
    o2, l2 = lr.libraspec_verify_attn_layers(layers, _i32(kv), _i32(L), ws, want_lse=True)
    torch.cuda.synchronize()
    for l in range(2):
        for b in range(B):
            assert torch.equal(outs[l][b, :L[b] + 1], o2[l][b, :L[b] + 1])
            assert torch.equal(lses[l][b, :L[b] + 1], l2[l][b, :L[b] + 1])


def test_tree_layers_in_one_launch_long_cache(orc):
    """Three layers in one launch, 8b-like heads, a 20k prefix split over many
    CTAs: sampled rows against the oracle."""
    K, Hq, Hkv, d = 16, 32, 8, 128
    kv, L = [20000, 300], [16, 12]
    S = (max(kv) + K + 1 + 63) // 64 * 64
    layers = _layers(2, K, Hq, Hkv, d, S, seed=8, n_layers=3)
    parent = workloads.draft_tree(2, K, L, seed=8, shape="topk")
    outs, lses, status = _run_tree(layers, parent, kv, L, K)
    assert status == 0
    rows = np.array([(b, h, t) for b in range(2) for h in (0, 13, Hq - 1) for t in range(L[b] + 1)], np.int32)
    for l in range(3):
        O_ref, lse_ref = orc.verify_attn_tree(layers[l]["Q"], layers[l]["Kc"], layers[l]["Vc"], np.array(kv),
                                              np.array(L), parent, rows=rows)
        check_attn(outs[l], lses[l], O_ref, lse_ref, L, rows=[tuple(r) for r in rows])


def test_tree_paged_is_bit_identical_to_dense():
    K, Hq, Hkv, d, P = 24, 32, 8, 128, 128
    kv = [0, 63, 700, 3000]
    L = [24, 10, 24, 7]
    B = len(kv)
    rng = np.random.default_rng(31)
    S = max(k + l + 1 for k, l in zip(kv, L))
    max_pages = -(-S // P)
    n_pages = B * max_pages + 3
    perm = rng.permutation(n_pages)[: B * max_pages].reshape(B, max_pages).astype(np.int32)
    dense = _layers(B, K, Hq, Hkv, d, max_pages * P, seed=31, n_layers=2)
    paged = []
    for lay in dense:
        Kp = torch.zeros((n_pages, Hkv, P, d), dtype=torch.bfloat16, device=cuda())
        Vp = torch.zeros_like(Kp)
        for b in range(B):
            for j in range(max_pages):
                Kp[perm[b, j]] = lay["Kc"][b, :, j * P:(j + 1) * P]
                Vp[perm[b, j]] = lay["Vc"][b, :, j * P:(j + 1) * P]
        paged.append({"Q": lay["Q"], "Kp": Kp, "Vp": Vp})
    parent = workloads.draft_tree(B, K, L, seed=31, shape="random")
    o_d, l_d, st = _run_tree(dense, parent, kv, L, K)
    assert st == 0
    ws = lr.Workspace(B, K, 1, Hq, Hkv, d, max_pages * P, device=cuda())
    o_p, l_p = lr.libraspec_verify_attn_tree_paged_layers(paged, _i32(parent), _i32(perm), _i32(kv), _i32(L), ws,
                                                         want_lse=True)
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) == 0
    for l in range(2):
        for b in range(B):
            assert torch.equal(o_p[l][b, :L[b] + 1], o_d[l][b, :L[b] + 1])
            assert torch.equal(l_p[l][b, :L[b] + 1], l_d[l][b, :L[b] + 1])


def test_tree_bad_parent_sets_status():
    K, Hq, Hkv, d = 4, 8, 2, 64
    kv, L = [100, 10], [3, 4]
    layers = _layers(2, K, Hq, Hkv, d, 128, seed=2)
    parent = workloads.draft_tree(2, K, L, seed=2, shape="random")
    parent[1, 3] = 3  # not below its own number
    _, _, status = _run_tree(layers, parent, kv, L, K)
    assert status & lr.ST_BAD_TREE


# ---------------------------------------------------------------------------
# greedy walk
# ---------------------------------------------------------------------------
def _walk_inputs(B, K, V, shape, seed, dtype=torch.float32, peak=6.0):
    """Trees with distinct sibling tokens; target rows whose argmax is often
    one of the node's children's tokens."""
    rng = np.random.default_rng(seed)
    L = rng.integers(0, K + 1, size=B).astype(np.int32)
    L[0], L[-1] = K, 0
    parent = workloads.draft_tree(B, K, L, seed=seed, shape=shape)
    tok = np.zeros((B, K), np.int32)
    g = torch.Generator(device="cuda").manual_seed(seed)
    x = torch.randn((B, K + 1, V), generator=g, device=cuda()) * 0.5
    for b in range(B):
        kids = [[] for _ in range(K + 1)]
        for t in range(1, int(L[b]) + 1):
            kids[parent[b, t]].append(t)
        for p in range(K + 1):
            vals = rng.choice(V, size=len(kids[p]), replace=False)
            for t, v in zip(kids[p], vals):
                tok[b, t - 1] = v
            if kids[p] and rng.random() < 0.85:
                x[b, p, int(tok[b, kids[p][rng.integers(len(kids[p]))] - 1])] = peak
    return x.to(dtype), tok, parent, L


@pytest.mark.parametrize("shape", ["topk", "random", "star", "chain"])
@pytest.mark.parametrize("V", [32000, 152064, 1000])
def test_tree_walk_matches_oracle(orc, shape, V):
    B, K = 48, 24
    x, tok, parent, L = _walk_inputs(B, K, V, shape, seed=V % 97 + len(shape))
    ws = lr.Workspace(B, K, V, 1, 1, 64, 1, device=cuda())
    n, last, bonus = lr.libraspec_accept_tree_greedy(x, _i32(tok), _i32(parent), _i32(L), ws)
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) == 0
    rn, rlast, rbonus = orc.accept_tree_greedy(x.cpu().numpy(), tok, parent, L)
    np.testing.assert_array_equal(n.cpu().numpy(), rn)
    np.testing.assert_array_equal(last.cpu().numpy(), rlast)
    np.testing.assert_array_equal(bonus.cpu().numpy(), rbonus)
    if shape != "star":
        assert rn.max() >= 3


def test_tree_walk_bf16_matches_oracle(orc):
    B, K, V = 32, 64, 128256
    x, tok, parent, L = _walk_inputs(B, K, V, "topk", seed=5, dtype=torch.bfloat16)
    ws = lr.Workspace(B, K, V, 1, 1, 64, 1, device=cuda())
    n, last, bonus = lr.libraspec_accept_tree_greedy(x, _i32(tok), _i32(parent), _i32(L), ws)
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) == 0
    # bf16 widens exactly to f32: the oracle sees the same values
    rn, rlast, rbonus = orc.accept_tree_greedy(x.float().cpu().numpy(), tok, parent, L)
    np.testing.assert_array_equal(n.cpu().numpy(), rn)
    np.testing.assert_array_equal(last.cpu().numpy(), rlast)
    np.testing.assert_array_equal(bonus.cpu().numpy(), rbonus)


def test_chain_tree_walk_equals_greedy_accept():
    B, K, V = 64, 16, 32000
    x, tok, _, L = _walk_inputs(B, K, V, "chain", seed=9)
    parent = workloads.draft_tree(B, K, L, seed=0, shape="chain")
    ws = lr.Workspace(B, K, V, 1, 1, 64, 1, device=cuda())
    n, last, bonus = lr.libraspec_accept_tree_greedy(x, _i32(tok), _i32(parent), _i32(L), ws)
    zeros = torch.zeros((B, K, V), device=cuda())
    n2, b2 = lr.libraspec_accept(x, zeros, _i32(tok), None, None, _i32(L), torch.zeros(B, device=cuda()), 0, ws)
    torch.cuda.synchronize()
    assert torch.equal(n, n2) and torch.equal(bonus, b2) and torch.equal(last, n)


def test_tree_walk_bad_inputs_set_status():
    B, K, V = 2, 4, 100
    x, tok, parent, L = _walk_inputs(B, K, V, "random", seed=1)
    L = np.array([4, 4], np.int32)
    parent = workloads.draft_tree(B, K, L, seed=1, shape="random")
    parent[0, 2] = 2
    tok[1, 0] = V + 3
    ws = lr.Workspace(B, K, V, 1, 1, 64, 1, device=cuda())
    lr.libraspec_accept_tree_greedy(x, _i32(tok), _i32(parent), _i32(L), ws)
    torch.cuda.synchronize()
    st = lr.libraspec_get_status(ws)
    assert st & lr.ST_BAD_TREE and st & lr.ST_BAD_TOKEN


# ---------------------------------------------------------------------------
# node budgets beyond 64 (DDTree runs 64 to 512 nodes): multi-word masks
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("N", [65, 128, 256, 512])
def test_large_tree_attn_matches_oracle(orc, N):
    Hq, Hkv, d = 32, 8, 128
    kv = [4096, 63, 1]
    L = [N, N - 1, N // 2]
    B = len(kv)
    S = (max(k + l + 1 for k, l in zip(kv, L)) + 63) // 64 * 64
    parent = workloads.draft_tree(B, N, L, seed=N, shape="ddtree", depth=16)
    layers = _layers(B, N, Hq, Hkv, d, S, seed=N + 1)
    outs, lses, status = _run_tree(layers, parent, kv, L, N)
    assert status == 0
    if N <= 128:
        O_ref, lse_ref = orc.verify_attn_tree(layers[0]["Q"], layers[0]["Kc"], layers[0]["Vc"], np.array(kv),
                                              np.array(L), parent)
        check_attn(outs[0], lses[0], O_ref, lse_ref, L)
    else:
        rng = np.random.default_rng(N)
        rows = [(b, h, t) for b in range(B) for h in (0, 17, Hq - 1)
                for t in sorted(set([0, 1, L[b]] + list(rng.integers(0, L[b] + 1, 12))))]
        rows = np.array(rows, np.int32)
        O_ref, lse_ref = orc.verify_attn_tree(layers[0]["Q"], layers[0]["Kc"], layers[0]["Vc"], np.array(kv),
                                              np.array(L), parent, rows=rows)
        check_attn(outs[0], lses[0], O_ref, lse_ref, L, rows=[tuple(r) for r in rows])


def test_large_tree_random_shape_small_heads(orc):
    """A uniform random recursive tree (deep, irregular ancestor sets) of 300
    nodes, 8/2 heads, d 64, two layers."""
    N, Hq, Hkv, d = 300, 8, 2, 64
    kv, L = [700, 0], [300, 257]
    S = (max(k + l + 1 for k, l in zip(kv, L)) + 63) // 64 * 64
    parent = workloads.draft_tree(2, N, L, seed=300, shape="random")
    layers = _layers(2, N, Hq, Hkv, d, S, seed=300, n_layers=2)
    outs, lses, status = _run_tree(layers, parent, kv, L, N)
    assert status == 0
    for l in range(2):
        O_ref, lse_ref = orc.verify_attn_tree(layers[l]["Q"], layers[l]["Kc"], layers[l]["Vc"], np.array(kv),
                                              np.array(L), parent)
        check_attn(outs[l], lses[l], O_ref, lse_ref, L)


@pytest.mark.parametrize("N", [128, 512])
def test_large_tree_walk_matches_oracle(orc, N):
    B, V = 16, 32000
    rng = np.random.default_rng(N)
    L = np.full(B, N, np.int32)
    L[1] = N // 3
    parent = workloads.draft_tree(B, N, L, seed=N, shape="ddtree", depth=16)
    tok = np.zeros((B, N), np.int32)
    g = torch.Generator(device="cuda").manual_seed(N)
    x = torch.randn((B, N + 1, V), generator=g, device=cuda()) * 0.5
    for b in range(B):
        kids = [[] for _ in range(N + 1)]
        for t in range(1, int(L[b]) + 1):
            kids[parent[b, t]].append(t)
        for p in range(N + 1):
            vals = rng.choice(V, size=len(kids[p]), replace=False)
            for t, v in zip(kids[p], vals):
                tok[b, t - 1] = v
            if kids[p] and rng.random() < 0.9:
                x[b, p, int(tok[b, kids[p][0] - 1])] = 6.0   # the best-ranked child
    ws = lr.Workspace(B, N, V, 1, 1, 64, 1, device=cuda())
    n, last, bonus = lr.libraspec_accept_tree_greedy(x, _i32(tok), _i32(parent), _i32(L), ws)
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) == 0
    rn, rlast, rbonus = orc.accept_tree_greedy(x.cpu().numpy(), tok, parent, L)
    np.testing.assert_array_equal(n.cpu().numpy(), rn)
    np.testing.assert_array_equal(last.cpu().numpy(), rlast)
    np.testing.assert_array_equal(bonus.cpu().numpy(), rbonus)
    assert rn.max() >= 4


def test_tree_rejects_node_budget_over_limit():
    N = lr.MAX_TREE_NODES + 1
    Q = torch.zeros((1, N + 1, 8, 64), dtype=torch.bfloat16, device=cuda())
    Kc = torch.zeros((1, 2, 1024, 64), dtype=torch.bfloat16, device=cuda())
    ws = lr.Workspace(1, lr.MAX_TREE_NODES, 1, 8, 2, 64, 1024, device=cuda())
    with pytest.raises(lr.LibraspecError):
        lr.libraspec_verify_attn_tree_layers([{"Q": Q, "Kc": Kc, "Vc": Kc}], _i32(np.zeros((1, N + 1))),
                                             _i32([0]), _i32([0]), ws)


# ---------------------------------------------------------------------------
# sampling walk (per-sequence temperature)
# ---------------------------------------------------------------------------
def _assert_exact_unless_flagged(gpu, ref, flag, what):
    gpu, ref, flag = (np.asarray(x) for x in (gpu, ref, flag))
    bad = (gpu != ref) & (flag == 0)
    assert not bad.any(), "%s differs on unflagged sequences %s" % (what, np.nonzero(bad)[0].tolist())


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("N,V", [(24, 32000), (24, 152064), (512, 32000), (130, 1003)])
def test_tree_sampling_walk_matches_oracle(orc, dtype, N, V):
    B = 24 if N <= 130 else 6
    x, tok, parent, L = _walk_inputs(B, N, V, "ddtree" if N > 24 else "topk", seed=N + V % 89, dtype=dtype,
                                     peak=14.0)
    # mixed batch: greedy, cool, neutral and hot sequences
    temps = np.array([[0.0, 0.6, 1.0, 1.6][b % 4] for b in range(B)], np.float32)
    ws = lr.Workspace(B, N, V, 1, 1, 64, 1, device=cuda())
    n, last, bonus = lr.libraspec_accept_tree(x, _i32(tok), _i32(parent), _i32(L),
                                              torch.from_numpy(temps).to(cuda()), 99, ws, round_offset=5,
                                              seq_offset=1000)
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) == 0
    rn, rlast, rbonus, flag = orc.accept_tree(x.float().cpu().numpy(), tok, parent, L, temps, seed=99,
                                              round_offset=5, seq_offset=1000)
    assert flag.sum() <= max(1, B // 10)
    _assert_exact_unless_flagged(n.cpu().numpy(), rn, flag, "n_accepted")
    _assert_exact_unless_flagged(last.cpu().numpy(), rlast, flag, "last_node")
    _assert_exact_unless_flagged(bonus.cpu().numpy(), rbonus, flag, "bonus")
    assert (rn[temps > 0] > 0).any()


def test_tree_sampling_at_zero_temperature_equals_greedy_entry():
    B, N, V = 16, 64, 32000
    x, tok, parent, L = _walk_inputs(B, N, V, "ddtree", seed=12)
    ws = lr.Workspace(B, N, V, 1, 1, 64, 1, device=cuda())
    a = lr.libraspec_accept_tree(x, _i32(tok), _i32(parent), _i32(L), torch.zeros(B, device=cuda()), 3, ws)
    b = lr.libraspec_accept_tree_greedy(x, _i32(tok), _i32(parent), _i32(L), ws)
    torch.cuda.synchronize()
    for u, v in zip(a, b):
        assert torch.equal(u, v)


def test_tree_sampling_root_draw_distribution_on_gpu():
    """Sequences that share one row and have no children: the bonus draws
    follow softmax(row / T) (chi-square, independent of the oracle)."""
    from scipy.stats import chi2

    B, V, T = 4096, 6, 0.9
    y = torch.tensor([0.3, 1.2, -0.4, 0.8, 0.0, 2.0])
    x = y.expand(B, 1, V).contiguous().to(cuda())
    ws = lr.Workspace(B, 0, V, 1, 1, 64, 1, device=cuda())
    _, _, bonus = lr.libraspec_accept_tree(x, torch.zeros((B, 0), dtype=torch.int32, device=cuda()),
                                           torch.zeros((B, 1), dtype=torch.int32, device=cuda()),
                                           torch.zeros(B, dtype=torch.int32, device=cuda()),
                                           torch.full((B,), T, device=cuda()), 11, ws)
    torch.cuda.synchronize()
    counts = np.bincount(bonus.cpu().numpy(), minlength=V)
    p = torch.softmax(y.double() / T, 0).numpy()
    stat = float(((counts - p * B) ** 2 / (p * B)).sum())
    assert stat < chi2.ppf(1 - 1e-4, V - 1), stat


def test_tree_edge_cases_empty_trees_and_fresh_caches(orc):
    """Trees of zero nodes (only the root), fresh caches (kv_len 0) and one
    sequence at the node budget, in one batch."""
    N, Hq, Hkv, d = 40, 8, 2, 128
    kv = [0, 0, 5, 64, 0]
    L = [0, N, 0, N, 1]
    B = len(kv)
    S = (max(k + l + 1 for k, l in zip(kv, L)) + 63) // 64 * 64
    parent = workloads.draft_tree(B, N, L, seed=17, shape="ddtree", depth=16)
    layers = _layers(B, N, Hq, Hkv, d, S, seed=17)
    outs, lses, status = _run_tree(layers, parent, kv, L, N)
    assert status == 0
    O_ref, lse_ref = orc.verify_attn_tree(layers[0]["Q"], layers[0]["Kc"], layers[0]["Vc"], np.array(kv),
                                          np.array(L), parent)
    check_attn(outs[0], lses[0], O_ref, lse_ref, L)
    # the walk of a root-only tree emits the root's argmax
    V = 500
    x, tok, _, _ = _walk_inputs(B, N, V, "random", seed=3)
    ws = lr.Workspace(B, N, V, 1, 1, 64, 1, device=cuda())
    n, last, bonus = lr.libraspec_accept_tree_greedy(x, _i32(tok), _i32(parent), _i32(L), ws)
    torch.cuda.synchronize()
    rn, rlast, rbonus = orc.accept_tree_greedy(x.cpu().numpy(), tok, parent, np.array(L, np.int32))
    np.testing.assert_array_equal(n.cpu().numpy(), rn)
    np.testing.assert_array_equal(bonus.cpu().numpy(), rbonus)
    assert n[0].item() == 0 and bonus[0].item() == int(x[0, 0].argmax())


def test_tree_attn_cost_weighted_split(orc):
    """Draft trees on a batch with more (sequence, kv head) pairs than CTAs
    (the kernel whose Stream-K ranges are cut by cost), two layers in one
    launch, against the oracle."""
    K, Hq, Hkv, d = 16, 32, 8, 128
    rng = np.random.default_rng(31)
    B = 24  # 192 (sequence, kv head) pairs
    kv = rng.integers(0, 1200, size=B).tolist()
    L = rng.integers(0, K + 1, size=B).tolist()
    S = (max(k + l + 1 for k, l in zip(kv, L)) + 63) // 64 * 64
    parent = workloads.draft_tree(B, K, L, seed=31, shape="random")
    layers = _layers(B, K, Hq, Hkv, d, S, seed=31, n_layers=2)
    outs, lses, status = _run_tree(layers, parent, kv, L, K)
    assert status == 0
    for l in range(2):
        O_ref, lse_ref = orc.verify_attn_tree(layers[l]["Q"], layers[l]["Kc"], layers[l]["Vc"], np.array(kv),
                                              np.array(L), parent)
        check_attn(outs[l], lses[l], O_ref, lse_ref, L)
