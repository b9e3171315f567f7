"""GPU parity: block-causal GQA verify attention vs. the fp64 oracle."""
import numpy as np
import pytest
import torch

from helpers import check_attn, cuda
from paper_2608_08721_gb300 import binding as lr
from paper_2608_08721_gb300 import workloads

pytestmark = pytest.mark.gpu


def _inputs(B, K, Hq, Hkv, d, kv, S_cap, seed, scale_k=1.0):
    g = torch.Generator(device="cuda").manual_seed(seed)
    Q = torch.randn((B, K + 1, Hq, d), generator=g, device=cuda()).to(torch.bfloat16)
    Kc = (torch.randn((B, Hkv, S_cap, d), generator=g, device=cuda()) * scale_k).to(torch.bfloat16)
    Vc = torch.randn((B, Hkv, S_cap, d), generator=g, device=cuda()).to(torch.bfloat16)
    return Q, Kc, Vc


def _run(Q, Kc, Vc, kv, L, K):
    B, _, Hq, d = Q.shape
    Hkv, S_cap = Kc.shape[1], Kc.shape[2]
    ws = lr.Workspace(B, K, 1, Hq, Hkv, d, S_cap, device=cuda())
    kv_t = torch.tensor(kv, dtype=torch.int32, device=cuda())
    L_t = torch.tensor(L, dtype=torch.int32, device=cuda())
    O, lse = lr.libraspec_verify_attn(Q, Kc, Vc, kv_t, L_t, ws, want_lse=True)
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) == 0
    return O, lse


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("Hq,Hkv", [(8, 2), (28, 4), (32, 8), (64, 8), (4, 4)])
def test_attn_small_ragged(orc, d, Hq, Hkv):
    K = 9
    kv = [0, 1, 63, 64, 200, 700]
    L = [0, 9, 3, 1, 9, 5]
    B = len(kv)
    S_cap = max(k + l + 1 for k, l in zip(kv, L)) + 3
    Q, Kc, Vc = _inputs(B, K, Hq, Hkv, d, kv, S_cap, seed=Hq * 7 + d, scale_k=2.0)
    O, lse = _run(Q, Kc, Vc, kv, L, K)
    O_ref, lse_ref = orc.verify_attn(Q, Kc, Vc, np.array(kv), np.array(L))
    check_attn(O, lse, O_ref, lse_ref, L)


def test_attn_rows_beyond_L_untouched():
    K, B, Hq, Hkv, d = 6, 2, 8, 2, 64
    kv, L = [30, 5], [2, 0]
    Q, Kc, Vc = _inputs(B, K, Hq, Hkv, d, kv, 48, seed=1)
    ws = lr.Workspace(B, K, 1, Hq, Hkv, d, 48, device=cuda())
    O = torch.full_like(Q, 7.0)
    lr.libraspec_verify_attn(Q, Kc, Vc, torch.tensor(kv, dtype=torch.int32, device=cuda()),
                             torch.tensor(L, dtype=torch.int32, device=cuda()), ws, O=O)
    torch.cuda.synchronize()
    assert torch.all(O[0, 3:] == 7.0) and torch.all(O[1, 1:] == 7.0)
    assert not torch.any(O[0, :3] == 7.0)


@pytest.mark.parametrize("kv", [5000, 20000])
def test_attn_long_split_kv_merge(orc, kv):
    # one sequence, long cache: its row groups spread over many CTAs and are merged
    K, Hq, Hkv, d = 16, 32, 8, 128
    L = [11]
    Q, Kc, Vc = _inputs(1, K, Hq, Hkv, d, [kv], kv + K + 1, seed=kv)
    O, lse = _run(Q, Kc, Vc, [kv], L, K)
    O_ref, lse_ref = orc.verify_attn(Q, Kc, Vc, np.array([kv]), np.array(L))
    check_attn(O, lse, O_ref, lse_ref, L)


@pytest.mark.parametrize("kv", [300, 20000])
@pytest.mark.parametrize("Hq,Hkv,d,L", [(32, 8, 128, 7), (32, 8, 64, 3), (64, 8, 128, 3), (8, 8, 128, 16),
                                        (32, 8, 128, 12)])
def test_attn_small_groups_long_cache(orc, kv, Hq, Hkv, d, L):
    """Row groups of 16 to 52 rows (a few block positions of g heads) over a
    short and a long cache: one CTA per group, and groups split over many
    CTAs whose parts are merged."""
    K = 16
    Q, Kc, Vc = _inputs(1, K, Hq, Hkv, d, [kv], kv + K + 1, seed=kv + Hq + L, scale_k=2.0)
    O, lse = _run(Q, Kc, Vc, [kv], [L], K)
    O_ref, lse_ref = orc.verify_attn(Q, Kc, Vc, np.array([kv]), np.array([L]))
    check_attn(O, lse, O_ref, lse_ref, [L])


@pytest.mark.parametrize("d", [64, 128])
def test_attn_small_groups_ragged(orc, d):
    """Several sequences with small row groups of different sizes, some
    covered by one CTA, some split."""
    K, Hq, Hkv = 9, 32, 8
    kv = [0, 3000, 64, 700, 9000]
    L = [7, 0, 3, 5, 1]
    S_cap = max(k + l + 1 for k, l in zip(kv, L)) + 3
    Q, Kc, Vc = _inputs(len(kv), K, Hq, Hkv, d, kv, S_cap, seed=d + 5, scale_k=2.0)
    O, lse = _run(Q, Kc, Vc, kv, L, K)
    O_ref, lse_ref = orc.verify_attn(Q, Kc, Vc, np.array(kv), np.array(L))
    check_attn(O, lse, O_ref, lse_ref, L)


def test_attn_peaky_scores(orc):
    w = workloads.WORKLOADS["sampling"].scaled(B=4, kv=("uniform", 100, 3000))
    kv = workloads.kv_lengths(w)
    lay = workloads.layer(w, 0, kv, device=cuda(), peaky=True)
    L = np.array([0, 16, 7, 3], np.int32)
    O, lse = _run(lay["Q"], lay["Kc"], lay["Vc"], kv.tolist(), L.tolist(), w.K)
    O_ref, lse_ref = orc.verify_attn(lay["Q"], lay["Kc"], lay["Vc"], kv, L)
    check_attn(O, lse, O_ref, lse_ref, L)


def test_attn_equal_keys_closed_form():
    # all keys equal: every row's output is the mean of its visible values
    B, K, Hq, Hkv, d = 1, 4, 4, 1, 64
    kv = [100]
    L = [4]
    S = 128
    g = torch.Generator(device="cuda").manual_seed(3)
    Q = torch.randn((B, K + 1, Hq, d), generator=g, device=cuda()).to(torch.bfloat16)
    Kc = torch.full((B, Hkv, S, d), 0.25, device=cuda(), dtype=torch.bfloat16)
    Vc = torch.randn((B, Hkv, S, d), generator=g, device=cuda()).to(torch.bfloat16)
    O, _ = _run(Q, Kc, Vc, kv, L, K)
    for t in range(5):
        mean = Vc[0, 0, : kv[0] + t + 1].float().mean(0)
        for h in range(Hq):
            assert torch.allclose(O[0, t, h].float(), mean, atol=1e-2, rtol=1e-2)


@pytest.mark.parametrize("name", ["tiny", "8b", "sampling", "ragged", "70b"])
def test_attn_full_size_sampled_rows(orc, name):
    """One layer at the workload's full size, in the launch configuration the
    benchmark uses; the oracle checks a sample of rows one by one."""
    w = workloads.WORKLOADS[name]
    kv = workloads.kv_lengths(w)
    rng = np.random.default_rng(len(name))
    L = rng.integers(0, w.K + 1, size=w.B).astype(np.int32)
    L[0] = w.K
    if w.B > 1:
        L[1] = 0
    lay = workloads.layer(w, 3, kv, device=cuda())
    O, lse = _run(lay["Q"], lay["Kc"], lay["Vc"], kv.tolist(), L.tolist(), w.K)
    rows = []
    for b in range(w.B):
        for h in rng.choice(w.Hq, size=min(3, w.Hq), replace=False):
            rows.append((b, int(h), int(L[b])))
            rows.append((b, int(h), int(rng.integers(0, L[b] + 1))))
    # complete (sequence, kv head) row groups: every head of the kv head at every verified
    # position, the rows the kernel's split-KV merge writes together (sequence 0 at L = K,
    # so (K + 1) g rows: one full 128-row tile or more; and the last sequence)
    g = w.Hq // w.Hkv
    for b in sorted({0, w.B - 1}):
        kvh = int(rng.integers(0, w.Hkv))
        rows += [(b, kvh * g + i, t) for i in range(g) for t in range(int(L[b]) + 1)]
    rows = np.array(sorted(set(rows)), np.int32)
    O_ref, lse_ref = orc.verify_attn(lay["Q"], lay["Kc"], lay["Vc"], kv, L, rows=rows)
    check_attn(O, lse, O_ref, lse_ref, L, rows=[tuple(r) for r in rows])


def test_attn_kv_overflow_sets_status_and_skips():
    B, K, Hq, Hkv, d, S = 2, 4, 4, 2, 64, 32
    Q, Kc, Vc = _inputs(B, K, Hq, Hkv, d, None, S, seed=2)
    ws = lr.Workspace(B, K, 1, Hq, Hkv, d, S, device=cuda())
    O = torch.zeros_like(Q)
    lr.libraspec_verify_attn(Q, Kc, Vc, torch.tensor([30, 5], dtype=torch.int32, device=cuda()),
                             torch.tensor([4, 4], dtype=torch.int32, device=cuda()), ws, O=O)
    assert lr.libraspec_get_status(ws) & lr.ST_KV_OVERFLOW
    assert torch.all(O[0] == 0) and torch.any(O[1] != 0)


def test_attn_deterministic():
    B, K, Hq, Hkv, d = 3, 16, 32, 8, 128
    kv = [9000, 300, 4000]
    L = [16, 2, 9]
    Q, Kc, Vc = _inputs(B, K, Hq, Hkv, d, kv, 9100, seed=11)
    outs = [_run(Q, Kc, Vc, kv, L, K) for _ in range(3)]
    for b in range(B):
        rows = slice(0, L[b] + 1)   # rows beyond L_b are never written
        for O, lse in outs[1:]:
            assert torch.equal(O[b, rows], outs[0][0][b, rows])
            assert torch.equal(lse[b, rows], outs[0][1][b, rows])


@pytest.mark.parametrize("B,kv_hi,d,seed", [(300, 200, 64, 1), (40, 9000, 128, 2), (129, 64, 128, 3),
                                             (1500, 40, 128, 4)])
def test_attn_many_sequences_stream_k_ranges(orc, B, kv_hi, d, seed):
    """Many ragged sequences: CTA tile ranges start and end inside row groups,
    one CTA covers several whole groups, and groups spread over many CTAs.
    B = 1500 is past the 1024 sequences whose lengths the kernel keeps in
    shared memory for its plan: that batch plans from global memory."""
    rng = np.random.default_rng(seed)
    K, Hq, Hkv = 12, 16, 4
    kv = rng.integers(0, kv_hi + 1, size=B).astype(np.int32)
    L = rng.integers(0, K + 1, size=B).astype(np.int32)
    S_cap = int((kv + L).max()) + 1
    Q, Kc, Vc = _inputs(B, K, Hq, Hkv, d, kv, S_cap, seed=seed * 101)
    rows = np.array([(b, h, t) for b in range(B) for h in (0, Hq - 1) for t in {0, int(L[b])}], np.int32)
    O_ref, lse_ref = orc.verify_attn(Q, Kc, Vc, kv, L, rows=rows)
    for _ in range(4):  # repeated: warps of one item race on shared memory if unsynchronised
        O, lse = _run(Q, Kc, Vc, kv.tolist(), L.tolist(), K)
        check_attn(O, lse, O_ref, lse_ref, L, rows=[tuple(r) for r in rows])


@pytest.mark.parametrize("name,n_layers,L_max", [("8b", 4, None), ("sampling", 3, None), ("tiny", 3, None),
                                                 ("8b", 3, 4)])
def test_attn_layer_chain_matches_per_layer_oracle(orc, name, n_layers, L_max):
    """libraspec_verify_attn_layers: all layers in one persistent launch; each
    layer's split groups are merged after the grid barrier that ends it."""
    w = workloads.WORKLOADS[name]
    kv = workloads.kv_lengths(w)
    rng = np.random.default_rng(7)
    L = rng.integers(0, (L_max if L_max is not None else w.K) + 1, size=w.B).astype(np.int32)
    layers = [workloads.layer(w, l, kv, device=cuda()) for l in range(n_layers)]
    S = layers[0]["Kc"].shape[2]
    ws = lr.Workspace(w.B, w.K, 1, w.Hq, w.Hkv, w.d, S, device=cuda())
    outs, lses = lr.libraspec_verify_attn_layers(layers, torch.tensor(kv, device=cuda()),
                                                 torch.tensor(L, device=cuda()), ws, want_lse=True)
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) == 0
    rows = np.array([(b, h, t) for b in range(w.B) for h in (0, w.Hq - 1) for t in {0, int(L[b])}], np.int32)
    for l in range(n_layers):
        O_ref, lse_ref = orc.verify_attn(layers[l]["Q"], layers[l]["Kc"], layers[l]["Vc"], kv, L, rows=rows)
        check_attn(outs[l], lses[l], O_ref, lse_ref, L, rows=[tuple(r) for r in rows])
    # the chain equals one layer at a time
    for l in range(n_layers):
        O1, lse1 = _run(layers[l]["Q"], layers[l]["Kc"], layers[l]["Vc"], kv.tolist(), L.tolist(), w.K)
        for b in range(w.B):
            assert torch.equal(O1[b, : L[b] + 1], outs[l][b, : L[b] + 1])
