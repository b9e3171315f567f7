"""The seeded input generators: they produce the recipe the benchmarks and the
parity tests state (shapes, value distributions, length mixes, tree
structure), and the same tensors for the same seed (no GPU)."""
import math

import numpy as np
import pytest
import torch

from paper_2608_08721_gb300 import workloads as wl

# (B, K, V, Hq, Hkv, d, layers) of the five workloads
RECIPE = {
    "tiny": (1, 16, 32000, 8, 2, 64, 1),
    "8b": (1, 16, 128256, 32, 8, 128, 32),
    "sampling": (16, 16, 152064, 28, 4, 128, 1),
    "ragged": (64, 32, 128256, 32, 8, 128, 1),
    "70b": (8, 16, 128256, 64, 8, 128, 80),
}


@pytest.mark.parametrize("name", sorted(RECIPE))
def test_shapes_are_the_stated_ones(name):
    w = wl.WORKLOADS[name]
    assert (w.B, w.K, w.V, w.Hq, w.Hkv, w.d, w.n_layers) == RECIPE[name]
    assert w.Hq % w.Hkv == 0


def test_kv_length_mixes():
    assert (wl.kv_lengths(wl.WORKLOADS["8b"]) == 4096).all()
    assert (wl.kv_lengths(wl.WORKLOADS["70b"]) == 131072).all()
    s = wl.kv_lengths(wl.WORKLOADS["sampling"])
    assert s.dtype == np.int32 and s.min() >= 1024 and s.max() <= 8192 and len(set(s.tolist())) > 8
    r = wl.kv_lengths(wl.WORKLOADS["ragged"])
    assert r.min() >= 512 and r.max() <= 32768
    # log-uniform on [512, 32768]: log2 lengths spread evenly over [9, 15]; half lie below 4096
    lg = np.log2(r)
    assert 0.3 < np.mean(lg < 12) < 0.7
    assert np.histogram(lg, bins=3, range=(9, 15))[0].min() >= 10
    np.testing.assert_array_equal(r, wl.kv_lengths(wl.WORKLOADS["ragged"]))   # seeded


def test_temperatures_and_modes():
    assert (wl.temperatures(wl.WORKLOADS["8b"]) == 0).all()
    assert (wl.temperatures(wl.WORKLOADS["sampling"]) == 1).all()
    assert (wl.temperatures(wl.WORKLOADS["70b"]) == np.float32(0.7)).all()
    t = wl.temperatures(wl.WORKLOADS["ragged"])
    assert (t[0::2] == 0).all() and (t[1::2] == np.float32(0.8)).all()


def test_cache_capacity_and_attention_bytes():
    w = wl.WORKLOADS["sampling"]
    kv = wl.kv_lengths(w)
    S = wl.s_cap(w, kv)
    assert S % 64 == 0 and S >= kv.max() + w.K + 1 and S - 64 < kv.max() + w.K + 1
    # one sequence by hand: K and V of kv+L+1 keys per kv head, Q in and O out for L+1 rows
    w1 = wl.WORKLOADS["tiny"]
    assert wl.attn_bytes(w1, np.array([512]), 3) == 2 * 516 * 64 * 4 + 4 * 8 * 64 * 4


@pytest.mark.parametrize("name", sorted(RECIPE))
def test_cost_tables_are_positive_and_non_decreasing(name):
    w = wl.WORKLOADS[name]
    t = wl.cost_table(w)
    assert t.shape == (w.K + 1,) and t.dtype == np.float32
    assert (t > 0).all() and (np.diff(t) >= 0).all()
    assert t[0] == np.float32(1.0)


def test_tiny_logit_distributions_and_greedy_drafts():
    w = wl.WORKLOADS["tiny"]
    a = wl.logits(w)
    tgt, drf, tok = a["target_logits"], a["draft_logits"], a["draft_tokens"]
    assert tgt.shape == (1, 17, 32000) and drf.shape == (1, 16, 32000) and tok.dtype == torch.int32
    assert abs(tgt.std().item() / 4.0 - 1) < 0.02              # target N(0, 4^2)
    assert abs((drf - tgt[:, :16]).std().item() - 1.0) < 0.02  # drafter = target + N(0, 1)
    assert abs(tgt.mean().item()) < 0.05
    torch.testing.assert_close(tok[0], drf[0].argmax(-1).to(torch.int32))
    b = wl.logits(w)
    assert torch.equal(a["target_logits"], b["target_logits"]) and torch.equal(tok, b["draft_tokens"])


def test_peaked_target_rows():
    """normal_peak: every row carries +peak at one index (8b: N(0, 6^2) + 12)."""
    w = wl.WORKLOADS["8b"].scaled(V=4096, data_seed=11)
    a = wl.logits(w)
    tgt = a["target_logits"].double()
    assert abs(tgt.std().item() / 6.0 - 1) < 0.03
    # the planted value shifts each row's sum by the peak: the mean over 17 rows of 4096 values
    # is 12 / 4096 above zero, far below the noise; check the shift exactly by regenerating
    # the unpeaked rows from the same generator stream
    g = torch.Generator().manual_seed(w.data_seed * 1000003 + 17)
    base = torch.randn((1, 17, 4096), generator=g) * 6.0
    diff = (a["target_logits"] - base)
    assert torch.count_nonzero(diff.abs() > 1e-3, dim=-1).eq(1).all()
    assert torch.allclose(diff.sum(-1), torch.full((1, 17), 12.0), atol=1e-3)


def test_sampled_drafts_follow_the_drafter_at_its_temperature():
    """Sampling sequences draft x ~ softmax(drafter / T): over many rows the
    mean of q(x) is the mean of sum_v q_v^2 (the expected probability of a
    draw), within CLT error; drawing at T = 1 instead of 0.5 would not be."""
    w = wl.WORKLOADS["tiny"].scaled(B=4, K=1000, V=6, temperature=("const", 0.5), data_seed=5)
    a = wl.logits(w)
    q = torch.softmax(a["draft_logits"].double() / 0.5, dim=-1)
    qx = torch.gather(q, 2, a["draft_tokens"].long()[..., None])[..., 0]
    want = (q * q).sum(-1)
    n = qx.numel()
    sd = (qx - want).std().item()
    assert abs(qx.mean().item() - want.mean().item()) < 4 * sd / math.sqrt(n)
    q1 = torch.softmax(a["draft_logits"].double(), dim=-1)
    g = torch.Generator().manual_seed(0)
    wrong = torch.gather(q, 2, torch.multinomial(q1.view(-1, 6), 1, generator=g).view(4, 1000, 1))[..., 0]
    assert abs(wrong.mean().item() - want.mean().item()) > 4 * sd / math.sqrt(n)


def test_layers_are_seeded_per_layer():
    w = wl.WORKLOADS["tiny"]
    kv = wl.kv_lengths(w)
    l0, l0b, l1 = wl.layer(w, 0, kv), wl.layer(w, 0, kv), wl.layer(w, 1, kv)
    assert l0["Q"].shape == (1, 17, 8, 64) and l0["Kc"].shape == (1, 2, wl.s_cap(w, kv), 64)
    assert l0["Kc"].dtype == torch.bfloat16
    assert torch.equal(l0["Kc"], l0b["Kc"]) and not torch.equal(l0["Kc"], l1["Kc"])
    assert abs(l0["Kc"].float().std().item() - 1.0) < 0.02


def test_peaky_layer_plants_a_dominant_key():
    w = wl.WORKLOADS["tiny"]
    kv = wl.kv_lengths(w)
    lay = wl.layer(w, 0, kv, peaky=True)
    q = lay["Q"][0, 0].float()                  # [Hq, d]
    k = lay["Kc"][0].float()[:, :512]           # [Hkv, kv, d]
    for h in range(8):
        s = k[h // 4] @ q[h]
        assert s.max().item() > 2.5 * (q[h] @ q[h]).item()


@pytest.mark.parametrize("shape", ["chain", "star", "random", "topk", "ddtree"])
def test_draft_trees_are_topological(shape):
    B, K = 5, 64
    L = np.array([0, 1, 7, 40, 64])
    par = wl.draft_tree(B, K, L, seed=3, shape=shape)
    assert par.shape == (B, K + 1) and par.dtype == np.int32
    for b in range(B):
        assert par[b, 0] == 0 and (par[b, L[b] + 1:] == 0).all()
        for t in range(1, L[b] + 1):
            assert 0 <= par[b, t] < t
    np.testing.assert_array_equal(par, wl.draft_tree(B, K, L, seed=3, shape=shape))


def test_tree_tokens_are_distinct_among_siblings_and_the_peak_follows():
    w = wl.WORKLOADS["tiny"]
    par = wl.draft_tree(2, 48, 48, seed=1, shape="ddtree")
    t = wl.tree_logits(w, par, 48)
    tok = t["draft_tokens"].numpy()
    tgt = t["target_logits"]
    assert tgt.shape == (2, 49, w.V)
    # the planted +12 of each row, found against the same generator stream without it
    g = torch.Generator().manual_seed(w.data_seed * 7919 + 77)
    diff = tgt - torch.randn((2, 49, w.V), generator=g) * 4.0
    assert torch.count_nonzero(diff.abs() > 1e-3, dim=-1).eq(1).all()
    peak = diff.argmax(-1)
    follow = 0
    parents = 0
    for b in range(2):
        kids = {}
        for n in range(1, 49):
            kids.setdefault(int(par[b, n]), []).append(n)
        for p, ks in kids.items():
            assert len(set(tok[b, [k - 1 for k in ks]].tolist())) == len(ks)
            parents += 1
            follow += int(peak[b, p]) == int(tok[b, ks[0] - 1])
    assert 0.6 < follow / parents < 0.95        # p_follow = 0.8 over about 70 parents


def test_lm_head_scales():
    w = wl.WORKLOADS["tiny"].scaled(V=2000, hidden=256)
    h = wl.lm_head(w, 8)
    assert h["H"].shape == (8, 256) and h["W"].shape == (2000, 256) and h["W"].dtype == torch.bfloat16
    x = h["H"].float() @ h["W"].float().T
    assert abs(x.std().item() / 4.0 - 1) < 0.05   # logits ~ N(0, 4^2)
