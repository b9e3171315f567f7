"""Pins of the oracle's block-causal GQA verify attention.

Pinned against torch's scaled_dot_product_attention run in float64 on the CPU
(an independent library routine) with an explicit per-row mask, and against
closed forms: equal keys give the mean of the visible values, a dominant key
gives its value row, a single visible key gives its value exactly, and equal
scores give lse = s + ln(n_keys). The paged-cache gather is pinned against
caches scattered into permuted pages by numpy indexing.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_08721_gb300 import workloads


def _bf16(shape, rng, scale=1.0):
    return torch.from_numpy((rng.standard_normal(shape) * scale).astype(np.float32)).to(torch.bfloat16)


def _sdpa_reference(Q, Kc, Vc, kv_len, L, scale):
    B, K1, Hq, d = Q.shape
    Hkv = Kc.shape[1]
    g = Hq // Hkv
    O = np.full((B, K1, Hq, d), np.nan)
    for b in range(B):
        n_all = int(kv_len[b]) + int(L[b]) + 1
        for h in range(Hq):
            q = Q[b, : L[b] + 1, h].double()[None, None]             # [1,1,T,d]
            k = Kc[b, h // g, :n_all].double()[None, None]
            v = Vc[b, h // g, :n_all].double()[None, None]
            t = torch.arange(L[b] + 1)[:, None]
            s = torch.arange(n_all)[None, :]
            mask = s <= (int(kv_len[b]) + t)
            out = torch.nn.functional.scaled_dot_product_attention(q, k, v, attn_mask=mask, scale=scale)
            O[b, : L[b] + 1, h] = out[0, 0].numpy()
    return O


@pytest.mark.parametrize("Hq,Hkv,d", [(4, 2, 16), (6, 2, 8), (8, 8, 32), (7, 1, 16)])
def test_attn_matches_torch_sdpa_fp64(orc, Hq, Hkv, d):
    rng = np.random.default_rng(Hq * 100 + d)
    B, K = 3, 5
    kv_len = np.array([0, 7, 33], np.int32)
    L = np.array([2, 0, 5], np.int32)
    S = 48
    Q = _bf16((B, K + 1, Hq, d), rng)
    Kc = _bf16((B, Hkv, S, d), rng, 2.0)
    Vc = _bf16((B, Hkv, S, d), rng)
    scale = 1.0 / np.sqrt(d)
    O, lse = orc.verify_attn(Q, Kc, Vc, kv_len, L, scale)
    ref = _sdpa_reference(Q, Kc, Vc, kv_len, L, scale)
    np.testing.assert_allclose(O, ref, rtol=1e-11, atol=1e-12, equal_nan=True)
    # rows beyond L_b are left untouched
    for b in range(B):
        assert np.all(np.isnan(O[b, L[b] + 1:]))
        assert np.all(np.isfinite(lse[b, : L[b] + 1]))


def test_attn_equal_keys_give_mean_of_values(orc):
    rng = np.random.default_rng(2)
    B, K, Hq, Hkv, d, S = 1, 3, 2, 1, 8, 16
    kv_len = np.array([9], np.int32)
    L = np.array([3], np.int32)
    Q = _bf16((B, K + 1, Hq, d), rng)
    Kc = torch.ones((B, Hkv, S, d), dtype=torch.bfloat16) * 0.5
    Vc = _bf16((B, Hkv, S, d), rng)
    O, lse = orc.verify_attn(Q, Kc, Vc, kv_len, L, 0.25)
    for t in range(L[0] + 1):
        n = kv_len[0] + t + 1
        mean = Vc[0, 0, :n].double().mean(0).numpy()
        for h in range(Hq):
            np.testing.assert_allclose(O[0, t, h], mean, rtol=1e-13, atol=1e-14)
            s = 0.25 * 0.5 * Q[0, t, h].double().sum().item()
            assert lse[0, t, h] == pytest.approx(s + np.log(n), rel=1e-13, abs=1e-13)


def test_attn_dominant_key_selects_its_value(orc):
    rng = np.random.default_rng(3)
    B, K, Hq, Hkv, d, S = 1, 1, 1, 1, 16, 32
    kv_len = np.array([20], np.int32)
    L = np.array([1], np.int32)
    Q = torch.ones((B, K + 1, Hq, d), dtype=torch.bfloat16)
    Kc = _bf16((B, Hkv, S, d), rng, 0.01)
    Kc[0, 0, 11] = 8.0                      # score 8*16*scale = 128 over the rest
    Vc = _bf16((B, Hkv, S, d), rng)
    O, _ = orc.verify_attn(Q, Kc, Vc, kv_len, L, 1.0)
    for t in range(2):
        np.testing.assert_allclose(O[0, t, 0], Vc[0, 0, 11].double().numpy(), rtol=1e-12, atol=1e-12)


def test_attn_single_visible_key_is_exact(orc):
    rng = np.random.default_rng(4)
    B, K, Hq, Hkv, d, S = 2, 2, 4, 2, 8, 8
    kv_len = np.array([0, 0], np.int32)
    L = np.array([0, 0], np.int32)
    Q = _bf16((B, K + 1, Hq, d), rng)
    Kc = _bf16((B, Hkv, S, d), rng)
    Vc = _bf16((B, Hkv, S, d), rng)
    O, _ = orc.verify_attn(Q, Kc, Vc, kv_len, L)
    for b in range(B):
        for h in range(Hq):
            np.testing.assert_array_equal(O[b, 0, h], Vc[b, h // 2, 0].double().numpy())


def test_attn_causal_row_t_ignores_later_block_keys(orc):
    # changing key kv_len + 2 must not change rows t = 0, 1
    rng = np.random.default_rng(5)
    B, K, Hq, Hkv, d, S = 1, 4, 2, 1, 8, 24
    kv_len = np.array([10], np.int32)
    L = np.array([4], np.int32)
    Q = _bf16((B, K + 1, Hq, d), rng)
    Kc = _bf16((B, Hkv, S, d), rng)
    Vc = _bf16((B, Hkv, S, d), rng)
    O1, _ = orc.verify_attn(Q, Kc, Vc, kv_len, L)
    Kc2, Vc2 = Kc.clone(), Vc.clone()
    Kc2[0, 0, 12] = 5.0
    Vc2[0, 0, 12] = -3.0
    O2, _ = orc.verify_attn(Q, Kc2, Vc2, kv_len, L)
    np.testing.assert_array_equal(O1[0, :2], O2[0, :2])
    assert np.max(np.abs(O1[0, 2:] - O2[0, 2:])) > 1e-3


def test_attn_row_subset_matches_full(orc):
    w = workloads.WORKLOADS["tiny"].scaled(kv=("const", 40))
    kv = workloads.kv_lengths(w)
    lay = workloads.layer(w, 0, kv)
    L = np.array([5], np.int32)
    O, lse = orc.verify_attn(lay["Q"], lay["Kc"], lay["Vc"], kv, L)
    rows = np.array([[0, 3, 2], [0, 7, 5], [0, 0, 0]], np.int32)
    Os, lses = orc.verify_attn(lay["Q"], lay["Kc"], lay["Vc"], kv, L, rows=rows)
    for b, h, t in rows:
        np.testing.assert_array_equal(Os[b, t, h], O[b, t, h])
        assert lses[b, t, h] == lse[b, t, h]


def test_attn_rejects_cache_overflow(orc):
    Q = torch.zeros((1, 3, 2, 8), dtype=torch.bfloat16)
    Kc = torch.zeros((1, 1, 10, 8), dtype=torch.bfloat16)
    with pytest.raises(orc.OracleError):
        orc.verify_attn(Q, Kc, Kc, np.array([8], np.int32), np.array([2], np.int32))
    with pytest.raises(orc.OracleError):
        orc.verify_attn(Q, Kc, Kc, np.array([1], np.int32), np.array([3], np.int32))


# ---- paged caches (the dense cache a block table describes) ----
def _scatter_to_pages(dense, page_size, rng, extra_pages=3):
    """Pool and block table holding `dense` [B,Hkv,S,d] in randomly permuted pages."""
    B, Hkv, S, d = dense.shape
    max_pages = -(-S // page_size)
    n_pages = B * max_pages + extra_pages
    perm = rng.permutation(n_pages)[: B * max_pages].reshape(B, max_pages).astype(np.int32)
    pool = rng.integers(0, 2**16, size=(n_pages, Hkv, page_size, d)).astype(np.uint16)
    for b in range(B):
        for j in range(max_pages):
            s0, s1 = j * page_size, min(S, (j + 1) * page_size)
            pool[perm[b, j], :, : s1 - s0] = dense[b, :, s0:s1]
    return pool, perm


@pytest.mark.parametrize("page_size", [1, 7, 64, 128])
def test_gather_pages_recovers_the_dense_cache(page_size):
    rng = np.random.default_rng(page_size)
    dense = rng.integers(0, 2**16, size=(3, 2, 300, 16)).astype(np.uint16)
    pool, table = _scatter_to_pages(dense, page_size, rng)
    np.testing.assert_array_equal(oracle.gather_pages(pool, table, 300), dense)
    np.testing.assert_array_equal(oracle.gather_pages(pool, table, 17), dense[:, :, :17])


def test_gather_pages_identity_table_is_a_reshape():
    rng = np.random.default_rng(9)
    B, Hkv, P, d, n = 2, 3, 64, 8, 4
    pool = rng.integers(0, 2**16, size=(B * n, Hkv, P, d)).astype(np.uint16)
    table = np.arange(B * n, dtype=np.int32).reshape(B, n)
    expect = pool.reshape(B, n, Hkv, P, d).transpose(0, 2, 1, 3, 4).reshape(B, Hkv, n * P, d)
    np.testing.assert_array_equal(oracle.gather_pages(pool, table, n * P), expect)


def test_gather_pages_rejects_bad_entries():
    pool = np.zeros((4, 1, 64, 8), np.uint16)
    for bad in (-1, 4):
        table = np.array([[0, bad]], np.int32)
        with pytest.raises(oracle.OracleError):
            oracle.gather_pages(pool, table, 100)
    # an entry no key reads is not looked at
    oracle.gather_pages(pool, np.array([[0, 99]], np.int32), 64)
