"""GPU parity: verify attention over a paged KV cache (block tables) vs. the
oracle on the dense cache the pages describe, and bit-for-bit vs. the dense
kernel on that cache (same tiles, same arithmetic)."""
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

from helpers import check_attn, cuda
from paper_2608_08721_gb300 import binding as lr

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _paged_inputs(B, K, Hq, Hkv, d, kv, L, page_size, seed, n_layers=1, extra_pages=5):
    """Dense caches and the same caches in randomly permuted pages."""
    g = torch.Generator(device="cuda").manual_seed(seed)
    rng = np.random.default_rng(seed)
    S = max(k + l + 1 for k, l in zip(kv, L))
    max_pages = -(-S // page_size)
    n_pages = B * max_pages + extra_pages
    perm = rng.permutation(n_pages)[: B * max_pages].reshape(B, max_pages).astype(np.int32)
    table = torch.from_numpy(perm).to(cuda())
    layers, dense = [], []
    for _ in range(n_layers):
        Q = torch.randn((B, K + 1, Hq, d), generator=g, device=cuda()).to(torch.bfloat16)
        Kd = (torch.randn((B, Hkv, max_pages * page_size, d), generator=g, device=cuda()) * 2.0).to(torch.bfloat16)
        Vd = torch.randn((B, Hkv, max_pages * page_size, d), generator=g, device=cuda()).to(torch.bfloat16)
        Kp = torch.randn((n_pages, Hkv, page_size, d), generator=g, device=cuda()).to(torch.bfloat16)
        Vp = torch.randn((n_pages, Hkv, page_size, d), generator=g, device=cuda()).to(torch.bfloat16)
        for b in range(B):
            for j in range(max_pages):
                Kp[perm[b, j]] = Kd[b, :, j * page_size:(j + 1) * page_size]
                Vp[perm[b, j]] = Vd[b, :, j * page_size:(j + 1) * page_size]
        layers.append({"Q": Q, "Kp": Kp, "Vp": Vp})
        dense.append({"Q": Q, "Kc": Kd, "Vc": Vd})
    return layers, dense, table, max_pages * page_size


def _run_paged(layers, table, kv, L, K, S_cap):
    B, _, Hq, d = layers[0]["Q"].shape
    Hkv = layers[0]["Kp"].shape[1]
    ws = lr.Workspace(B, K, 1, Hq, Hkv, d, S_cap, device=cuda())
    kv_t = torch.tensor(kv, dtype=torch.int32, device=cuda())
    L_t = torch.tensor(L, dtype=torch.int32, device=cuda())
    outs, lses = lr.libraspec_verify_attn_paged_layers(layers, table, kv_t, L_t, ws, want_lse=True)
    torch.cuda.synchronize()
    return outs, lses, lr.libraspec_get_status(ws)


@pytest.mark.parametrize("page_size", [64, 128, 256])
@pytest.mark.parametrize("d,Hq,Hkv", [(128, 32, 8), (64, 8, 2), (128, 28, 4)])
def test_paged_matches_oracle_and_dense(orc, page_size, d, Hq, Hkv):
    K = 12
    kv = [0, 63, 64, 700, 3000, 129]
    L = [0, 12, 5, 1, 12, 7]
    B = len(kv)
    layers, dense, table, S_cap = _paged_inputs(B, K, Hq, Hkv, d, kv, L, page_size, seed=page_size + d + Hq)
    outs, lses, status = _run_paged(layers, table, kv, L, K, S_cap)
    assert status == 0
    O_ref, lse_ref = orc.verify_attn_paged(layers[0]["Q"], layers[0]["Kp"], layers[0]["Vp"], table.cpu().numpy(),
                                           np.array(kv), np.array(L))
    check_attn(outs[0], lses[0], O_ref, lse_ref, L)
    # the dense kernel on the cache the pages describe: same tiles, same arithmetic
    ws = lr.Workspace(B, K, 1, Hq, Hkv, d, S_cap, device=cuda())
    O_d, lse_d = lr.libraspec_verify_attn(dense[0]["Q"], dense[0]["Kc"], dense[0]["Vc"],
                                          torch.tensor(kv, dtype=torch.int32, device=cuda()),
                                          torch.tensor(L, dtype=torch.int32, device=cuda()), ws, want_lse=True)
    torch.cuda.synchronize()
    for b in range(B):
        assert torch.equal(outs[0][b, : L[b] + 1], O_d[b, : L[b] + 1])
        assert torch.equal(lses[0][b, : L[b] + 1], lse_d[b, : L[b] + 1])


def test_paged_layer_chain_long_cache(orc):
    """Three layers in one launch; a long sequence split over many CTAs."""
    K, Hq, Hkv, d, P = 16, 32, 8, 128, 128
    kv, L = [20000, 300], [9, 16]
    layers, dense, table, S_cap = _paged_inputs(2, K, Hq, Hkv, d, kv, L, P, seed=5, n_layers=3)
    outs, lses, status = _run_paged(layers, table, kv, L, K, S_cap)
    assert status == 0
    rows = np.array([(b, h, t) for b in range(2) for h in (0, 13, Hq - 1) for t in {0, L[b] // 2, L[b]}], np.int32)
    for l in range(3):
        O_ref, lse_ref = orc.verify_attn_paged(layers[l]["Q"], layers[l]["Kp"], layers[l]["Vp"], table.cpu().numpy(),
                                               np.array(kv), np.array(L), rows=rows)
        check_attn(outs[l], lses[l], O_ref, lse_ref, L, rows=[tuple(r) for r in rows])


def test_paged_bad_page_sets_status():
    K, Hq, Hkv, d, P = 4, 8, 2, 64, 64
    kv, L = [100, 10], [2, 3]
    layers, _, table, S_cap = _paged_inputs(2, K, Hq, Hkv, d, kv, L, P, seed=3)
    table[0, 1] = layers[0]["Kp"].shape[0] + 7  # outside the pool
    _, _, status = _run_paged(layers, table, kv, L, K, S_cap)
    assert status & 0x40  # LIBRASPEC_ST_BAD_PAGE


def test_paged_rejects_unsupported_page_size():
    B, K, Hq, Hkv, d = 1, 4, 8, 2, 64
    Q = torch.zeros((B, K + 1, Hq, d), dtype=torch.bfloat16, device=cuda())
    Kp = torch.zeros((4, Hkv, 48, d), dtype=torch.bfloat16, device=cuda())
    table = torch.zeros((B, 4), dtype=torch.int32, device=cuda())
    ws = lr.Workspace(B, K, 1, Hq, Hkv, d, 4 * 48, device=cuda())
    with pytest.raises(lr.LibraspecError):
        lr.libraspec_verify_attn_paged_layers([{"Q": Q, "Kp": Kp, "Vp": Kp}], table,
                                              torch.zeros(B, dtype=torch.int32, device=cuda()),
                                              torch.zeros(B, dtype=torch.int32, device=cuda()), ws)


def test_paged_uncached_block_table_path():
    """With the page-id cache switched off (LIBRASPEC_ATTN_PAGE_CACHE=0, read
    once per process) every tile reads the block table: same result."""
    code = r'''
import sys, numpy as np, torch
sys.path.insert(0, %r)
sys.path.insert(0, %r)
from test_gpu_attn_paged import _paged_inputs, _run_paged
kv, L = [5000, 64, 0], [7, 3, 12]
layers, dense, table, S = _paged_inputs(3, 12, 32, 8, 128, kv, L, 64, seed=11)
outs, lses, status = _run_paged(layers, table, kv, L, 12, S)
np.save(sys.argv[1], outs[0].float().cpu().numpy())
print("status", status)
''' % (ROOT, os.path.join(ROOT, "tests"))
    import tempfile
    with tempfile.TemporaryDirectory() as td:
        res = {}
        for cache in ("0", "4096"):
            path = os.path.join(td, "o_%s.npy" % cache)
            env = dict(os.environ, LIBRASPEC_ATTN_PAGE_CACHE=cache)
            out = subprocess.run([sys.executable, "-c", code, path], env=env, capture_output=True, text=True,
                                 timeout=600)
            assert out.returncode == 0, out.stderr[-2000:]
            assert "status 0" in out.stdout
            res[cache] = np.load(path)
        np.testing.assert_array_equal(res["0"], res["4096"])


def test_paged_cost_weighted_split(orc):
    """More (sequence, kv head) pairs than CTAs: the launch takes the kernel
    whose Stream-K ranges are cut by cost (tiles plus each item's fixed
    cost). Paged against the oracle and bit for bit against the dense kernel
    (the same split, tiles and arithmetic)."""
    K, Hq, Hkv, d, P = 12, 32, 8, 128, 128
    rng = np.random.default_rng(21)
    B = 40  # 320 (sequence, kv head) pairs
    kv = rng.integers(0, 1500, size=B).tolist()
    L = rng.integers(0, K + 1, size=B).tolist()
    layers, dense, table, S_cap = _paged_inputs(B, K, Hq, Hkv, d, kv, L, P, seed=21, n_layers=2)
    outs, lses, status = _run_paged(layers, table, kv, L, K, S_cap)
    assert status == 0
    for l in range(2):
        O_ref, lse_ref = orc.verify_attn_paged(layers[l]["Q"], layers[l]["Kp"], layers[l]["Vp"],
                                               table.cpu().numpy(), np.array(kv), np.array(L))
        check_attn(outs[l], lses[l], O_ref, lse_ref, L)
    ws = lr.Workspace(B, K, 1, Hq, Hkv, d, S_cap, device=cuda())
    O_d, lse_d = lr.libraspec_verify_attn_layers(dense, torch.tensor(kv, dtype=torch.int32, device=cuda()),
                                                 torch.tensor(L, dtype=torch.int32, device=cuda()), ws,
                                                 want_lse=True)
    torch.cuda.synchronize()
    for l in range(2):
        for b in range(B):
            assert torch.equal(outs[l][b, : L[b] + 1], O_d[l][b, : L[b] + 1])
            assert torch.equal(lses[l][b, : L[b] + 1], lse_d[l][b, : L[b] + 1])
