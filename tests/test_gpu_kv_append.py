"""GPU: appending the verified block's keys and values to dense and paged
caches (libraspec_kv_append[_paged]) against torch slicing, and the staged
host API that uses it."""
import numpy as np
import pytest
import torch

from helpers import cuda
from paper_2608_08721_gb300 import api
from paper_2608_08721_gb300 import binding as lr
from paper_2608_08721_gb300 import workloads

pytestmark = pytest.mark.gpu


def _bf(shape, g):
    return torch.randn(shape, generator=g, device=cuda()).to(torch.bfloat16)


@pytest.mark.parametrize("d,Hkv", [(128, 8), (64, 2)])
def test_kv_append_dense(d, Hkv):
    g = torch.Generator(device="cuda").manual_seed(d)
    n_layers, B, T, S = 3, 5, 17, 320
    kv = np.array([0, 63, 100, 303, 250], np.int32)     # 303 + 17 = 320: the last row fits exactly
    caches = [{"Kc": _bf((B, Hkv, S, d), g), "Vc": _bf((B, Hkv, S, d), g)} for _ in range(n_layers)]
    ref = [{k: v.clone() for k, v in c.items()} for c in caches]
    kv_new = _bf((n_layers, 2, B, Hkv, T, d), g)
    ws = lr.Workspace(B, 16, 1, Hkv, Hkv, d, S, device=cuda())
    lr.libraspec_kv_append(kv_new, caches, torch.from_numpy(kv).to(cuda()), ws)
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) == 0
    for l in range(n_layers):
        for b in range(B):
            ref[l]["Kc"][b, :, kv[b]:kv[b] + T] = kv_new[l, 0, b]
            ref[l]["Vc"][b, :, kv[b]:kv[b] + T] = kv_new[l, 1, b]
        assert torch.equal(caches[l]["Kc"], ref[l]["Kc"]) and torch.equal(caches[l]["Vc"], ref[l]["Vc"])


def test_kv_append_overflow_sets_status_and_skips_rows():
    g = torch.Generator(device="cuda").manual_seed(1)
    B, Hkv, T, S, d = 2, 2, 5, 64, 64
    kv = np.array([62, 10], np.int32)  # rows 62..66 of sequence 0: 64..66 do not fit
    caches = [{"Kc": _bf((B, Hkv, S, d), g), "Vc": _bf((B, Hkv, S, d), g)}]
    before = caches[0]["Kc"].clone()
    kv_new = _bf((1, 2, B, Hkv, T, d), g)
    ws = lr.Workspace(B, 4, 1, Hkv, Hkv, d, S, device=cuda())
    lr.libraspec_kv_append(kv_new, caches, torch.from_numpy(kv).to(cuda()), ws)
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) & lr.ST_KV_OVERFLOW
    assert torch.equal(caches[0]["Kc"][0, :, 62:64], kv_new[0, 0, 0, :, :2])
    assert torch.equal(caches[0]["Kc"][0, :, :62], before[0, :, :62])
    assert torch.equal(caches[0]["Kc"][1, :, 10:15], kv_new[0, 0, 1])


@pytest.mark.parametrize("P", [64, 256])
def test_kv_append_paged_matches_dense(P):
    g = torch.Generator(device="cuda").manual_seed(P)
    n_layers, B, Hkv, T, d = 2, 4, 8, 33, 128
    kv = np.array([0, 200, 511 - 33, 64], np.int32)
    max_pages = 512 // P
    n_pages = B * max_pages + 3
    perm = np.random.default_rng(P).permutation(n_pages)[: B * max_pages].reshape(B, max_pages).astype(np.int32)
    pools = [{"Kp": _bf((n_pages, Hkv, P, d), g), "Vp": _bf((n_pages, Hkv, P, d), g)} for _ in range(n_layers)]
    dense = []
    for c in pools:   # the dense caches the pages describe
        dense.append({k2: torch.stack([torch.cat([c[k1][perm[b, j]] for j in range(max_pages)], dim=1)
                                       for b in range(B)]) for k1, k2 in (("Kp", "Kc"), ("Vp", "Vc"))})
    kv_new = _bf((n_layers, 2, B, Hkv, T, d), g)
    kv_t = torch.from_numpy(kv).to(cuda())
    ws = lr.Workspace(B, 32, 1, Hkv, Hkv, d, 512, device=cuda())
    lr.libraspec_kv_append(kv_new, dense, kv_t, ws)
    lr.libraspec_kv_append(kv_new, pools, kv_t, ws, block_table=torch.from_numpy(perm).to(cuda()))
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) == 0
    for l in range(n_layers):
        for b in range(B):
            for j in range(max_pages):
                assert torch.equal(pools[l]["Kp"][perm[b, j]], dense[l]["Kc"][b, :, j * P:(j + 1) * P])
                assert torch.equal(pools[l]["Vp"][perm[b, j]], dense[l]["Vc"][b, :, j * P:(j + 1) * P])


@pytest.mark.parametrize("in_place", [True, False])
def test_staged_round_appends_and_matches_device_round(in_place):
    """run_staged: the block rows land in the caches, and the round's outputs
    equal run_device on the same (already appended) inputs; the kernels read
    the pinned inputs in place, or the parts are copied to the device."""
    w = workloads.WORKLOADS["tiny"]
    kv = workloads.kv_lengths(w)
    lay = workloads.layer(w, 0, kv, device=cuda())
    inp = workloads.logits(w)
    K1 = w.K + 1
    caches = [{"Kc": lay["Kc"].clone(), "Vc": lay["Vc"].clone()}]
    runner = api.VerifyRound(w.B, w.K, w.V, w.Hq, w.Hkv, w.d, lay["Kc"].shape[2], caches, torch.tensor(kv),
                             inputs_in_place=in_place)
    h = runner.host_inputs()
    for name in ("draft_logits", "target_logits", "draft_tokens", "temperature"):
        h[name].copy_(inp[name])
    h["cost_table"].copy_(torch.tensor(workloads.cost_table(w)))
    h["Q"][0].copy_(lay["Q"].cpu())
    g = torch.Generator().manual_seed(3)
    new = torch.randn((2, w.B, w.Hkv, K1, w.d), generator=g).to(torch.bfloat16)
    h["kv_new"][0].copy_(new)
    n, bonus = runner.run_staged(seed=w.philox_seed)
    kvb = int(kv[0])
    assert torch.equal(caches[0]["Kc"][:, :, kvb:kvb + K1].cpu(), new[0])
    assert torch.equal(caches[0]["Vc"][:, :, kvb:kvb + K1].cpu(), new[1])
    O_staged = runner.out.O[0].clone()
    n2, b2 = n.copy(), bonus.copy()
    runner.run_device(seed=w.philox_seed)
    torch.cuda.synchronize()
    assert torch.equal(runner.out.O[0], O_staged)
    np.testing.assert_array_equal(runner.out.n_accepted.cpu().numpy(), n2)
    np.testing.assert_array_equal(runner.out.bonus_token.cpu().numpy(), b2)
    assert runner.h2d_bytes() >= h["draft_logits"].numel() * 4 + h["target_logits"].numel() * 4
    if in_place:  # given the round's lengths, only the verified target rows count
        L = runner.out.L.cpu().numpy()
        assert runner.h2d_bytes(L) == runner.h2d_bytes() - (w.K - int(L.sum())) * w.V * 4 * w.B


def test_staged_round_bf16_logits_matches_device_round():
    w = workloads.WORKLOADS["tiny"]
    kv = workloads.kv_lengths(w)
    lay = workloads.layer(w, 0, kv, device=cuda())
    inp = workloads.logits(w)
    caches = [{"Kc": lay["Kc"].clone(), "Vc": lay["Vc"].clone()}]
    runner = api.VerifyRound(w.B, w.K, w.V, w.Hq, w.Hkv, w.d, lay["Kc"].shape[2], caches, torch.tensor(kv),
                             logits_dtype=torch.bfloat16)
    h = runner.host_inputs()
    h["draft_logits"].copy_(inp["draft_logits"].to(torch.bfloat16))
    h["target_logits"].copy_(inp["target_logits"].to(torch.bfloat16))
    for name in ("draft_tokens", "temperature"):
        h[name].copy_(inp[name])
    h["cost_table"].copy_(torch.tensor(workloads.cost_table(w)))
    h["Q"][0].copy_(lay["Q"].cpu())
    K1 = w.K + 1
    kvb = int(kv[0])
    h["kv_new"][0, 0].copy_(lay["Kc"][:, :, kvb:kvb + K1].cpu())
    h["kv_new"][0, 1].copy_(lay["Vc"][:, :, kvb:kvb + K1].cpu())
    n, bonus = runner.run_staged(seed=w.philox_seed, round_offset=2)
    O = runner.out.O[0].clone()
    runner.run_device(seed=w.philox_seed, round_offset=2)
    torch.cuda.synchronize()
    assert torch.equal(runner.out.O[0], O)
    np.testing.assert_array_equal(runner.out.n_accepted.cpu().numpy(), n)
    np.testing.assert_array_equal(runner.out.bonus_token.cpu().numpy(), bonus)
    assert lr.libraspec_get_status(runner.ws) == 0


def test_staged_round_graph_replays_follow_seed_and_round():
    """From the second call on, a staged round replays a captured graph; the
    generator's arguments come from the host buffer, so every round's draws
    still follow its own seed and round offset (compared with the eager
    device round)."""
    w = workloads.WORKLOADS["tiny"].scaled(B=8, temperature=("const", 1.0))
    kv = workloads.kv_lengths(w)
    lay = workloads.layer(w, 0, kv, device=cuda())
    inp = workloads.logits(w)
    caches = [{"Kc": lay["Kc"].clone(), "Vc": lay["Vc"].clone()}]
    runner = api.VerifyRound(w.B, w.K, w.V, w.Hq, w.Hkv, w.d, lay["Kc"].shape[2], caches, torch.tensor(kv))
    h = runner.host_inputs()
    for name in ("draft_logits", "target_logits", "draft_tokens", "temperature"):
        h[name].copy_(inp[name])
    h["cost_table"].copy_(torch.tensor(workloads.cost_table(w)))
    h["Q"][0].copy_(lay["Q"].cpu())
    K1 = w.K + 1
    for b in range(w.B):
        kvb = int(kv[b])
        h["kv_new"][0, 0, b].copy_(lay["Kc"][b, :, kvb:kvb + K1].cpu())
        h["kv_new"][0, 1, b].copy_(lay["Vc"][b, :, kvb:kvb + K1].cpu())
    seen = set()
    for r, (seed, ro) in enumerate([(5, 0), (5, 1), (5, 2), (9, 2), (5, 0)]):
        n, bonus = runner.run_staged(seed=seed, round_offset=ro, seq_offset=3)
        runner.run_device(seed=seed, round_offset=ro, seq_offset=3)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(runner.out.n_accepted.cpu().numpy(), n)
        np.testing.assert_array_equal(runner.out.bonus_token.cpu().numpy(), bonus)
        seen.add(tuple(bonus.tolist()))
    assert len(seen) >= 3   # different rounds draw differently
    assert lr.libraspec_get_status(runner.ws) == 0


def test_kv_append_empty_block_is_a_no_op():
    g = torch.Generator(device="cuda").manual_seed(4)
    caches = [{"Kc": _bf((2, 2, 64, 64), g), "Vc": _bf((2, 2, 64, 64), g)}]
    before = caches[0]["Kc"].clone()
    ws = lr.Workspace(2, 4, 1, 2, 2, 64, 64, device=cuda())
    lr.libraspec_kv_append(torch.empty((1, 2, 2, 2, 0, 64), dtype=torch.bfloat16, device=cuda()), caches,
                           torch.tensor([3, 9], dtype=torch.int32, device=cuda()), ws)
    torch.cuda.synchronize()
    assert torch.equal(caches[0]["Kc"], before) and lr.libraspec_get_status(ws) == 0
