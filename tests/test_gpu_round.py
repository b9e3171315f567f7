"""GPU parity of the whole round (libraspec_verify_round and the host-buffer API)."""
import numpy as np
import pytest
import torch

from helpers import assert_exact_unless_flagged, assert_flag_budget, check_attn, cuda
from paper_2608_08721_gb300 import api
from paper_2608_08721_gb300 import binding as lr
from paper_2608_08721_gb300 import workloads

pytestmark = pytest.mark.gpu


def _oracle_round(orc, w, inp, kv, layers, cost, L_gpu, rows=None):
    """The oracle's confidence and selection, and its acceptance and attention
    given the GPU's lengths (equal to the oracle's unless a flagged selection
    differs), so that every step is compared whatever the selection."""
    dl = inp["draft_logits"].float().cpu().numpy()
    q, _ = orc.confidence(dl, inp["draft_tokens"].cpu().numpy(), inp["temperature"].cpu().numpy())
    L, sflag = orc.select_lengths(q, cost.astype(np.float64))
    n, bonus, aflag = orc.accept(inp["target_logits"].float().cpu().numpy(), dl,
                                 inp["draft_tokens"].cpu().numpy(), L_gpu, inp["temperature"].cpu().numpy(),
                                 w.philox_seed)
    outs = [orc.verify_attn(lay["Q"], lay["Kc"], lay["Vc"], kv, L_gpu, rows=rows) for lay in layers]
    return q, L, sflag, n, bonus, aflag, outs


def _group_rows(w, L, seqs):
    """Every verified row of each listed sequence's first kv head (g heads x
    (L_b + 1) positions: the query rows one attention row group serves)."""
    g = w.Hq // w.Hkv
    return np.array([(b, h, t) for b in seqs for h in range(g) for t in range(int(L[b]) + 1)], np.int32)


@pytest.mark.parametrize("logits", ["f32", "bf16"])
@pytest.mark.parametrize("name,n_layers", [("tiny", 1), ("8b", 2), ("sampling", 1), ("ragged", 1)])
def test_verify_round_matches_oracle(orc, name, n_layers, logits):
    """libraspec_verify_round, and libraspec_verify_round_bf16 on the same
    logits rounded to bf16 (the oracle gets the rounded values). The ragged
    batch's attention is compared on complete row groups of four sequences."""
    w = workloads.WORKLOADS[name]
    kv = workloads.kv_lengths(w)
    inp = workloads.logits(w, device=cuda())
    if logits == "bf16":
        for k in ("draft_logits", "target_logits"):
            inp[k] = inp[k].to(torch.bfloat16)
    layers = [workloads.layer(w, l, kv, device=cuda()) for l in range(n_layers)]
    cost = workloads.cost_table(w)
    S = layers[0]["Kc"].shape[2]
    ws = lr.Workspace(w.B, w.K, w.V, w.Hq, w.Hkv, w.d, S, device=cuda())
    out = lr.libraspec_verify_round(inp["draft_logits"], inp["draft_tokens"], inp["temperature"],
                                    torch.tensor(cost, device=cuda()), inp["target_logits"], layers,
                                    torch.tensor(kv, device=cuda()), w.philox_seed, ws, want_lse=True)
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) == 0
    L_gpu = out.L.cpu().numpy()
    rows = None
    if name == "ragged":
        longest = int(np.argmax(L_gpu))
        rows = _group_rows(w, L_gpu, sorted({0, longest, w.B // 2, w.B - 1}))
    q, L, sflag, n, bonus, aflag, outs = _oracle_round(orc, w, inp, kv, layers, cost, L_gpu, rows=rows)
    nsel = assert_exact_unless_flagged(L_gpu, L, sflag, "L")
    assert_flag_budget(nsel, w.B, "%s selection" % name, per=32)
    nacc = assert_exact_unless_flagged(out.n_accepted.cpu().numpy(), n, aflag, "n_accepted")
    assert_exact_unless_flagged(out.bonus_token.cpu().numpy(), bonus, aflag, "bonus_token")
    assert_flag_budget(nacc, w.B, "%s acceptance" % name)
    for l in range(n_layers):
        check_attn(out.O[l], out.lse[l], outs[l][0], outs[l][1], L_gpu,
                   rows=None if rows is None else [tuple(r) for r in rows])


@pytest.mark.parametrize("in_place", [True, False])
def test_host_buffer_api_round_trip(orc, in_place):
    w = workloads.WORKLOADS["tiny"]
    kv = workloads.kv_lengths(w)
    lay = workloads.layer(w, 0, kv, device=cuda())
    inp = workloads.logits(w)
    K1 = w.K + 1
    caches = [{"Kc": lay["Kc"].clone(), "Vc": lay["Vc"].clone()}]
    runner = api.VerifyRound(w.B, w.K, w.V, w.Hq, w.Hkv, w.d, lay["Kc"].shape[2], caches, torch.tensor(kv),
                             inputs_in_place=in_place)
    host = {k: v.pin_memory() for k, v in inp.items()}
    host["cost_table"] = torch.tensor(workloads.cost_table(w)).pin_memory()
    kvb = int(kv[0])
    host["layers"] = [{"Q": lay["Q"].cpu().pin_memory(),
                       "K_new": lay["Kc"][:, :, kvb:kvb + K1].cpu().contiguous().pin_memory(),
                       "V_new": lay["Vc"][:, :, kvb:kvb + K1].cpu().contiguous().pin_memory()}]
    n, bonus = runner.run_host(host, seed=w.philox_seed)
    q, _ = orc.confidence(inp["draft_logits"].numpy(), inp["draft_tokens"].numpy(), inp["temperature"].numpy())
    L, sflag = orc.select_lengths(q, workloads.cost_table(w).astype(np.float64))
    n_ref, b_ref, aflag = orc.accept(inp["target_logits"].numpy(), inp["draft_logits"].numpy(),
                                     inp["draft_tokens"].numpy(), L, inp["temperature"].numpy(), w.philox_seed)
    assert not sflag.any()
    np.testing.assert_array_equal(n, n_ref)
    np.testing.assert_array_equal(bonus, b_ref)
    O_ref, lse_ref = orc.verify_attn(lay["Q"], lay["Kc"], lay["Vc"], kv, L)
    check_attn(runner.out.O[0], None, O_ref, lse_ref, L)
