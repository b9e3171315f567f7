"""GPU parity: acceptance (greedy and rejection sampling) vs. the oracle."""
import numpy as np
import pytest
import torch

from helpers import assert_exact_unless_flagged, assert_flag_budget, cuda
from paper_2608_08721_gb300 import binding as lr
from paper_2608_08721_gb300 import workloads

pytestmark = pytest.mark.gpu


def _gpu_accept(inp, L, seed, round_offset=0, seq_offset=0):
    B, K1, V = inp["target_logits"].shape
    ws = lr.Workspace(B, K1 - 1, V, device=cuda())
    conf, dstat = lr.libraspec_confidence(inp["draft_logits"], inp["draft_tokens"], inp["temperature"], ws)
    L_t = torch.as_tensor(np.asarray(L, np.int32)).to(cuda())
    n, bonus = lr.libraspec_accept(inp["target_logits"], inp["draft_logits"], inp["draft_tokens"], conf, dstat,
                                   L_t, inp["temperature"], seed, ws, round_offset=round_offset,
                                   seq_offset=seq_offset)
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) == 0
    return n.cpu().numpy(), bonus.cpu().numpy()


def _oracle_accept(orc, inp, L, seed, round_offset=0, seq_offset=0):
    return orc.accept(inp["target_logits"].cpu().numpy(), inp["draft_logits"].cpu().numpy(),
                      inp["draft_tokens"].cpu().numpy(), np.asarray(L, np.int32),
                      inp["temperature"].cpu().numpy(), seed, round_offset, seq_offset)


@pytest.mark.parametrize("name", ["tiny", "8b", "sampling", "ragged", "70b"])
def test_accept_full_size_selected_lengths(orc, name):
    """Lengths from the GPU selector (bit-exact vs. the oracle elsewhere)."""
    w = workloads.WORKLOADS[name]
    inp = workloads.logits(w, device=cuda())
    ws = lr.Workspace(w.B, w.K, w.V, device=cuda())
    conf, _ = lr.libraspec_confidence(inp["draft_logits"], inp["draft_tokens"], inp["temperature"], ws)
    L = lr.libraspec_select_lengths(conf, torch.tensor(workloads.cost_table(w), device=cuda()), ws).cpu().numpy()
    n, bonus = _gpu_accept(inp, L, w.philox_seed)
    n_ref, b_ref, flag = _oracle_accept(orc, inp, L, w.philox_seed)
    nf = assert_exact_unless_flagged(n, n_ref, flag, "n_accepted")
    assert_exact_unless_flagged(bonus, b_ref, flag, "bonus_token")
    assert_flag_budget(nf, w.B, "%s acceptance" % name)
    greedy = inp["temperature"].cpu().numpy() == 0
    assert not flag[greedy].any(), "greedy decisions are exact and never flagged"


@pytest.mark.parametrize("name", ["sampling", "ragged"])
@pytest.mark.parametrize("which", ["zero", "full", "random"])
def test_accept_length_extremes(orc, name, which):
    w = workloads.WORKLOADS[name]
    inp = workloads.logits(w, device=cuda())
    rng = np.random.default_rng(4)
    L = {"zero": np.zeros(w.B), "full": np.full(w.B, w.K),
         "random": rng.integers(0, w.K + 1, size=w.B)}[which].astype(np.int32)
    for round_offset in (0, 7):
        n, bonus = _gpu_accept(inp, L, w.philox_seed, round_offset=round_offset)
        n_ref, b_ref, flag = _oracle_accept(orc, inp, L, w.philox_seed, round_offset=round_offset)
        assert_exact_unless_flagged(n, n_ref, flag, "n_accepted")
        assert_exact_unless_flagged(bonus, b_ref, flag, "bonus_token")


def test_accept_small_vocab_many_sequences(orc):
    """Many short rows: residual and bonus draws over tiny vocabularies, both
    vectorised (V % 4 == 0) and scalar (V % 4 != 0) paths."""
    for V in (8, 13, 4096, 50001):
        B, K = 96, 4
        g = torch.Generator(device="cuda").manual_seed(V)
        tgt = torch.randn((B, K + 1, V), generator=g, device=cuda()) * 1.5
        dr = tgt[:, :K] + torch.randn((B, K, V), generator=g, device=cuda())
        T = torch.where(torch.arange(B, device=cuda()) % 3 == 0, 0.0, 0.9).float()
        tok = torch.empty((B, K), dtype=torch.int32, device=cuda())
        for b in range(B):
            t = float(T[b])
            if t == 0:
                tok[b] = dr[b].argmax(-1).int()
            else:
                u = torch.rand((K, V), generator=g, device=cuda()).clamp_(1e-30, 1 - 1e-7)
                tok[b] = (dr[b] / t - torch.log(-torch.log(u))).argmax(-1).int()
        inp = {"target_logits": tgt.contiguous(), "draft_logits": dr.contiguous(), "draft_tokens": tok,
               "temperature": T}
        L = np.random.default_rng(V).integers(0, K + 1, size=B).astype(np.int32)
        n, bonus = _gpu_accept(inp, L, seed=77 + V, seq_offset=1000)
        n_ref, b_ref, flag = _oracle_accept(orc, inp, L, 77 + V, seq_offset=1000)
        assert_exact_unless_flagged(n, n_ref, flag, "n_accepted")
        assert_exact_unless_flagged(bonus, b_ref, flag, "bonus_token")


def test_accept_sequence_offset_sharding(orc):
    w = workloads.WORKLOADS["sampling"].scaled(V=4096)
    inp = workloads.logits(w, device=cuda())
    L = np.full(w.B, 8, np.int32)
    n_all, b_all = _gpu_accept(inp, L, 1234)
    half = {k: v[8:].contiguous() for k, v in inp.items()}
    n_hi, b_hi = _gpu_accept(half, L[8:], 1234, seq_offset=8)
    np.testing.assert_array_equal(n_all[8:], n_hi)
    np.testing.assert_array_equal(b_all[8:], b_hi)


def test_accept_bad_length_sets_status():
    B, K, V = 2, 4, 64
    inp = {"target_logits": torch.zeros((B, K + 1, V), device=cuda()),
           "draft_logits": torch.zeros((B, K, V), device=cuda()),
           "draft_tokens": torch.zeros((B, K), dtype=torch.int32, device=cuda()),
           "temperature": torch.zeros(B, device=cuda())}
    ws = lr.Workspace(B, K, V, device=cuda())
    L = torch.tensor([1, 9], dtype=torch.int32, device=cuda())
    n, bonus = lr.libraspec_accept(inp["target_logits"], inp["draft_logits"], inp["draft_tokens"], None, None, L,
                                   inp["temperature"], 0, ws)
    assert lr.libraspec_get_status(ws) & lr.ST_BAD_LENGTH
    assert int(n[1]) == 0


def test_accept_missing_confidence_for_sampling_sets_status():
    B, K, V = 1, 2, 64
    ws = lr.Workspace(B, K, V, device=cuda())
    lr.libraspec_accept(torch.zeros((B, K + 1, V), device=cuda()), torch.zeros((B, K, V), device=cuda()),
                        torch.zeros((B, K), dtype=torch.int32, device=cuda()), None, None,
                        torch.ones(B, dtype=torch.int32, device=cuda()), torch.ones(B, device=cuda()), 0, ws)
    assert lr.libraspec_get_status(ws) & lr.ST_MISSING_INPUT


def _race_rows(V, seed):
    """Ten sampling sequences (T = 1, K = 2) whose draws stress the races'
    screens: bonus draws (L = 0) from a flat row, a flat row with every other
    token at -inf, a row with one dominant token, a very peaked row, a row
    with three finite tokens and a plain row; residual draws (L = 2, the
    drafted token's target logit lowered so that it is rejected) from plain
    rows, and one (the last) where the drafter only raises its drafted token,
    so that every other token's residual max(0, p - q) is a small difference
    of nearly equal probabilities."""
    g = torch.Generator().manual_seed(seed)
    B, K = 10, 2
    tgt = torch.randn((B, K + 1, V), generator=g)
    tgt[0] = 0.0
    tgt[1] = 0.0
    tgt[1, :, ::2] = -float("inf")
    tgt[2, :, 17] += 25.0
    tgt[3] *= 8.0
    tgt[4] = -float("inf")
    tgt[4, :, 3], tgt[4, :, V // 2], tgt[4, :, V - 1] = 0.0, 0.5, 1.0
    tgt[6:] *= 2.0
    dr = tgt[:, :K] + torch.randn((B, K, V), generator=g) * 3.0
    dr[9] = tgt[9, :K]
    tok = dr.argmax(-1).int()
    for b in range(6, 9):
        for j in range(K):
            tgt[b, j, int(tok[b, j])] -= 8.0
    for j in range(K):
        dr[9, j, int(tok[9, j])] += 6.0
    L = np.array([0] * 6 + [2] * 4, np.int32)
    inp = {"target_logits": tgt.contiguous().to(cuda()), "draft_logits": dr.contiguous().to(cuda()),
           "draft_tokens": tok.to(cuda()), "temperature": torch.ones(B, device=cuda())}
    return inp, L


@pytest.mark.parametrize("V", [50000, 50001])
def test_accept_race_degenerate_rows(orc, V):
    """The exponential races on flat, masked, dominated and peaked rows and on
    residuals obtained by cancellation, in both vector paths, against the
    oracle (exact unless flagged)."""
    inp, L = _race_rows(V, seed=V)
    unflagged = 0
    for round_offset in (0, 3):
        n, bonus = _gpu_accept(inp, L, seed=11, round_offset=round_offset)
        n_ref, b_ref, flag = _oracle_accept(orc, inp, L, 11, round_offset=round_offset)
        assert_exact_unless_flagged(n, n_ref, flag, "n_accepted")
        assert_exact_unless_flagged(bonus, b_ref, flag, "bonus_token")
        unflagged += int((flag == 0).sum())
        assert n_ref[6:9].tolist() == [0, 0, 0], "the lowered drafted tokens are rejected at once"
        assert bonus[2] == 17 or flag[2], "the dominant token wins the bonus draw"
        assert bonus[4] in (3, V // 2, V - 1) and bonus[1] % 2 == 1, "only finite logits can be drawn"
    assert unflagged >= 16, "%d of 20 draws unflagged" % unflagged
