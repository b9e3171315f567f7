"""GPU parity: drafter confidence and the LibraSpec selector vs. the oracle."""
import numpy as np
import pytest
import torch

from helpers import PROB_ATOL, assert_exact_unless_flagged, assert_flag_budget, cuda
from paper_2608_08721_gb300 import binding as lr
from paper_2608_08721_gb300 import workloads

pytestmark = pytest.mark.gpu


def _ws(B, K, V):
    return lr.Workspace(B, K, V, device=cuda())


@pytest.mark.parametrize("name", ["tiny", "8b", "sampling", "ragged", "70b"])
def test_confidence_full_size(orc, name):
    w = workloads.WORKLOADS[name]
    inp = workloads.logits(w, device=cuda())
    ws = _ws(w.B, w.K, w.V)
    conf, dstat = lr.libraspec_confidence(inp["draft_logits"], inp["draft_tokens"], inp["temperature"], ws)
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) == 0
    q_ref, d_ref = orc.confidence(inp["draft_logits"].cpu().numpy(), inp["draft_tokens"].cpu().numpy(),
                                  inp["temperature"].cpu().numpy())
    q = conf.cpu().numpy().astype(np.float64)
    assert np.max(np.abs(q - q_ref)) <= PROB_ATOL
    rel = np.abs(q - q_ref) / np.maximum(q_ref, 1e-30)
    assert np.max(rel[q_ref > 1e-6]) < 2e-6, "relative error of q %.3e" % np.max(rel[q_ref > 1e-6])
    d = dstat.cpu().numpy()
    np.testing.assert_array_equal(d[..., 0], d_ref[..., 0].astype(np.float32))
    np.testing.assert_allclose(d[..., 1], d_ref[..., 1], rtol=2e-6)


@pytest.mark.parametrize("V", [1, 3, 5, 4097, 32000])
@pytest.mark.parametrize("K", [1, 7, 64])
def test_confidence_ragged_shapes(orc, V, K):
    g = torch.Generator(device="cuda").manual_seed(V * 31 + K)
    B = 3
    x = torch.randn((B, K, V), generator=g, device=cuda()) * 3
    tok = torch.randint(0, V, (B, K), generator=g, device=cuda(), dtype=torch.int32)
    temp = torch.tensor([0.0, 0.7, 1.3], device=cuda())
    ws = _ws(B, K, V)
    conf, dstat = lr.libraspec_confidence(x, tok, temp, ws)
    q_ref, _ = orc.confidence(x.cpu().numpy(), tok.cpu().numpy(), temp.cpu().numpy())
    assert np.max(np.abs(conf.cpu().numpy() - q_ref)) <= PROB_ATOL


def test_confidence_unaligned_rows_use_scalar_path(orc):
    # a view starting one float in: rows are not 16-byte aligned
    g = torch.Generator(device="cuda").manual_seed(5)
    B, K, V = 2, 3, 1000
    base = torch.randn(B * K * V + 1, generator=g, device=cuda())
    x = base[1:].view(B, K, V)
    tok = torch.randint(0, V, (B, K), generator=g, device=cuda(), dtype=torch.int32)
    temp = torch.tensor([0.0, 0.5], device=cuda())
    conf, _ = lr.libraspec_confidence(x, tok, temp, _ws(B, K, V))
    q_ref, _ = orc.confidence(x.cpu().numpy(), tok.cpu().numpy(), temp.cpu().numpy())
    assert np.max(np.abs(conf.cpu().numpy() - q_ref)) <= PROB_ATOL


def test_confidence_bad_token_sets_status():
    B, K, V = 1, 2, 64
    x = torch.zeros((B, K, V), device=cuda())
    tok = torch.tensor([[3, 64]], dtype=torch.int32, device=cuda())
    ws = _ws(B, K, V)
    lr.libraspec_confidence(x, tok, torch.zeros(1, device=cuda()), ws)
    assert lr.libraspec_get_status(ws) & lr.ST_BAD_TOKEN
    assert lr.libraspec_get_status(ws) == 0  # reading clears it


@pytest.mark.parametrize("name", ["tiny", "8b", "sampling", "ragged", "70b"])
def test_select_on_gpu_confidence_is_exact(orc, name):
    """Same fp32 confidences on both sides: L must be identical unless flagged."""
    w = workloads.WORKLOADS[name]
    inp = workloads.logits(w, device=cuda())
    ws = _ws(w.B, w.K, w.V)
    conf, _ = lr.libraspec_confidence(inp["draft_logits"], inp["draft_tokens"], inp["temperature"], ws)
    cost = torch.tensor(workloads.cost_table(w), device=cuda())
    L = lr.libraspec_select_lengths(conf, cost, ws)
    L_ref, flag = orc.select_lengths(conf.cpu().numpy().astype(np.float64),
                                     cost.cpu().numpy().astype(np.float64))
    assert_exact_unless_flagged(L.cpu().numpy(), L_ref, flag, "L")


@pytest.mark.parametrize("name", ["tiny", "8b", "sampling", "ragged", "70b"])
def test_round_selection_matches_oracle_chain(orc, name):
    """Whole chain from the logits: GPU conf+select vs. oracle conf+select (fp64)."""
    w = workloads.WORKLOADS[name]
    inp = workloads.logits(w, device=cuda())
    ws = _ws(w.B, w.K, w.V)
    conf, _ = lr.libraspec_confidence(inp["draft_logits"], inp["draft_tokens"], inp["temperature"], ws)
    cost = workloads.cost_table(w)
    L = lr.libraspec_select_lengths(conf, torch.tensor(cost, device=cuda()), ws).cpu().numpy()
    q_ref, _ = orc.confidence(inp["draft_logits"].cpu().numpy(), inp["draft_tokens"].cpu().numpy(),
                              inp["temperature"].cpu().numpy())
    L_ref, flag = orc.select_lengths(q_ref, cost.astype(np.float64))
    nf = assert_exact_unless_flagged(L, L_ref, flag, "L")
    assert_flag_budget(nf, w.B, "%s selection" % name, per=32)
    if name == "ragged":
        # the per-sequence peakedness spreads the selected lengths: the measured cost table is a
        # staircase (flat between the latency steps at L = 1, 5, 8, ...), so the scan stops just
        # below a step, at several different lengths
        assert L_ref.min() == 0 and L_ref.max() >= 4 and len(set(L_ref.tolist())) >= 3, \
            "ragged lengths: %s" % L_ref


def test_select_edge_cases(orc):
    K = 64
    B = 8
    q = np.zeros((B, K), np.float32)
    q[0] = 1.0                        # all confident: L = K (linear cost with a > c)
    q[1, 0] = 0.0                     # first draft hopeless: L = 0
    q[2] = 0.5
    q[3, :40] = 0.999
    q[4] = np.linspace(1, 0, K)
    q[5] = 1.0
    q[5, 33] = 0.0                    # crosses the 32-lane chunk boundary
    q[6] = np.float32(0.9)
    q[7, :] = np.float32(1e-3)
    cost = (1.0 + 0.01 * np.arange(K + 1)).astype(np.float32)
    ws = _ws(B, K, 1)
    L = lr.libraspec_select_lengths(torch.tensor(q, device=cuda()), torch.tensor(cost, device=cuda()), ws)
    L_ref, flag = orc.select_lengths(q.astype(np.float64), cost.astype(np.float64))
    assert_exact_unless_flagged(L.cpu().numpy(), L_ref, flag, "L")
    assert int(L[0]) == K and int(L[1]) == 0


def test_select_rejects_nonpositive_cost_on_device():
    K = 4
    ws = _ws(2, K, 1)
    conf = torch.full((2, K), 0.9, device=cuda())
    cost = torch.tensor([1.0, 1.1, 0.0, 1.3, 1.4], device=cuda())
    L = lr.libraspec_select_lengths(conf, cost, ws)
    assert lr.libraspec_get_status(ws) & lr.ST_BAD_COST
    assert L.cpu().tolist() == [0, 0]


def test_select_random_adversarial(orc):
    rng = np.random.default_rng(9)
    B, K = 512, 33
    q = (rng.uniform(0, 1, size=(B, K)) ** rng.uniform(0.05, 3, size=(B, 1))).astype(np.float32)
    q[::7] = np.round(q[::7] * 4) / 4     # exact quarters: ties and zeros
    cost = (1.0 + 0.02 * np.arange(K + 1) + 0.001 * np.arange(K + 1) ** 2).astype(np.float32)
    ws = _ws(B, K, 1)
    L = lr.libraspec_select_lengths(torch.tensor(q, device=cuda()), torch.tensor(cost, device=cuda()), ws)
    L_ref, flag = orc.select_lengths(q.astype(np.float64), cost.astype(np.float64))
    assert_exact_unless_flagged(L.cpu().numpy(), L_ref, flag, "L")


@pytest.mark.parametrize("name", ["tiny", "8b", "sampling", "ragged"])
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_fused_confidence_select_equals_the_two_calls(name, dtype):
    """libraspec_confidence_select: the same conf, dstat and L as
    libraspec_confidence followed by libraspec_select_lengths, bit for bit."""
    w = workloads.WORKLOADS[name]
    inp = workloads.logits(w, device=cuda())
    x = inp["draft_logits"].to(dtype)
    cost = torch.tensor(workloads.cost_table(w), device=cuda())
    ws = lr.Workspace(w.B, w.K, w.V, device=cuda())
    c1, d1 = lr.libraspec_confidence(x, inp["draft_tokens"], inp["temperature"], ws)
    L1 = lr.libraspec_select_lengths(c1, cost, ws)
    for _ in range(2):   # the tickets reset themselves between calls
        c2, d2, L2 = lr.libraspec_confidence_select(x, inp["draft_tokens"], inp["temperature"], cost, ws)
        torch.cuda.synchronize()
        assert torch.equal(c1, c2) and torch.equal(d1, d2) and torch.equal(L1, L2)
    assert lr.libraspec_get_status(ws) == 0


def test_fused_confidence_select_bad_cost_sets_status():
    w = workloads.WORKLOADS["tiny"]
    inp = workloads.logits(w, device=cuda())
    cost = torch.tensor(workloads.cost_table(w), device=cuda())
    cost[3] = -1.0
    ws = lr.Workspace(w.B, w.K, w.V, device=cuda())
    _, _, L = lr.libraspec_confidence_select(inp["draft_logits"], inp["draft_tokens"], inp["temperature"], cost, ws)
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) & lr.ST_BAD_COST
    assert (L == 0).all()
