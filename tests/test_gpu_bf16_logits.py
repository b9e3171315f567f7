"""GPU parity with bf16 logits (libraspec_confidence_bf16, libraspec_accept_bf16).

The logits are rounded to bf16 once; the oracle receives the same values
widened to binary64 (exact), so the tolerances and the exact-unless-flagged
rule of the fp32 tests apply unchanged."""
import numpy as np
import pytest
import torch

from helpers import PROB_ATOL, assert_exact_unless_flagged, cuda
from paper_2608_08721_gb300 import binding as lr
from paper_2608_08721_gb300 import workloads

pytestmark = pytest.mark.gpu


def _bf16_inputs(w):
    inp = workloads.logits(w, device=cuda())
    out = dict(inp)
    out["draft_logits"] = inp["draft_logits"].to(torch.bfloat16)
    out["target_logits"] = inp["target_logits"].to(torch.bfloat16)
    del inp
    return out


def _np64(t):
    return t.float().cpu().numpy().astype(np.float64)


def _check_conf(orc, logits, tokens, temperature):
    B, K, V = logits.shape
    ws = lr.Workspace(B, K, V, device=cuda())
    conf, dstat = lr.libraspec_confidence(logits, tokens, temperature, ws)
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) == 0
    q_ref, d_ref = orc.confidence(_np64(logits), tokens.cpu().numpy(), temperature.cpu().numpy())
    q = conf.cpu().numpy().astype(np.float64)
    assert np.max(np.abs(q - q_ref)) <= PROB_ATOL
    rel = np.abs(q - q_ref) / np.maximum(q_ref, 1e-30)
    if (q_ref > 1e-6).any():
        assert np.max(rel[q_ref > 1e-6]) < 2e-6, "relative error of q %.3e" % np.max(rel[q_ref > 1e-6])
    d = dstat.cpu().numpy()
    np.testing.assert_array_equal(d[..., 0], d_ref[..., 0].astype(np.float32))
    np.testing.assert_allclose(d[..., 1], d_ref[..., 1], rtol=2e-6)
    return conf, dstat


@pytest.mark.parametrize("name", ["tiny", "8b", "sampling", "70b"])
def test_confidence_bf16_full_size(orc, name):
    w = workloads.WORKLOADS[name]
    inp = _bf16_inputs(w)
    _check_conf(orc, inp["draft_logits"], inp["draft_tokens"], inp["temperature"])


@pytest.mark.parametrize("V", [1, 3, 8, 13, 4097, 32000])
@pytest.mark.parametrize("K", [1, 7, 64])
def test_confidence_bf16_ragged_shapes(orc, V, K):
    """V % 8 != 0 (and odd) rows take the element-wise path; V % 8 == 0 the
    128-bit one."""
    g = torch.Generator(device="cuda").manual_seed(V * 7 + K)
    B = 3
    x = (torch.randn((B, K, V), generator=g, device=cuda()) * 3.0).to(torch.bfloat16)
    tok = torch.randint(0, V, (B, K), generator=g, device=cuda(), dtype=torch.int32)
    T = torch.tensor([0.0, 0.7, 1.3], device=cuda())
    _check_conf(orc, x, tok, T)


def test_confidence_bf16_misaligned_rows(orc):
    """A base that is 2-byte but not 16-byte aligned takes the element-wise path."""
    g = torch.Generator(device="cuda").manual_seed(11)
    B, K, V = 2, 5, 4096
    buf = (torch.randn(B * K * V + 1, generator=g, device=cuda()) * 2.0).to(torch.bfloat16)
    x = buf[1:].view(B, K, V)
    tok = torch.randint(0, V, (B, K), generator=g, device=cuda(), dtype=torch.int32)
    _check_conf(orc, x, tok, torch.tensor([0.0, 1.0], device=cuda()))


@pytest.mark.parametrize("name", ["tiny", "8b", "sampling", "70b"])
def test_accept_bf16_full_size(orc, name):
    w = workloads.WORKLOADS[name]
    inp = _bf16_inputs(w)
    ws = lr.Workspace(w.B, w.K, w.V, device=cuda())
    conf, dstat = lr.libraspec_confidence(inp["draft_logits"], inp["draft_tokens"], inp["temperature"], ws)
    L = lr.libraspec_select_lengths(conf, torch.tensor(workloads.cost_table(w), device=cuda()), ws)
    rng = np.random.default_rng(5)
    for Lh in (L.cpu().numpy(), rng.integers(0, w.K + 1, size=w.B).astype(np.int32)):
        L_t = torch.as_tensor(Lh).to(cuda())
        n, bonus = lr.libraspec_accept(inp["target_logits"], inp["draft_logits"], inp["draft_tokens"], conf,
                                       dstat, L_t, inp["temperature"], w.philox_seed, ws)
        torch.cuda.synchronize()
        assert lr.libraspec_get_status(ws) == 0
        n_ref, b_ref, flag = orc.accept(_np64(inp["target_logits"]), _np64(inp["draft_logits"]),
                                        inp["draft_tokens"].cpu().numpy(), Lh, inp["temperature"].cpu().numpy(),
                                        w.philox_seed, 0, 0)
        assert_exact_unless_flagged(n.cpu().numpy(), n_ref, flag, "n_accepted")
        assert_exact_unless_flagged(bonus.cpu().numpy(), b_ref, flag, "bonus_token")


@pytest.mark.parametrize("V", [8, 13, 4096, 50001])
def test_accept_bf16_small_vocab(orc, V):
    B, K = 48, 4
    g = torch.Generator(device="cuda").manual_seed(V + 3)
    tgt = torch.randn((B, K + 1, V), generator=g, device=cuda()) * 1.5
    dr = tgt[:, :K] + torch.randn((B, K, V), generator=g, device=cuda())
    T = torch.where(torch.arange(B, device=cuda()) % 3 == 0, 0.0, 0.9).float()
    tok = torch.randint(0, V, (B, K), generator=g, device=cuda(), dtype=torch.int32)
    tgt16, dr16 = tgt.to(torch.bfloat16).contiguous(), dr.to(torch.bfloat16).contiguous()
    ws = lr.Workspace(B, K, V, device=cuda())
    conf, dstat = lr.libraspec_confidence(dr16, tok, T, ws)
    L = torch.full((B,), K, dtype=torch.int32, device=cuda())
    n, bonus = lr.libraspec_accept(tgt16, dr16, tok, conf, dstat, L, T, 77, ws)
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) == 0
    n_ref, b_ref, flag = orc.accept(_np64(tgt16), _np64(dr16), tok.cpu().numpy(), L.cpu().numpy(),
                                    T.cpu().numpy(), 77, 0, 0)
    assert_exact_unless_flagged(n.cpu().numpy(), n_ref, flag, "n_accepted")
    assert_exact_unless_flagged(bonus.cpu().numpy(), b_ref, flag, "bonus_token")


def test_bf16_mixed_dtypes_rejected():
    B, K, V = 1, 2, 16
    tgt = torch.zeros((B, K + 1, V), dtype=torch.bfloat16, device=cuda())
    dr = torch.zeros((B, K, V), device=cuda())
    tok = torch.zeros((B, K), dtype=torch.int32, device=cuda())
    ws = lr.Workspace(B, K, V, device=cuda())
    with pytest.raises((TypeError, ValueError, RuntimeError)):
        lr.libraspec_accept(tgt, dr, tok, None, None, torch.zeros(B, dtype=torch.int32, device=cuda()),
                            torch.zeros(B, device=cuda()), 1, ws)
