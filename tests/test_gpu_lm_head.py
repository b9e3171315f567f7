"""GPU parity: row statistics straight from the LM head (tcgen05 GEMM with the
statistics in its epilogue) against the oracle, and against the confidence
kernel run on the materialised logits."""
import numpy as np
import pytest
import torch

from helpers import PROB_ATOL, cuda
from paper_2608_08721_gb300 import binding as lr

pytestmark = pytest.mark.gpu


def _inputs(M, V, Dm, seed, sigma=4.0):
    g = torch.Generator(device="cuda").manual_seed(seed)
    H = torch.randn((M, Dm), generator=g, device=cuda()).to(torch.bfloat16)
    W = (torch.randn((V, Dm), generator=g, device=cuda()) * (sigma / Dm ** 0.5)).to(torch.bfloat16)
    return H, W


def _check(orc, H, W, T, rows_per_seq, tok, out):
    row_stat, arg, tp = (None if x is None else x.cpu().numpy() for x in out)
    mx, Z, rarg, rtp, flag = orc.lm_head_stats(H, W, T, rows_per_seq, tok)
    np.testing.assert_allclose(row_stat[:, 0], mx, rtol=1e-5, atol=1e-4)
    np.testing.assert_allclose(row_stat[:, 1], Z, rtol=1e-4)
    bad = (arg != rarg) & (flag == 0)
    assert not bad.any(), np.nonzero(bad)[0]
    if tp is not None:
        np.testing.assert_allclose(tp, rtp, rtol=0, atol=PROB_ATOL)
    return flag


@pytest.mark.parametrize("M,V,Dm", [(33, 32000, 512), (16, 1003, 256), (300, 5000, 128), (128, 4096, 4096),
                                    (17, 128256, 256)])
def test_lm_head_stats_match_oracle(orc, M, V, Dm):
    H, W = _inputs(M, V, Dm, seed=M + V % 97 + Dm)
    rps = 1 if M % 3 else 3
    T = torch.tensor([[0.0, 0.7, 1.0, 1.8][i % 4] for i in range(M // rps)], device=cuda())
    rng = np.random.default_rng(M)
    tok = rng.integers(-1, V, size=M).astype(np.int32)
    ws = lr.LmHeadWorkspace(M, V)
    out = lr.libraspec_lm_head_stats(H, W, ws, temperature=T, rows_per_seq=rps,
                                     tokens=torch.from_numpy(tok).to(cuda()))
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) == 0
    flag = _check(orc, H, W, T.cpu().numpy(), rps, tok, out)
    assert flag.sum() <= max(1, M // 20)


def test_lm_head_stats_without_tokens_or_temperature(orc):
    H, W = _inputs(40, 3000, 192, seed=4)
    ws = lr.LmHeadWorkspace(40, 3000)
    out = lr.libraspec_lm_head_stats(H, W, ws)
    torch.cuda.synchronize()
    assert out[2] is None
    _check(orc, H, W, None, 1, None, out)


def test_lm_head_confidence_equals_confidence_kernel_on_logits():
    """With the drafter rows and tokens, token_prob / row_stat are the conf /
    dstat that libraspec_confidence computes from the materialised logits."""
    B, K, V, Dm = 4, 16, 32000, 1024
    H, W = _inputs(B * K, V, Dm, seed=9)
    logits = (H.float() @ W.float().T).reshape(B, K, V).contiguous()
    g = torch.Generator(device="cuda").manual_seed(1)
    tok = torch.randint(0, V, (B, K), generator=g, device=cuda(), dtype=torch.int32)
    tok[:, ::2] = logits.argmax(-1)[:, ::2].int()     # high-probability drafts too
    T = torch.tensor([0.0, 1.0, 0.6, 1.4], device=cuda())
    ws = lr.LmHeadWorkspace(B * K, V)
    row_stat, _, tp = lr.libraspec_lm_head_stats(H, W, ws, temperature=T, rows_per_seq=K, tokens=tok.reshape(-1))
    ws2 = lr.Workspace(B, K, V, device=cuda())
    conf, dstat = lr.libraspec_confidence(logits, tok, T, ws2)
    torch.cuda.synchronize()
    np.testing.assert_allclose(tp.reshape(B, K).cpu().numpy(), conf.cpu().numpy(), rtol=0, atol=PROB_ATOL)
    np.testing.assert_allclose(row_stat.reshape(B, K, 2)[..., 0].cpu().numpy(), dstat[..., 0].cpu().numpy(),
                               rtol=1e-5, atol=1e-4)
    np.testing.assert_allclose(row_stat.reshape(B, K, 2)[..., 1].cpu().numpy(), dstat[..., 1].cpu().numpy(),
                               rtol=1e-4)


def test_lm_head_bad_token_sets_status():
    H, W = _inputs(8, 1000, 64, seed=2)
    ws = lr.LmHeadWorkspace(8, 1000)
    tok = torch.zeros(8, dtype=torch.int32, device=cuda())
    tok[3] = 1000
    _, _, tp = lr.libraspec_lm_head_stats(H, W, ws, tokens=tok)
    torch.cuda.synchronize()
    assert lr.libraspec_get_status(ws) & lr.ST_BAD_TOKEN
    assert np.isnan(tp[3].item()) and np.isfinite(tp[:3].cpu().numpy()).all()


def test_lm_head_rejects_unsupported_model_dim():
    H, W = _inputs(4, 100, 64, seed=3)
    ws = lr.LmHeadWorkspace(4, 100)
    with pytest.raises(lr.LibraspecError):
        lr.libraspec_lm_head_stats(H[:, :48].contiguous(), W[:, :48].contiguous(), ws)


def test_lm_head_single_row_and_single_tile_vocabulary(orc):
    for M, V in ((1, 77), (1, 128), (129, 64)):
        H, W = _inputs(M, V, 64, seed=M * 1000 + V)
        ws = lr.LmHeadWorkspace(M, V)
        tok = torch.arange(M, dtype=torch.int32, device=cuda()) % V
        out = lr.libraspec_lm_head_stats(H, W, ws, tokens=tok)
        torch.cuda.synchronize()
        assert lr.libraspec_get_status(ws) == 0
        _check(orc, H, W, None, 1, tok.cpu().numpy(), out)
