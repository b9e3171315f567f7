"""Pins of the oracle's LM-head row statistics (confidence and acceptance
row statistics from hidden states and LM-head weights, logits never stored).

With small-integer hidden states and weights the logits are exact in
binary32, so the statistics must equal the (separately pinned) confidence
oracle run on the materialised logits; closed forms cover a zero head (the
uniform distribution) and a head whose rows are scaled copies of the hidden
state; the tie flag is checked on planted ties."""
import numpy as np
import pytest
import torch

import oracle


def _bf16(a):
    return torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(torch.bfloat16)


def test_matches_confidence_oracle_on_exact_logits():
    rng = np.random.default_rng(0)
    B, K, V, Dm = 3, 5, 211, 96
    H = rng.integers(-3, 4, size=(B * K, Dm)).astype(np.float32)
    W = rng.integers(-2, 3, size=(V, Dm)).astype(np.float32)
    logits = (H.astype(np.float64) @ W.T.astype(np.float64))
    assert np.abs(logits).max() < 2 ** 24                    # exact in binary32
    logits = (logits / 8.0).astype(np.float32)               # a power-of-two scale stays exact
    W = W / 8.0
    T = np.array([0.0, 0.7, 1.3], np.float32)
    tok = rng.integers(0, V, size=(B, K)).astype(np.int32)
    mx, Z, arg, tp, flag = oracle.lm_head_stats(_bf16(H), _bf16(W), T, K, tok.reshape(-1))
    conf, dstat = oracle.confidence(logits.reshape(B, K, V), tok, T)
    np.testing.assert_allclose(tp.reshape(B, K), conf, rtol=1e-13, atol=0)
    np.testing.assert_allclose(mx.reshape(B, K), dstat[..., 0], rtol=0, atol=0)
    np.testing.assert_allclose(Z.reshape(B, K), dstat[..., 1], rtol=1e-13)
    flat = logits.reshape(B * K, V)
    np.testing.assert_array_equal(arg, np.argmax(flat, axis=1))
    # integer logits tie often; a tie at the top is flagged, a clear top is not
    top2 = np.sort(flat, axis=1)[:, -2:]
    np.testing.assert_array_equal(flag, (top2[:, 1] == top2[:, 0]).astype(np.int32))


def test_zero_head_is_uniform():
    M, V, Dm = 4, 50, 64
    H = np.random.default_rng(1).standard_normal((M, Dm)).astype(np.float32)
    mx, Z, arg, tp, flag = oracle.lm_head_stats(_bf16(H), _bf16(np.zeros((V, Dm))), None, 1,
                                                np.array([0, 7, 49, -1], np.int32))
    np.testing.assert_array_equal(mx, 0.0)
    np.testing.assert_allclose(Z, float(V), rtol=1e-15)
    np.testing.assert_array_equal(arg, 0)
    np.testing.assert_allclose(tp[:3], 1.0 / V, rtol=1e-14)
    assert tp[3] == 0.0
    assert flag.all()   # every logit ties


def test_scaled_copies_of_the_hidden_state():
    """W[v] = c_v * h: the logits are c_v |h|^2, so the argmax is the largest
    c_v and Z is a closed-form sum."""
    Dm, V = 64, 9
    h = np.zeros(Dm, np.float32)
    h[:4] = [1.0, -2.0, 0.5, 0.25]                           # |h|^2 = 5.3125
    c = np.array([0.0, 0.5, -1.0, 2.0, 0.25, 1.5, -0.5, 1.0, 0.75], np.float32)
    W = c[:, None] * h[None, :]
    T = 2.0
    mx, Z, arg, tp, flag = oracle.lm_head_stats(_bf16(h[None]), _bf16(W), np.array([T], np.float32), 1,
                                                np.array([5], np.int32))
    x = c.astype(np.float64) * 5.3125
    assert arg[0] == 3 and mx[0] == x[3]
    np.testing.assert_allclose(Z[0], np.exp((x - x[3]) / T).sum(), rtol=1e-14)
    np.testing.assert_allclose(tp[0], np.exp((x[5] - x[3]) / T) / Z[0], rtol=1e-14)
    assert flag[0] == 0


def test_rejects_bad_arguments():
    H = _bf16(np.zeros((2, 64)))
    W = _bf16(np.zeros((5, 64)))
    with pytest.raises(oracle.OracleError):
        oracle.lm_head_stats(H, W, None, 1, np.array([0, 5], np.int32))     # token >= V
    with pytest.raises(oracle.OracleError):
        oracle.lm_head_stats(H, _bf16(np.zeros((5, 32))), None, 1, None)      # Dm mismatch
