"""Pins of the oracle's drafter-confidence step (Assumption 1, Algorithm 1's q_k).

q_k is the drafter's softmax probability (at the sequence's temperature, T = 1
for greedy sequences) of the token it drafted. Pinned against scipy's softmax
(an independent library routine) and closed forms.
"""
import numpy as np
import pytest
from scipy.special import softmax

from paper_2608_08721_gb300 import workloads


def _rand_case(rng, B, K, V, scale=4.0):
    x = (rng.standard_normal((B, K, V)) * scale).astype(np.float32)
    tok = rng.integers(0, V, size=(B, K)).astype(np.int32)
    return x, tok


@pytest.mark.parametrize("T", [0.0, 1.0, 0.7, 2.5])
def test_conf_matches_scipy_softmax(orc, T):
    rng = np.random.default_rng(1)
    x, tok = _rand_case(rng, 3, 5, 257)
    temp = np.full(3, T, np.float32)
    q, dstat = orc.confidence(x, tok, temp)
    Teff = 1.0 if T == 0.0 else float(np.float32(T))
    for b in range(3):
        for k in range(5):
            ref = softmax(x[b, k].astype(np.float64) / Teff)[tok[b, k]]
            assert q[b, k] == pytest.approx(ref, rel=1e-12, abs=1e-300)
            assert dstat[b, k, 0] == float(x[b, k].max())
            # Z * exp(m/T) is the softmax normaliser of x/T
            logZ = np.log(dstat[b, k, 1]) + dstat[b, k, 0] / Teff
            ref_logZ = np.log(np.sum(np.exp(x[b, k].astype(np.float64) / Teff)))
            assert logZ == pytest.approx(ref_logZ, rel=1e-12)


def test_conf_uniform_row_is_one_over_V(orc):
    V = 1000
    x = np.full((1, 2, V), 3.25, np.float32)
    tok = np.array([[0, 999]], np.int32)
    q, _ = orc.confidence(x, tok, np.array([0.0], np.float32))
    np.testing.assert_allclose(q, 1.0 / V, rtol=1e-14)


def test_conf_one_hot_closed_form(orc):
    V = 50
    x = np.zeros((1, 2, V), np.float32)
    x[0, 0, 7] = 20.0
    x[0, 1, 7] = 20.0
    tok = np.array([[7, 8]], np.int32)
    T = 0.5
    q, _ = orc.confidence(x, tok, np.array([T], np.float32))
    e = np.exp(-20.0 / T)
    assert q[0, 0] == pytest.approx(1.0 / (1.0 + (V - 1) * e), rel=1e-14)
    assert q[0, 1] == pytest.approx(e / (1.0 + (V - 1) * e), rel=1e-12)


def test_conf_is_shift_invariant(orc):
    rng = np.random.default_rng(5)
    x, tok = _rand_case(rng, 2, 3, 64)
    x = (np.round(x * 1024) / 1024).astype(np.float32)   # so that x + 64 is exact
    temp = np.array([1.0, 0.6], np.float32)
    q1, _ = orc.confidence(x, tok, temp)
    q2, _ = orc.confidence(x + np.float32(64.0), tok, temp)
    np.testing.assert_allclose(q1, q2, rtol=1e-12)


def test_conf_greedy_uses_native_distribution(orc):
    rng = np.random.default_rng(6)
    x, tok = _rand_case(rng, 2, 4, 100)
    q0, _ = orc.confidence(x, tok, np.zeros(2, np.float32))
    q1, _ = orc.confidence(x, tok, np.ones(2, np.float32))
    np.testing.assert_array_equal(q0, q1)


def test_conf_rejects_bad_tokens(orc):
    x = np.zeros((1, 1, 4), np.float32)
    with pytest.raises(orc.OracleError):
        orc.confidence(x, np.array([[4]], np.int32), np.zeros(1, np.float32))
    with pytest.raises(orc.OracleError):
        orc.confidence(x, np.array([[-1]], np.int32), np.zeros(1, np.float32))


def test_conf_on_workload_rows(orc):
    w = workloads.WORKLOADS["tiny"]
    inp = workloads.logits(w)
    x = inp["draft_logits"].numpy()
    tok = inp["draft_tokens"].numpy()
    q, _ = orc.confidence(x, tok, inp["temperature"].numpy())
    # greedy drafts are the drafter's argmax: their probability is the row maximum
    for k in range(w.K):
        p = softmax(x[0, k].astype(np.float64))
        assert q[0, k] == pytest.approx(p.max(), rel=1e-12)
