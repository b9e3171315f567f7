"""Pins of the oracle's acceptance step (Sec. 3.1; the rule of Leviathan et al.).

Greedy: exact constructed cases (prefix of argmax matches, lowest-index ties).
Sampling: Monte Carlo over many sequences (each sequence draws its own
uniforms) against closed forms:
* a fixed draft x is accepted with probability min(1, p(x)/q(x));
* with x ~ q the acceptance rate is sum_v min(p_v, q_v), and the emitted token
  is distributed as p (the verification is lossless, Sec. 3.1);
* after a rejection the emitted token follows norm(max(0, p - q));
* with nothing to verify the emitted token follows p;
* the expected number of accepted drafts is sum_j prod_{k<=j} beta_k
  (prefix acceptance, proof of Thm. 2), beta_k = sum_v min(p_k, q_k).
"""
import numpy as np
import pytest
from scipy.special import softmax
from scipy.stats import chisquare

N_MC = 120000


def _logits(rng, V, scale=1.5):
    return (rng.standard_normal(V) * scale).astype(np.float32)


def _tile(row_list, B):
    arr = np.stack(row_list)[None]            # [1, R, V]
    return np.ascontiguousarray(np.broadcast_to(arr, (B,) + arr.shape[1:]))


def _chi2_ok(counts, probs, min_p=1e-3):
    probs = np.asarray(probs, np.float64)
    probs = probs / probs.sum()
    exp = probs * counts.sum()
    keep = exp > 5
    obs = counts[keep].astype(np.float64)
    e = exp[keep]
    e = e * obs.sum() / e.sum()
    assert counts[~keep].sum() <= max(10, 0.002 * counts.sum())
    return chisquare(obs, e).pvalue > min_p


def test_greedy_prefix_match_and_bonus(orc):
    V, K = 10, 4
    tgt = np.zeros((3, K + 1, V), np.float32)
    argmaxes = [[1, 2, 3, 4, 5], [1, 2, 9, 4, 5], [7, 2, 3, 4, 5]]
    for b in range(3):
        for j in range(K + 1):
            tgt[b, j, argmaxes[b][j]] = 1.0
    draft = np.zeros((3, K, V), np.float32)
    tokens = np.array([[1, 2, 3, 4]] * 3, np.int32)
    L = np.array([4, 4, 4], np.int32)
    n, bonus, flag = orc.accept(tgt, draft, tokens, L, np.zeros(3, np.float32), seed=0)
    np.testing.assert_array_equal(n, [4, 2, 0])
    np.testing.assert_array_equal(bonus, [5, 9, 7])
    np.testing.assert_array_equal(flag, 0)
    # shorter selected lengths: only the first L_b drafts are checked
    n, bonus, _ = orc.accept(tgt, draft, tokens, np.array([0, 2, 3], np.int32), np.zeros(3, np.float32), 0)
    np.testing.assert_array_equal(n, [0, 2, 0])
    np.testing.assert_array_equal(bonus, [1, 9, 7])


def test_greedy_ties_go_to_lowest_index(orc):
    V = 6
    tgt = np.zeros((1, 2, V), np.float32)
    tgt[0, 0, [2, 4]] = 3.0
    tgt[0, 1, [1, 5]] = 3.0
    draft = np.zeros((1, 1, V), np.float32)
    n, bonus, _ = orc.accept(tgt, draft, np.array([[4]], np.int32), np.array([1], np.int32),
                             np.zeros(1, np.float32), 0)
    assert (n[0], bonus[0]) == (0, 2)
    n, bonus, _ = orc.accept(tgt, draft, np.array([[2]], np.int32), np.array([1], np.int32),
                             np.zeros(1, np.float32), 0)
    assert (n[0], bonus[0]) == (1, 1)


@pytest.mark.parametrize("T", [1.0, 0.7])
def test_fixed_draft_acceptance_probability(orc, T):
    rng = np.random.default_rng(21)
    V = 8
    yp, yq = _logits(rng, V), _logits(rng, V)
    p = softmax(yp.astype(np.float64) / np.float64(np.float32(T)))
    q = softmax(yq.astype(np.float64) / np.float64(np.float32(T)))
    for x in (int(np.argmax(q / p)), int(np.argmin(q / p))):
        B = N_MC
        tgt = _tile([yp, yp], B)
        dr = _tile([yq], B)
        tok = np.full((B, 1), x, np.int32)
        n, bonus, flag = orc.accept(tgt, dr, tok, np.ones(B, np.int32), np.full(B, T, np.float32), seed=5)
        a = min(1.0, p[x] / q[x])
        rate = n.mean()
        assert abs(rate - a) <= 4 * np.sqrt(a * (1 - a) / B) + 1e-12
        # rejected draws follow the residual norm(max(0, p - q)), never x itself
        res = np.maximum(p - q, 0)
        rej = bonus[n == 0]
        if rej.size > 1000:
            assert res[x] == 0 and not np.any(rej == x)
            assert _chi2_ok(np.bincount(rej, minlength=V), res)


@pytest.mark.parametrize("T", [1.0, 0.8])
def test_lossless_first_token_law(orc, T):
    rng = np.random.default_rng(22)
    V = 8
    yp, yq = _logits(rng, V, 1.2), _logits(rng, V, 1.2)
    Tf = np.float64(np.float32(T))
    p = softmax(yp.astype(np.float64) / Tf)
    q = softmax(yq.astype(np.float64) / Tf)
    B = N_MC
    x = rng.choice(V, size=B, p=q).astype(np.int32)[:, None]
    tgt = _tile([yp, yp], B)
    dr = _tile([yq], B)
    n, bonus, _ = orc.accept(tgt, dr, x, np.ones(B, np.int32), np.full(B, T, np.float32), seed=77)
    beta = np.minimum(p, q).sum()
    assert abs(n.mean() - beta) <= 4 * np.sqrt(beta * (1 - beta) / B)
    first = np.where(n == 1, x[:, 0], bonus)
    assert _chi2_ok(np.bincount(first, minlength=V), p)


def test_bonus_draw_law_with_nothing_to_verify(orc):
    rng = np.random.default_rng(23)
    V = 12
    yp = _logits(rng, V, 2.0)
    B = N_MC
    tgt = _tile([yp], B)
    dr = np.zeros((B, 0, V), np.float32)
    tok = np.zeros((B, 0), np.int32)
    n, bonus, _ = orc.accept(tgt, dr, tok, np.zeros(B, np.int32), np.full(B, 0.9, np.float32), seed=3)
    assert np.all(n == 0)
    assert _chi2_ok(np.bincount(bonus, minlength=V), softmax(yp.astype(np.float64) / np.float64(np.float32(0.9))))


def test_expected_accepted_count_is_sum_of_prefix_products(orc):
    rng = np.random.default_rng(24)
    V, K = 6, 3
    B = N_MC
    yps = [_logits(rng, V, s) for s in (0.5, 1.0, 2.0, 1.0)]
    yqs = [_logits(rng, V, s) for s in (0.5, 1.0, 2.0)]
    p = [softmax(y.astype(np.float64)) for y in yps]
    q = [softmax(y.astype(np.float64)) for y in yqs]
    x = np.stack([rng.choice(V, size=B, p=q[j]) for j in range(K)], 1).astype(np.int32)
    n, _, _ = orc.accept(_tile(yps, B), _tile(yqs, B), x, np.full(B, K, np.int32),
                         np.ones(B, np.float32), seed=11)
    beta = [np.minimum(p[j], q[j]).sum() for j in range(K)]
    expect = sum(np.prod(beta[: j + 1]) for j in range(K))
    sd = n.std() / np.sqrt(B)
    assert abs(n.mean() - expect) <= 4 * sd


def test_sequence_offset_reproduces_unsplit_batch(orc):
    rng = np.random.default_rng(25)
    B, K, V = 10, 4, 16
    tgt = (rng.standard_normal((B, K + 1, V)) * 2).astype(np.float32)
    dr = (tgt[:, :K] + rng.standard_normal((B, K, V))).astype(np.float32)
    tok = rng.integers(0, V, size=(B, K)).astype(np.int32)
    L = rng.integers(0, K + 1, size=B).astype(np.int32)
    T = np.where(np.arange(B) % 2 == 0, 0.0, 0.9).astype(np.float32)
    full = orc.accept(tgt, dr, tok, L, T, seed=123, round_offset=4)
    lo = orc.accept(tgt[:6], dr[:6], tok[:6], L[:6], T[:6], seed=123, round_offset=4)
    hi = orc.accept(tgt[6:], dr[6:], tok[6:], L[6:], T[6:], seed=123, round_offset=4, seq_offset=6)
    for i in range(3):
        np.testing.assert_array_equal(full[i], np.concatenate([lo[i], hi[i]]))
    # another round draws other numbers
    other = orc.accept(tgt, dr, tok, L, T, seed=123, round_offset=5)
    assert not (np.array_equal(full[0], other[0]) and np.array_equal(full[1], other[1]))


def test_rejects_bad_lengths(orc):
    tgt = np.zeros((1, 3, 4), np.float32)
    dr = np.zeros((1, 2, 4), np.float32)
    with pytest.raises(orc.OracleError):
        orc.accept(tgt, dr, np.zeros((1, 2), np.int32), np.array([3], np.int32), np.zeros(1, np.float32), 0)
    with pytest.raises(orc.OracleError):
        orc.accept(tgt, dr, np.full((1, 2), 4, np.int32), np.array([2], np.int32), np.zeros(1, np.float32), 0)


def test_bonus_after_full_acceptance_follows_last_row(orc):
    # drafter == target on rows 0..1, so every draft is accepted (ratio 1) and
    # the emitted token is drawn from the bonus row L_b = 2, not from row 0
    rng = np.random.default_rng(26)
    V, K = 10, 2
    B = N_MC // 2
    y0, y1, y2 = _logits(rng, V), _logits(rng, V), _logits(rng, V, 2.5)
    tok = np.stack([rng.choice(V, size=B, p=softmax(y0.astype(np.float64))),
                    rng.choice(V, size=B, p=softmax(y1.astype(np.float64)))], 1).astype(np.int32)
    n, bonus, _ = orc.accept(_tile([y0, y1, y2], B), _tile([y0, y1], B), tok, np.full(B, K, np.int32),
                             np.ones(B, np.float32), seed=8)
    assert np.all(n == K)
    assert _chi2_ok(np.bincount(bonus, minlength=V), softmax(y2.astype(np.float64)))
    assert not _chi2_ok(np.bincount(bonus, minlength=V), softmax(y0.astype(np.float64)))
