"""Pins of the oracle's length selector.

* Exact brute force: with a positive, convex cost table (non-decreasing
  marginal cost) the scan must return the smallest argmax over L of
  E[eta_L] = E_L / T(L) (Eq. 2 with negligible drafting; Thm. 4's
  unimodality), evaluated here in exact rational arithmetic.
* Thm. 5: iterated single beneficial adjustments started at 0 and at K
  strictly increase E[eta] at every step and end at that argmax.
* Closed forms and invariants: q = 1 with a linear table; q_1 = 0; scaling the
  table by a power of two; the hand-worked fixture in tests/golden.
"""
import json
import os
from fractions import Fraction

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _exact_eta(q, cost, L, e0=1):
    P, E = Fraction(1), Fraction(e0)
    for j in range(L):
        P *= Fraction(float(q[j]))
        E += P
    return E / Fraction(float(cost[L]))


def _exact_argmax(q, cost, e0=1):
    K = len(q)
    vals = [_exact_eta(q, cost, L, e0) for L in range(K + 1)]
    best = max(vals)
    return vals.index(best), vals


def _convex_cost(rng, K):
    c0 = rng.uniform(0.5, 2.0)
    marg = np.sort(rng.uniform(0.0, 0.3, size=K))  # non-decreasing marginal cost
    return np.concatenate([[c0], c0 + np.cumsum(marg)])


@pytest.mark.parametrize("K", [1, 2, 3, 5, 8])
def test_scan_equals_exact_bruteforce_argmax(orc, K):
    rng = np.random.default_rng(100 + K)
    n_cases, flagged = 400, 0
    for case in range(n_cases):
        kind = case % 4
        if kind == 0:
            q = rng.uniform(0, 1, size=K)
        elif kind == 1:
            q = 1 - rng.uniform(0, 1, size=K) ** 4          # confident drafter
        elif kind == 2:
            q = rng.uniform(0, 1, size=K) ** 4              # weak drafter
        else:
            q = rng.choice([0.0, 0.25, 0.5, 1.0], size=K)   # adversarial: exact ties, zeros
        cost = _convex_cost(rng, K) if case % 5 else 1.0 + 0.25 * np.arange(K + 1)
        L, flag = orc.select_lengths(q[None, :], cost)
        best, vals = _exact_argmax(q, cost)
        if flag[0]:
            flagged += 1
            # a flagged decision may go either way, but must be a maximiser
            # up to the flag tolerance
            assert float(vals[int(L[0])]) >= float(vals[best]) * (1 - 1e-5)
            continue
        assert int(L[0]) == best, (q, cost, vals)
    assert flagged < n_cases // 4


@pytest.mark.parametrize("K", [3, 6, 10])
def test_iterated_adjustments_converge_monotonically(orc, K):
    rng = np.random.default_rng(7 + K)
    for _ in range(150):
        q = rng.uniform(0, 1, size=K) ** rng.uniform(0.2, 3)
        cost = _convex_cost(rng, K)
        cost = cost + np.arange(K + 1) * 1e-3       # strictly increasing
        best, vals = _exact_argmax(q, cost)
        for start in (0, K, int(rng.integers(0, K + 1))):
            path = orc.select_iterate(q, cost, start)
            assert path[0] == start
            etas = [vals[d] for d in path]
            assert all(b > a for a, b in zip(etas, etas[1:])), "Def. 1: every step raises E[eta]"
            assert all(abs(b - a) == 1 for a, b in zip(path, path[1:]))
            # Thm. 5: ends in the optimal set (exact ties may stop at any maximiser)
            assert vals[path[-1]] == vals[best]
            # unimodality: the walk never reverses direction
            steps = np.sign(np.diff(path))
            assert len(set(steps.tolist())) <= 1


def test_iterate_from_scan_result_does_not_move(orc):
    rng = np.random.default_rng(3)
    for _ in range(100):
        K = 12
        q = rng.uniform(0, 1, size=K) ** 0.5
        cost = 1.0 + 0.05 * np.arange(K + 1) + 0.002 * np.arange(K + 1) ** 2
        L, flag = orc.select_lengths(q[None, :], cost)
        if flag[0]:
            continue
        assert orc.select_iterate(q, cost, int(L[0])) == [int(L[0])]


@pytest.mark.parametrize("a,c,expect", [(1.0, 0.5, "K"), (1.0, 2.0, 0), (3.0, 0.25, "K"), (0.5, 0.75, 0)])
def test_all_confident_linear_cost_closed_form(orc, a, c, expect):
    # q = 1: E_L = 1 + L, T(L) = a + cL; extending from L is beneficial iff
    # (a + cL) > c (1 + L), i.e. iff a > c, for every L.
    K = 10
    q = np.ones((1, K))
    cost = a + c * np.arange(K + 1)
    L, flag = orc.select_lengths(q, cost)
    assert int(L[0]) == (K if expect == "K" else expect)
    assert flag[0] == 0


def test_exact_tie_does_not_extend_and_is_flagged(orc):
    K = 6
    q = np.ones((1, K))
    cost = 1.0 + 1.0 * np.arange(K + 1)      # a == c: every step is a tie
    L, flag = orc.select_lengths(q, cost)
    assert int(L[0]) == 0 and flag[0] == 1


def test_zero_first_confidence_gives_zero_length(orc):
    q = np.array([[0.0, 1.0, 1.0, 1.0]])
    L, _ = orc.select_lengths(q, 1.0 + 0.01 * np.arange(5))
    assert int(L[0]) == 0


def test_zero_marginal_cost_extends_while_probability_positive(orc):
    q = np.array([[0.5, 0.5, 0.0, 1.0]])
    L, _ = orc.select_lengths(q, np.ones(5))
    assert int(L[0]) == 2


@pytest.mark.parametrize("k", [-3, 1, 5])
def test_power_of_two_cost_scaling_is_invariant(orc, k):
    rng = np.random.default_rng(11)
    q = rng.uniform(0, 1, size=(200, 16)) ** 0.3
    cost = 1.0 + 0.015 * np.arange(17) + 0.0005 * np.arange(17) ** 2
    L1, f1 = orc.select_lengths(q, cost)
    L2, f2 = orc.select_lengths(q, cost * 2.0**k)
    np.testing.assert_array_equal(L1, L2)
    np.testing.assert_array_equal(f1, f2)


def test_longer_prefix_of_confident_tokens_never_shortens(orc):
    # raising one confidence never lowers the product at any later position,
    # so the selected length cannot drop
    rng = np.random.default_rng(12)
    cost = 1.0 + 0.02 * np.arange(9)
    for _ in range(200):
        q = rng.uniform(0, 1, size=8)
        j = int(rng.integers(0, 8))
        q2 = q.copy()
        q2[j] = min(1.0, q[j] + rng.uniform(0, 0.5))
        L1, f1 = orc.select_lengths(q[None], cost)
        L2, f2 = orc.select_lengths(q2[None], cost)
        if f1[0] or f2[0]:
            continue
        assert L2[0] >= L1[0]


def test_golden_worked_example(orc):
    with open(os.path.join(GOLDEN, "select_worked.json")) as f:
        gold = json.load(f)
    for case in gold["cases"]:
        q = np.array([case["q"]])
        L, flag = orc.select_lengths(q, np.array(case["cost_table"]), e0=case.get("e0", 1.0))
        assert int(L[0]) == case["L"], case["name"]
        assert int(flag[0]) == 0


def test_bonus_reading_switch(orc):
    # with e0 = 0 the first extension is beneficial whenever q_1 > 0
    q = np.array([[1e-9, 0.0]])
    cost = np.array([1.0, 100.0, 200.0])
    assert int(orc.select_lengths(q, cost, e0=0.0)[0][0]) == 1
    assert int(orc.select_lengths(q, cost, e0=1.0)[0][0]) == 0


def test_rejects_nonpositive_cost(orc):
    with pytest.raises(orc.OracleError):
        orc.select_lengths(np.ones((1, 2)), np.array([1.0, 0.0, 1.0]))
    with pytest.raises(orc.OracleError):
        orc.select_lengths(np.ones((1, 2)), np.array([1.0, np.inf, 1.0]))
