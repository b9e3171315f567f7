"""Pins of the oracle's alpha-mode length search (Algorithm 1; the
position-wise bounds of Thm. 2 / Thm. 3 weighted by alpha, Sec. 4 uses
alpha = 2.0 / 2.2).

eps_i = floor(alpha * sum_{j=i}^{d} prod_{k=i}^{j} q_k + i), eps* = min_i eps_i;
from d = n (one drafted block) while d < d_max: eps* <= d rolls back once and
stops, else d = eps* (clamped to d_max) and blocks are drafted to cover it.
The pins use closed forms and hand-worked cases, not the oracle's own sums."""
import math

import numpy as np
import pytest

import oracle


def test_hand_worked_rollback_example():
    # q = 0.9, 0.5, 0.2, 0.9 ... ; n = 2, alpha = 2.
    # d = 2: eps_1 = floor(2 (0.9 + 0.45) + 1) = floor(3.7) = 3,
    #        eps_2 = floor(2 * 0.5 + 2) = 3            -> eps* = 3 > 2: extend,
    #        budget 0 - 1 = -1 -> one more block (blocks = 2, budget 1).
    # d = 3: eps_1 = floor(2 (0.9 + 0.45 + 0.09) + 1) = floor(3.88) = 3,
    #        eps_2 = floor(2 (0.5 + 0.1) + 2) = floor(3.2) = 3,
    #        eps_3 = floor(2 * 0.2 + 3) = floor(3.4) = 3  -> eps* = 3 <= 3: stop.
    q = np.array([[0.9, 0.5, 0.2, 0.9, 0.9, 0.9, 0.9, 0.9]])
    L, blocks, _ = oracle.select_alpha(q, 2, 2.0)
    assert L.tolist() == [3] and blocks.tolist() == [2]


def test_hand_worked_shrink_below_block():
    # n = 4 with q = 0.3, 0.1, 0.9, 0.9 ..., alpha = 2.2, d_max = 6:
    # eps_1 = floor(2.2 (0.3 + 0.03 + 0.027 + 0.0243) + 1) = floor(1.83746) = 1
    # -> eps* = 1 <= 4: the single rollback to d = 1 (no block drafted).
    q = np.array([[0.3, 0.1, 0.9, 0.9, 0.9, 0.9]])
    L, blocks, _ = oracle.select_alpha(q, 4, 2.2)
    assert L.tolist() == [1] and blocks.tolist() == [1]


def _geometric_eps_star(c, d, alpha):
    # sum_{j=i}^{d} c^(j-i+1) = c (1 - c^m) / (1 - c), m = d - i + 1
    best = None
    for i in range(1, d + 1):
        m = d - i + 1
        S = m if c == 1.0 else c * (1.0 - c ** m) / (1.0 - c)
        e = math.floor(alpha * S + i)
        best = e if best is None else min(best, e)
    return best


@pytest.mark.parametrize("c", [0.35, 0.6, 0.8, 0.93, 0.99])
@pytest.mark.parametrize("alpha", [1.3, 2.0, 2.2, 3.7])
@pytest.mark.parametrize("n,K", [(1, 8), (3, 16), (8, 16), (16, 24), (5, 40)])
def test_constant_confidence_matches_geometric_closed_form(c, alpha, n, K):
    # Algorithm 1's control flow with the sums in closed form (geometric series)
    d, blocks, budget = n, 1, 0
    while d < K:
        e = _geometric_eps_star(c, d, alpha)
        if e <= d:
            d = e
            break
        e = min(e, K)
        budget -= e - d
        d = e
        if budget < 0:
            more = -(-(-budget) // n)
            blocks += more
            budget += more * n
    L, b, flag = oracle.select_alpha(np.full((1, K), c), n, alpha)
    if not flag[0]:
        assert (int(L[0]), int(b[0])) == (d, blocks)


@pytest.mark.parametrize("n,K", [(1, 8), (4, 16), (16, 24), (7, 64)])
def test_full_confidence_runs_to_dmax_with_minimal_blocks(n, K):
    # q = 1: sum = d - i + 1, eps_i = floor(alpha (d - i + 1) + i) >= d + floor(alpha)
    # for alpha >= 1, so d only grows; the blocks drafted just cover d_max.
    L, blocks, _ = oracle.select_alpha(np.ones((1, K)), n, 2.2)
    assert int(L[0]) == K and int(blocks[0]) == -(-K // n)


@pytest.mark.parametrize("n,K", [(1, 8), (4, 16), (16, 24)])
def test_zero_confidence_rolls_back_to_one(n, K):
    # q = 0: every sum is 0, eps_i = i, eps* = 1 (for n = K the loop never runs)
    L, blocks, _ = oracle.select_alpha(np.zeros((1, K)), n, 2.2)
    expect = K if n == K else 1
    assert int(L[0]) == expect and int(blocks[0]) == 1


def test_tiny_and_huge_alpha():
    rng = np.random.default_rng(3)
    q = rng.uniform(0.05, 0.95, size=(50, 24))
    L, blocks, _ = oracle.select_alpha(q, 16, 1e-9)
    assert np.all(L == 1) and np.all(blocks == 1)  # eps_i = i
    L, blocks, _ = oracle.select_alpha(q, 16, 1e9)
    assert np.all(L == 24) and np.all(blocks == 2)  # every eps_i > d_max: clamp


def test_block_of_ones_then_zeros_rolls_back_past_the_block():
    # q = 1 for the first n positions, 0 after: from d = n, eps* = n + 2
    # (at i = n: 2*1 + n); at d = n + 2, eps_{n+1} = n + 1 (its sum is 0)
    # is the minimum, so the rollback lands on n + 1.
    n, K = 5, 16
    q = np.array([[1.0] * n + [0.0] * (K - n)])
    L, blocks, _ = oracle.select_alpha(q, n, 2.0)
    assert int(L[0]) == n + 1 and int(blocks[0]) == 2


def test_flags_integer_bounds():
    # alpha * S + i exactly an integer: floor and the theorems' ceil(x) - 1 differ
    q = np.array([[0.5, 0.5, 0.5, 0.5]])
    _, _, flag = oracle.select_alpha(q, 1, 2.0)   # eps_1 = floor(2 * 0.5 + 1) = 2 exactly
    assert flag[0] == 1
    _, _, flag = oracle.select_alpha(np.array([[0.37, 0.41, 0.29, 0.33]]), 1, 2.2)
    assert flag[0] == 0


@pytest.mark.parametrize("n,alpha", [(0, 2.0), (5, 2.0), (2, 0.0), (2, -1.0)])
def test_invalid_arguments(n, alpha):
    with pytest.raises(oracle.OracleError):
        oracle.select_alpha(np.full((1, 4), 0.5), n, alpha)
