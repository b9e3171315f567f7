"""Host logic of the benchmark: the algorithmic bytes and flops its roofline
divides by (no GPU)."""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2608_08721_gb300 import workloads  # noqa: E402


def test_round_bytes_of_a_chain_round():
    w = workloads.WORKLOADS["8b"]
    kv = workloads.kv_lengths(w)
    L = np.array([4])
    by = bench.round_bytes(w, kv, L, np.zeros(1), np.array([4]))
    assert by["conf"] == w.B * w.K * w.V * 4
    assert by["accept"] == 5 * w.V * 4                      # rows 0..L of the target, greedy
    per_layer = w.Hkv * (4096 + 5) * w.d * 2 * 2 + 5 * w.Hq * w.d * 2 * 2
    assert by["attn_per_launch"] == per_layer
    assert by["total"] == by["conf"] + by["select"] + by["accept"] + per_layer * w.n_layers
    # a rejected sampling sequence reads its residual's two rows again
    by2 = bench.round_bytes(w, kv, L, np.ones(1), np.array([2]))
    assert by2["accept"] == by["accept"] + 2 * w.V * 4
    # bf16 logits halve the logits bytes
    assert bench.round_bytes(w, kv, L, np.zeros(1), np.array([4]), logit_bytes=2)["conf"] == by["conf"] // 2


def test_round_bytes_of_a_tree_reads_every_node_row():
    w = workloads.WORKLOADS["8b"]
    kv = workloads.kv_lengths(w)
    by = bench.round_bytes(w, kv, np.array([4]), np.zeros(1), np.array([0]), L_tree=np.array([64]))
    assert by["accept"] == 65 * w.V * 4
    assert by["attn_per_launch"] == w.Hkv * (4096 + 65) * w.d * 4 + 65 * w.Hq * w.d * 4


def test_tree_flops_count_visible_keys_only():
    kv = np.array([100, 7])
    N = 9
    chain = workloads.draft_tree(2, N, N, seed=0, shape="chain")
    star = workloads.draft_tree(2, N, N, seed=0, shape="star")
    Hq, d = 4, 16
    # chain: node t sees kv + t + 1 keys; star: the root sees kv + 1, every other node kv + 2
    want_chain = sum(Hq * 4 * d * (k + t + 1) for k in kv for t in range(N + 1))
    want_star = sum(Hq * 4 * d * ((k + 1) + N * (k + 2)) for k in kv)
    assert bench.tree_flops(chain, kv, np.full(2, N), Hq, d) == want_chain
    assert bench.tree_flops(star, kv, np.full(2, N), Hq, d) == want_star
