"""Seeded synthetic inputs for the verify round, shaped like the paper's workloads.

The paper evaluates on Qwen2.5 / Qwen3 targets with diffusion drafters over
MATH-500, GSM8K, HumanEval and MT-Bench (Sec. 4, Table 5). Neither the models
nor the datasets are used here: these generators stand in for them with the
same tensor shapes (vocabularies 32000 / 128256 / 152064, GQA 8/2, 32/8, 28/4,
64/8, head dim 64 / 128), logit value distributions chosen so that the
selected lengths span 0..K, and KV-length mixes from uniform to log-uniform.

This module holds none of the verify round's arithmetic. It draws random
tensors with ``torch`` generators and is the only code shared by the CUDA path
and the CPU oracle in tests and benchmarks.
"""
from __future__ import annotations

import dataclasses
import json
import math
import os
from typing import List, Optional

import numpy as np
import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    B: int                 # sequences
    K: int                 # drafter block length (= d_max of the selector)
    V: int                 # vocabulary
    Hq: int                # query heads
    Hkv: int               # kv heads
    d: int                 # head dim
    n_layers: int          # verify-attention layers per round
    kv: tuple              # ("const", n) | ("uniform", lo, hi) | ("loguniform", lo, hi)
    temperature: tuple     # ("const", T) | ("alternate", T_even, T_odd)
    target: tuple          # ("normal", sigma) | ("normal_peak", sigma, peak) | ("normal_sigma_u", lo, hi)
    draft_noise: tuple     # ("const", s) | ("uniform", lo, hi)
    cost: tuple            # ("poly", c0, c1, c2) | ("measured", file) | ("attn_bytes",)
    philox_seed: int
    data_seed: int
    resident_layers: int = 0   # >0: distinct KV buffers kept on the device (rest reuse them)
    hidden: int = 4096         # model dimension of the LM head (Llama-3-8B / 70B: 4096 / 8192, Qwen2.5-7B 3584)

    def scaled(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


# The five workloads (batch 1..64). Values their shapes leave open (data seeds
# of the larger configs, the sampling config's target sigma, the ragged
# config's odd-sequence temperature and drafter noise, layer counts of the
# single-layer configs) are fixed here once.
WORKLOADS = {
    "tiny": Workload("tiny", B=1, K=16, V=32000, Hq=8, Hkv=2, d=64, n_layers=1,
                     kv=("const", 512), temperature=("const", 0.0), target=("normal", 4.0),
                     draft_noise=("const", 1.0), cost=("poly", 1.0, 0.02, 0.0),
                     philox_seed=0, data_seed=0),
    "8b": Workload("8b", B=1, K=16, V=128256, Hq=32, Hkv=8, d=128, n_layers=32,
                   kv=("const", 4096), temperature=("const", 0.0), target=("normal_peak", 6.0, 12.0),
                   draft_noise=("const", 1.5), cost=("poly", 1.0, 0.01, 0.0),
                   philox_seed=1, data_seed=1, hidden=4096),
    "sampling": Workload("sampling", B=16, K=16, V=152064, Hq=28, Hkv=4, d=128, n_layers=1,
                         kv=("uniform", 1024, 8192), temperature=("const", 1.0), target=("normal", 4.0),
                         draft_noise=("uniform", 0.5, 3.0), cost=("poly", 1.0, 0.015, 0.0005),
                         philox_seed=1234, data_seed=2, hidden=3584),
    "ragged": Workload("ragged", B=64, K=32, V=128256, Hq=32, Hkv=8, d=128, n_layers=1,
                       kv=("loguniform", 512, 32768), temperature=("alternate", 0.0, 0.8),
                       target=("normal_sigma_u", 1.0, 8.0), draft_noise=("const", 1.0),
                       cost=("measured", "ragged_verify_attn_cost.json"), philox_seed=3, data_seed=3),
    "70b": Workload("70b", B=8, K=16, V=128256, Hq=64, Hkv=8, d=128, n_layers=80,
                    kv=("const", 131072), temperature=("const", 0.7), target=("normal", 4.0),
                    draft_noise=("const", 1.0), cost=("poly", 1.0, 0.008, 0.0),
                    philox_seed=4, data_seed=4, resident_layers=16, hidden=8192),
}


def _np_rng(w: Workload, stream: int) -> np.random.Generator:
    return np.random.default_rng([w.data_seed, stream])


def kv_lengths(w: Workload) -> np.ndarray:
    """Per-sequence KV-cache length before the verified block, int32 [B]."""
    kind = w.kv[0]
    rng = _np_rng(w, 1)
    if kind == "const":
        out = np.full(w.B, w.kv[1])
    elif kind == "uniform":
        out = rng.integers(w.kv[1], w.kv[2] + 1, size=w.B)
    elif kind == "loguniform":
        lo, hi = math.log(w.kv[1]), math.log(w.kv[2])
        out = np.floor(np.exp(rng.uniform(lo, hi, size=w.B))).astype(np.int64)
        out = np.clip(out, w.kv[1], w.kv[2])
    else:
        raise ValueError(kind)
    return out.astype(np.int32)


def temperatures(w: Workload) -> np.ndarray:
    """Per-sequence temperature, float32 [B]; 0 means greedy decoding."""
    if w.temperature[0] == "const":
        return np.full(w.B, w.temperature[1], np.float32)
    even, odd = w.temperature[1], w.temperature[2]
    return np.array([even if b % 2 == 0 else odd for b in range(w.B)], np.float32)


def s_cap(w: Workload, kv: Optional[np.ndarray] = None) -> int:
    """Cache capacity per (sequence, kv head): room for the block, rounded to 64."""
    kv = kv_lengths(w) if kv is None else kv
    need = int(kv.max()) + w.K + 1
    return (need + 63) // 64 * 64


def attn_bytes(w: Workload, kv: np.ndarray, L) -> float:
    """Bytes one verify-attention layer must move: K and V of the visible keys
    plus Q read and O written for the verified rows (bf16)."""
    L = np.broadcast_to(np.asarray(L, np.int64), kv.shape)
    keys = kv.astype(np.int64) + L + 1
    rows = L + 1
    return float(np.sum(w.Hkv * keys * w.d * 2 * 2 + rows * w.Hq * w.d * 2 * 2))


# Fixed per-launch latency folded into the byte-count cost model, expressed
# in bytes at the measured copy bandwidth (about 3 us at 6.76 TB/s).
_LAUNCH_BYTES = 3e-6 * 6.756e12
_DATA = os.path.join(os.path.dirname(os.path.abspath(__file__)), "data")


def cost_table(w: Workload, kv: Optional[np.ndarray] = None) -> np.ndarray:
    """T_verify(L) for L = 0..K, float32 [K+1], positive.

    Polynomial tables are the workloads' stated ones. A measured table (the
    ragged workload's) is the verify-attention kernel's own latency with
    every sequence at length L, frozen to JSON by ``measure_cost_table``
    (normalised to T(0) = 1, running maximum). ``attn_bytes`` models one
    launch as a fixed latency plus the bytes it must move at a fixed
    bandwidth (normalised, running maximum); it is also the fallback of a
    measured table whose file is missing."""
    Ls = np.arange(w.K + 1)
    kind = w.cost[0]
    if kind == "measured":
        path = os.path.join(_DATA, w.cost[1])
        if os.path.exists(path):
            with open(path) as f:
                rec = json.load(f)
            t = np.asarray(rec["T"], np.float64)
            if t.shape != (w.K + 1,):
                raise ValueError("%s holds %d entries, the workload needs %d" % (path, t.size, w.K + 1))
            return t.astype(np.float32)
        kind = "attn_bytes"
    if kind == "poly":
        c0, c1, c2 = w.cost[1:]
        t = c0 + c1 * Ls + c2 * Ls * Ls
    elif kind == "attn_bytes":
        kv = kv_lengths(w) if kv is None else kv
        t = np.array([_LAUNCH_BYTES + attn_bytes(w, kv, L) for L in Ls])
        t = t / t[0]
        t = np.maximum.accumulate(t)
    else:
        raise ValueError(w.cost[0])
    return t.astype(np.float32)


def _randn(shape, gen, device, dtype=torch.float32):
    return torch.randn(shape, generator=gen, device=device, dtype=dtype)


def logits(w: Workload, device="cpu") -> dict:
    """Target logits [B,K+1,V], drafter logits [B,K,V] (fp32), draft tokens
    [B,K] (int32) and temperatures [B] (fp32) on ``device``.

    Drafter logits are the target's plus Gaussian noise (the drafter is close
    to the target). Greedy sequences draft the drafter's argmax; sampling
    sequences draft a token sampled from the drafter's softmax at their
    temperature (Gumbel-max with the torch generator), so that the rejection
    sampler sees drafts distributed as q.

    The values are drawn on the host with torch's CPU generator whatever the
    device, then moved there, so every consumer (the GPU path, the oracle, the
    reference arm of the benchmark) sees the same tensors for a workload."""
    out_device = device
    device = "cpu"
    g = torch.Generator(device=device)
    g.manual_seed(w.data_seed * 1000003 + 17)
    B, K, V = w.B, w.K, w.V
    rng = _np_rng(w, 2)
    kind = w.target[0]
    if kind == "normal":
        sig = np.full(B, w.target[1])
    elif kind == "normal_peak":
        sig = np.full(B, w.target[1])
    elif kind == "normal_sigma_u":
        sig = rng.uniform(w.target[1], w.target[2], size=B)
    else:
        raise ValueError(kind)
    if w.draft_noise[0] == "const":
        noise = np.full(B, w.draft_noise[1])
    else:
        noise = rng.uniform(w.draft_noise[1], w.draft_noise[2], size=B)
    sig_t = torch.tensor(sig, dtype=torch.float32, device=device).view(B, 1, 1)
    noise_t = torch.tensor(noise, dtype=torch.float32, device=device).view(B, 1, 1)
    target = _randn((B, K + 1, V), g, device) * sig_t
    if kind == "normal_peak":
        idx = torch.randint(0, V, (B, K + 1, 1), generator=g, device=device)
        target.scatter_add_(2, idx, torch.full((B, K + 1, 1), float(w.target[2]), device=device))
    draft = target[:, :K, :] + _randn((B, K, V), g, device) * noise_t
    temp = torch.tensor(temperatures(w), device=device)
    tokens = torch.empty((B, K), dtype=torch.int32, device=device)
    for b in range(B):
        T = float(temp[b])
        if T == 0.0:
            tokens[b] = torch.argmax(draft[b], dim=-1).to(torch.int32)
        else:
            u = torch.rand((K, V), generator=g, device=device).clamp_(1e-30, 1.0 - 1e-7)
            gumbel = -torch.log(-torch.log(u))
            tokens[b] = torch.argmax(draft[b] / T + gumbel, dim=-1).to(torch.int32)
    out = {"target_logits": target, "draft_logits": draft, "draft_tokens": tokens, "temperature": temp}
    return {k: v.contiguous().to(out_device) for k, v in out.items()}


def layer(w: Workload, l: int, kv: np.ndarray, device="cpu", peaky: bool = False,
          scap: Optional[int] = None) -> dict:
    """Q [B,K+1,Hq,d] and the KV cache Kc, Vc [B,Hkv,S_cap,d] (bf16, ~N(0,1))
    of verify-attention layer ``l``, each layer seeded independently.

    ``peaky``: plant, for every (sequence, query head), one key equal to 3x
    the head's first verified query so that one score dominates its row."""
    g = torch.Generator(device=device)
    g.manual_seed(w.data_seed * 7919 + 1000 + l)
    S = s_cap(w, kv) if scap is None else scap
    B, K1 = w.B, w.K + 1
    Q = _randn((B, K1, w.Hq, w.d), g, device, torch.bfloat16)
    Kc = _randn((B, w.Hkv, S, w.d), g, device, torch.bfloat16)
    Vc = _randn((B, w.Hkv, S, w.d), g, device, torch.bfloat16)
    if peaky:
        gsz = w.Hq // w.Hkv
        for b in range(B):
            for h in range(w.Hq):
                pos = int(torch.randint(0, int(kv[b]), (1,), generator=g, device=device))
                Kc[b, h // gsz, pos] = (Q[b, 0, h].float() * 3.0).to(torch.bfloat16)
    return {"Q": Q, "Kc": Kc, "Vc": Vc}


def draft_tree(B: int, K: int, L, seed: int, shape: str = "topk", depth: int = 16) -> np.ndarray:
    """Parent array [B, K+1] (int32) of a draft tree per sequence.

    Node 0 is the root (the last accepted token); node t in [1, L_b] has
    parent[b, t] in [0, t), so node numbers are a topological order; entries
    t > L_b and the root's are 0. Shapes: ``chain`` (parent t-1, the chain
    draft), ``star`` (every node a child of the root), ``random`` (uniform
    recursive tree) and ``topk``: the shape tree drafters grow from
    per-position candidate lists, a main path with up to three alternatives
    hanging off each depth (breadth-first: depth by depth, candidates in rank
    order, each alternative a child of the previous depth's best node);
    ``ddtree``: the shape a diffusion drafter's tree takes under a node budget
    (DDTree): per depth d <= ``depth`` (the block length) a ranked candidate
    list with probabilities q_d (softmax of N(0, s^2) scores, s per sequence
    in [1, 6]); nodes are added best-first by the product of the
    candidates' probabilities along the path (a child of node t is candidate
    k at depth(t) + 1), so a confident drafter grows one long path and an
    unsure one a bushy top."""
    rng = np.random.default_rng([seed, 77])
    L = np.broadcast_to(np.asarray(L, np.int64), (B,))
    par = np.zeros((B, K + 1), np.int32)
    for b in range(B):
        n = int(L[b])
        if shape == "chain":
            par[b, 1:n + 1] = np.arange(0, n)
        elif shape == "star":
            par[b, 1:n + 1] = 0
        elif shape == "random":
            for t in range(1, n + 1):
                par[b, t] = rng.integers(0, t)
        elif shape == "topk":
            t, best = 1, 0
            while t <= n:
                width = int(rng.integers(1, 5))
                first = t
                for _ in range(width):
                    if t > n:
                        break
                    par[b, t] = best
                    t += 1
                best = first
        elif shape == "ddtree":
            par[b] = _ddtree_parents(rng, n, K, depth)
        else:
            raise ValueError(shape)
    return par


def _ddtree_parents(rng: np.random.Generator, n: int, K: int, depth: int) -> np.ndarray:
    import heapq

    width = 32
    s = rng.uniform(1.0, 6.0)
    z = rng.standard_normal((depth + 1, width)) * s
    q = np.exp(z - z.max(axis=1, keepdims=True))
    q = -np.sort(-q / q.sum(axis=1, keepdims=True), axis=1)   # ranked, descending
    logq = np.log(q)
    out = np.zeros(K + 1, np.int32)
    node_depth = [0]
    # candidates: (-path log-prob, tie, parent node, rank at depth(parent)+1)
    heap = [(-logq[1, 0], 0, 0, 0)]
    tie, t = 1, 1
    while t <= n and heap:
        neg, _, p, k = heapq.heappop(heap)
        out[t] = p
        d = node_depth[p] + 1
        node_depth.append(d)
        if k + 1 < width:      # the next sibling candidate
            heapq.heappush(heap, (neg + logq[d, k] - logq[d, k + 1], tie, p, k + 1))
            tie += 1
        if d < depth:          # the first child candidate of the new node
            heapq.heappush(heap, (neg - logq[d + 1, 0], tie, t, 0))
            tie += 1
        t += 1
    return out


def tree_logits(w: Workload, parent: np.ndarray, L, device="cpu", p_follow: float = 0.8) -> dict:
    """Draft tokens [B, N] (int32) and target logits [B, N+1, V] (f32) of draft trees.

    Siblings carry distinct random tokens. Node p's target row is N(0, 4^2)
    with +12 at one token: with probability ``p_follow`` (when p has
    children) the token of its lowest-numbered child (the drafter's
    best-ranked candidate), else a uniformly random token."""
    B, N1 = parent.shape
    N = N1 - 1
    L = np.broadcast_to(np.asarray(L, np.int64), (B,))
    rng = np.random.default_rng([w.data_seed, 91])
    tok = np.zeros((B, N), np.int32)
    peak = np.zeros((B, N1), np.int64)
    for b in range(B):
        kids = [[] for _ in range(N1)]
        for t in range(1, int(L[b]) + 1):
            kids[int(parent[b, t])].append(t)
        for p in range(N1):
            if kids[p]:
                vals = rng.choice(w.V, size=len(kids[p]), replace=False)
                for t, v in zip(kids[p], vals):
                    tok[b, t - 1] = v
            if kids[p] and rng.random() < p_follow:
                peak[b, p] = tok[b, kids[p][0] - 1]
            else:
                peak[b, p] = rng.integers(0, w.V)
    g = torch.Generator(device=device)
    g.manual_seed(w.data_seed * 7919 + 77)
    target = _randn((B, N1, w.V), g, device) * 4.0
    idx = torch.from_numpy(peak).to(device)
    target.scatter_add_(2, idx[:, :, None], torch.full((B, N1, 1), 12.0, device=device))
    return {"draft_tokens": torch.from_numpy(tok).to(device), "target_logits": target.contiguous()}


def lm_head(w: Workload, rows: int, device="cpu", sigma: float = 4.0) -> dict:
    """Hidden states H [rows, hidden] ~ N(0, 1) and LM-head weights W [V, hidden] ~ N(0, sigma^2 / hidden),
    bf16, so that logits are ~ N(0, sigma^2)."""
    g = torch.Generator(device=device)
    g.manual_seed(w.data_seed * 7919 + 555)
    H = _randn((rows, w.hidden), g, device).to(torch.bfloat16)
    W = (_randn((w.V, w.hidden), g, device) * (sigma / w.hidden ** 0.5)).to(torch.bfloat16)
    return {"H": H, "W": W}


def reference_inputs_summary(w: Workload) -> List[str]:
    """One line per input recipe, for reports."""
    return [
        "target logits %s, drafter = target + N(0, %s^2)" % (w.target, w.draft_noise),
        "kv lengths %s, %d layer(s), GQA %d/%d, head dim %d" % (w.kv, w.n_layers, w.Hq, w.Hkv, w.d),
        "temperature %s, cost %s, philox seed %d, data seed %d" % (w.temperature, w.cost, w.philox_seed,
                                                                    w.data_seed),
    ]
