"""CPU oracle of the LibraSpec verify round (test infrastructure only).

Plain fp64 C (``oracle.c``) behind ``ctypes``. Only the tests, the smoke check
and the benchmark's CPU-baseline leg may import this package. It shares no code
with the CUDA library in ``paper_2608_08721_gb300`` and does not import it.

Every function takes and returns numpy arrays; see ``oracle.c`` for the
definitions and the passages of the paper they follow.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import sys

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")

EINVAL = -1


def build(force: bool = False) -> str:
    """Compile ``oracle.c`` into ``liboracle.so`` with gcc (OpenMP if available)."""
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    base = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off", "-Wall"]
    tmp = _LIB_PATH + ".tmp%d" % os.getpid()
    try:
        subprocess.check_call(base + ["-fopenmp", _SRC, "-o", tmp, "-lm"])
    except subprocess.CalledProcessError:
        print("oracle: building without OpenMP", file=sys.stderr)
        subprocess.check_call(base + [_SRC, "-o", tmp, "-lm"])
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


_lib = None


def _load():
    global _lib
    if _lib is not None:
        return _lib
    build()
    lib = ctypes.CDLL(_LIB_PATH)
    P = ctypes.c_void_p
    i32, u32, u64, f64 = ctypes.c_int, ctypes.c_uint32, ctypes.c_uint64, ctypes.c_double
    lib.oracle_set_threads.argtypes = [i32]
    lib.oracle_get_threads.restype = i32
    lib.oracle_has_openmp.restype = i32
    lib.oracle_philox4x32_10.argtypes = [P, P, P]
    lib.oracle_uniform.argtypes = [u64, u32, u32, u32, u32, u64, i32]
    lib.oracle_uniform.restype = f64
    lib.oracle_confidence.argtypes = [P, P, P, i32, i32, i32, P, P]
    lib.oracle_select_lengths.argtypes = [P, P, i32, i32, f64, P, P]
    lib.oracle_select_iterate.argtypes = [P, P, i32, f64, i32, P, i32]
    lib.oracle_select_alpha.argtypes = [P, i32, i32, i32, f64, P, P, P]
    lib.oracle_gather_pages.argtypes = [P, P, i32, i32, i32, i32, i32, i32, i32, P]
    lib.oracle_verify_attn.argtypes = [P, P, P, P, P, i32, i32, i32, i32, i32, i32, f64, P, P, P, i32]
    lib.oracle_verify_attn_tree.argtypes = [P, P, P, P, P, P, i32, i32, i32, i32, i32, i32, f64, P, P, P, i32]
    lib.oracle_accept.argtypes = [P, P, P, P, P, i32, i32, i32, u64, u64, u32, P, P, P]
    lib.oracle_accept_tree_greedy.argtypes = [P, P, P, P, i32, i32, i32, P, P, P]
    lib.oracle_accept_tree.argtypes = [P, P, P, P, P, i32, i32, i32, u64, u64, u32, P, P, P, P]
    lib.oracle_lm_head_stats.argtypes = [P, P, P, i32, P, i32, i32, i32, P, P, P, P, P]
    for name in ("oracle_confidence", "oracle_select_lengths", "oracle_select_iterate", "oracle_select_alpha",
                 "oracle_gather_pages", "oracle_verify_attn_tree", "oracle_accept_tree_greedy", "oracle_accept_tree", "oracle_lm_head_stats",
                 "oracle_verify_attn", "oracle_accept"):
        getattr(lib, name).restype = i32
    _lib = lib
    return lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


class OracleError(ValueError):
    pass


def _check(rc, what):
    if rc < 0:
        raise OracleError("%s rejected its arguments (status %d)" % (what, rc))
    return rc


def set_threads(n: int) -> None:
    _load().oracle_set_threads(int(n))


def get_threads() -> int:
    return int(_load().oracle_get_threads())


def has_openmp() -> bool:
    return bool(_load().oracle_has_openmp())


def philox4x32_10(counter, key) -> np.ndarray:
    ctr = _c(counter, np.uint32)
    k = _c(key, np.uint32)
    out = np.zeros(4, np.uint32)
    _load().oracle_philox4x32_10(_ptr(ctr), _ptr(k), _ptr(out))
    return out


def uniform(seed, idx, j, seq, purpose, round_offset, word) -> float:
    return float(_load().oracle_uniform(int(seed), int(idx), int(j), int(seq), int(purpose),
                                        int(round_offset), int(word)))


def confidence(draft_logits, draft_tokens, temperature):
    """q[B,K] (fp64) and dstat[B,K,2] = (row max, sum of exp) of the drafter rows."""
    x = _c(draft_logits, np.float32)
    B, K, V = x.shape
    tok = _c(draft_tokens, np.int32)
    T = _c(temperature, np.float32)
    conf = np.zeros((B, K), np.float64)
    dstat = np.zeros((B, K, 2), np.float64)
    _check(_load().oracle_confidence(_ptr(x), _ptr(tok), _ptr(T), B, K, V, _ptr(conf), _ptr(dstat)),
           "oracle_confidence")
    return conf, dstat


def select_lengths(conf, cost_table, e0: float = 1.0):
    """L[B] (int32) and flag[B] from the Thm. 4 scan."""
    q = _c(conf, np.float64)
    B, K = q.shape
    cost = _c(cost_table, np.float64)
    if cost.shape != (K + 1,):
        raise OracleError("cost_table must have K+1 entries")
    L = np.zeros(B, np.int32)
    flag = np.zeros(B, np.int32)
    _check(_load().oracle_select_lengths(_ptr(q), _ptr(cost), B, K, float(e0), _ptr(L), _ptr(flag)),
           "oracle_select_lengths")
    return L, flag


def select_iterate(q, cost_table, start: int, e0: float = 1.0):
    """Lengths visited by iterated single beneficial adjustments from ``start``."""
    qq = _c(q, np.float64)
    K = qq.shape[0]
    cost = _c(cost_table, np.float64)
    cap = 4 * (K + 2)
    path = np.zeros(cap, np.int32)
    n = _check(_load().oracle_select_iterate(_ptr(qq), _ptr(cost), K, float(e0), int(start),
                                             _ptr(path), cap), "oracle_select_iterate")
    return [int(v) for v in path[:n]]


def select_alpha(conf, n: int, alpha: float):
    """Algorithm 1's alpha-mode search: L[B], blocks drafted[B], flag[B] (int32)."""
    q = _c(conf, np.float64)
    B, K = q.shape
    L = np.zeros(B, np.int32)
    blocks = np.zeros(B, np.int32)
    flag = np.zeros(B, np.int32)
    _check(_load().oracle_select_alpha(_ptr(q), B, K, int(n), float(alpha), _ptr(L), _ptr(blocks), _ptr(flag)),
           "oracle_select_alpha")
    return L, blocks, flag


def gather_pages(pool, block_table, S_out: int):
    """Dense [B,Hkv,S_out,d] bf16 bit patterns from a page pool [n_pages,Hkv,P,d] and a block table [B,max_pages]."""
    pb = _as_bf16_bits(pool)
    n_pages, Hkv, P, d = pb.shape
    bt = _c(block_table, np.int32)
    B, max_pages = bt.shape
    dense = np.zeros((B, Hkv, S_out, d), np.uint16)
    _check(_load().oracle_gather_pages(_ptr(pb), _ptr(bt), B, max_pages, P, n_pages, Hkv, d, int(S_out), _ptr(dense)),
           "oracle_gather_pages")
    return dense


def verify_attn_paged(Q, Kp, Vp, block_table, kv_len, L, scale=None, rows=None, fill=np.nan):
    """verify_attn over the dense cache the pages describe."""
    S = int(np.max(np.asarray(kv_len) + np.asarray(L))) + 1 if len(kv_len) else 1
    return verify_attn(Q, gather_pages(Kp, block_table, S), gather_pages(Vp, block_table, S), kv_len, L,
                       scale=scale, rows=rows, fill=fill)


def verify_attn(Q, Kc, Vc, kv_len, L, scale=None, rows=None, fill=np.nan):
    """Block-causal GQA attention in fp64.

    Q [B,K+1,Hq,d], Kc/Vc [B,Hkv,S_cap,d] as bf16 bit patterns (uint16) or
    torch bf16 tensors. Returns O [B,K+1,Hq,d] (fp64; rows not computed hold
    ``fill``) and lse [B,K+1,Hq].
    """
    Qb, Kb, Vb = (_as_bf16_bits(t) for t in (Q, Kc, Vc))
    B, K1, Hq, d = Qb.shape
    _, Hkv, S_cap, d2 = Kb.shape
    if d2 != d or Vb.shape != Kb.shape or Kb.shape[0] != B:
        raise OracleError("shape mismatch")
    if scale is None:
        scale = 1.0 / np.sqrt(d)
    kl = _c(kv_len, np.int32)
    LL = _c(L, np.int32)
    O = np.full((B, K1, Hq, d), fill, np.float64)
    lse = np.full((B, K1, Hq), fill, np.float64)
    rws = None if rows is None else _c(rows, np.int32).reshape(-1, 3)
    n_rows = 0 if rws is None else rws.shape[0]
    _check(_load().oracle_verify_attn(_ptr(Qb), _ptr(Kb), _ptr(Vb), _ptr(kl), _ptr(LL), B, K1 - 1, Hq,
                                      Hkv, d, S_cap, float(scale), _ptr(O), _ptr(lse), _ptr(rws), n_rows),
           "oracle_verify_attn")
    return O, lse


def verify_attn_tree(Q, Kc, Vc, kv_len, L, parent, scale=None, rows=None, fill=np.nan):
    """verify_attn of a draft tree: parent [B,K+1] (int32; parent[b,t] in [0,t) for 1 <= t <= L_b)."""
    Qb, Kb, Vb = (_as_bf16_bits(t) for t in (Q, Kc, Vc))
    B, K1, Hq, d = Qb.shape
    _, Hkv, S_cap, d2 = Kb.shape
    if d2 != d or Vb.shape != Kb.shape or Kb.shape[0] != B:
        raise OracleError("shape mismatch")
    par = _c(parent, np.int32)
    if par.shape != (B, K1):
        raise OracleError("parent must be [B,K+1]")
    if scale is None:
        scale = 1.0 / np.sqrt(d)
    kl = _c(kv_len, np.int32)
    LL = _c(L, np.int32)
    O = np.full((B, K1, Hq, d), fill, np.float64)
    lse = np.full((B, K1, Hq), fill, np.float64)
    rws = None if rows is None else _c(rows, np.int32).reshape(-1, 3)
    n_rows = 0 if rws is None else rws.shape[0]
    _check(_load().oracle_verify_attn_tree(_ptr(Qb), _ptr(Kb), _ptr(Vb), _ptr(kl), _ptr(LL), _ptr(par), B, K1 - 1,
                                           Hq, Hkv, d, S_cap, float(scale), _ptr(O), _ptr(lse), _ptr(rws), n_rows),
           "oracle_verify_attn_tree")
    return O, lse


def accept_tree_greedy(target_logits, draft_tokens, parent, L):
    """Greedy walk of a draft tree: n_accepted[B], last_node[B], bonus_token[B] (int32)."""
    t = _c(target_logits, np.float32)
    B, K1, V = t.shape
    tok = _c(draft_tokens, np.int32)
    if tok.shape != (B, K1 - 1):
        raise OracleError("draft_tokens must be [B,K]")
    par = _c(parent, np.int32)
    if par.shape != (B, K1):
        raise OracleError("parent must be [B,K+1]")
    LL = _c(L, np.int32)
    n = np.zeros(B, np.int32)
    last = np.zeros(B, np.int32)
    bonus = np.zeros(B, np.int32)
    _check(_load().oracle_accept_tree_greedy(_ptr(t), _ptr(tok), _ptr(par), _ptr(LL), B, K1 - 1, V,
                                             _ptr(n), _ptr(last), _ptr(bonus)), "oracle_accept_tree_greedy")
    return n, last, bonus


def accept_tree(target_logits, draft_tokens, parent, L, temperature, seed, round_offset=0, seq_offset=0):
    """Walk of a draft tree drawing the target's token at each node (greedy where temperature is 0):
    n_accepted[B], last_node[B], bonus_token[B], flag[B] (int32)."""
    t = _c(target_logits, np.float32)
    B, K1, V = t.shape
    tok = _c(draft_tokens, np.int32)
    if tok.shape != (B, K1 - 1):
        raise OracleError("draft_tokens must be [B,K]")
    par = _c(parent, np.int32)
    if par.shape != (B, K1):
        raise OracleError("parent must be [B,K+1]")
    LL = _c(L, np.int32)
    T = _c(temperature, np.float32)
    n = np.zeros(B, np.int32)
    last = np.zeros(B, np.int32)
    bonus = np.zeros(B, np.int32)
    flag = np.zeros(B, np.int32)
    _check(_load().oracle_accept_tree(_ptr(t), _ptr(tok), _ptr(par), _ptr(LL), _ptr(T), B, K1 - 1, V,
                                      int(seed) & (2**64 - 1), int(round_offset), int(seq_offset), _ptr(n),
                                      _ptr(last), _ptr(bonus), _ptr(flag)), "oracle_accept_tree")
    return n, last, bonus, flag


def lm_head_stats(H, W, temperature=None, rows_per_seq=1, tokens=None):
    """Row statistics of logits H @ W^T (bf16 inputs, binary64 sums): row_max, row_Z (at the row's
    temperature, 1 where 0), row_argmax, token_prob (0 where token < 0 or tokens is None), flag."""
    Hb, Wb = _as_bf16_bits(H), _as_bf16_bits(W)
    M, Dm = Hb.shape
    V, Dm2 = Wb.shape
    if Dm2 != Dm:
        raise OracleError("H and W disagree on the model dimension")
    T = None if temperature is None else _c(temperature, np.float32)
    tok = None if tokens is None else _c(tokens, np.int32)
    mx, Z, tp = (np.zeros(M, np.float64) for _ in range(3))
    arg, flag = np.zeros(M, np.int32), np.zeros(M, np.int32)
    _check(_load().oracle_lm_head_stats(_ptr(Hb), _ptr(Wb), _ptr(T), int(rows_per_seq), _ptr(tok), M, V, Dm,
                                        _ptr(mx), _ptr(Z), _ptr(arg), _ptr(tp), _ptr(flag)), "oracle_lm_head_stats")
    return mx, Z, arg, tp, flag


def accept(target_logits, draft_logits, draft_tokens, L, temperature, seed, round_offset=0,
           seq_offset=0):
    """n_accepted[B], bonus_token[B], flag[B]."""
    t = _c(target_logits, np.float32)
    B, K1, V = t.shape
    dr = _c(draft_logits, np.float32)
    if dr.shape != (B, K1 - 1, V):
        raise OracleError("draft_logits must be [B,K,V]")
    tok = _c(draft_tokens, np.int32)
    LL = _c(L, np.int32)
    T = _c(temperature, np.float32)
    n = np.zeros(B, np.int32)
    bonus = np.zeros(B, np.int32)
    flag = np.zeros(B, np.int32)
    _check(_load().oracle_accept(_ptr(t), _ptr(dr), _ptr(tok), _ptr(LL), _ptr(T), B, K1 - 1, V,
                                 int(seed) & (2**64 - 1), int(round_offset), int(seq_offset),
                                 _ptr(n), _ptr(bonus), _ptr(flag)), "oracle_accept")
    return n, bonus, flag


def _as_bf16_bits(t):
    """numpy uint16 view of a bf16 tensor (torch bf16 or uint16 array)."""
    if isinstance(t, np.ndarray):
        if t.dtype != np.uint16:
            raise OracleError("expected bf16 bit patterns as uint16")
        return np.ascontiguousarray(t)
    import torch  # only for converting caller tensors

    if t.dtype != torch.bfloat16:
        raise OracleError("expected a bf16 tensor")
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
