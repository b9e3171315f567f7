"""Thin ctypes binding of libraspec.so (include/libraspec.h).

Functions carry the C names and take torch tensors; they only check and
marshal arguments (dtype, device, contiguity, shapes) and pass the current
CUDA stream. Every step of the verify round runs in the library's kernels.
A missing or unloadable library raises; there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence, Tuple

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libraspec.so")

OK, EINVAL, EUNSUPPORTED, ECUDA, EDEVICE = 0, -1, -2, -3, -4
ST_BAD_LENGTH, ST_BAD_COST, ST_KV_OVERFLOW, ST_BAD_TOKEN, ST_TIMEOUT, ST_MISSING_INPUT = 1, 2, 4, 8, 16, 32
ST_BAD_PAGE, ST_BAD_TREE = 0x40, 0x80
MAX_K = 64
MAX_TREE_NODES = 512

# Every entry point declared in include/libraspec.h, with its ctypes signature.
_P, _I, _U32, _U64, _F, _SZ = (ctypes.c_void_p, ctypes.c_int, ctypes.c_uint32, ctypes.c_uint64, ctypes.c_float,
                               ctypes.c_size_t)
SIGNATURES = {
    "libraspec_version": (ctypes.c_char_p, []),
    "libraspec_status_string": (ctypes.c_char_p, [_I]),
    "libraspec_workspace_size": (_SZ, [_I, _I, _I, _I, _I, _I, _I]),
    "libraspec_workspace_init": (_I, [_P, _SZ, _P]),
    "libraspec_get_status": (_I, [_P, _P, _P]),
    "libraspec_selftest_wait": (_I, [_P, _U64, _P, _P, _SZ, _P]),
    "libraspec_confidence": (_I, [_P, _P, _P, _I, _I, _I, _P, _P, _P, _SZ, _P]),
    "libraspec_confidence_bf16": (_I, [_P, _P, _P, _I, _I, _I, _P, _P, _P, _SZ, _P]),
    "libraspec_confidence_noalloc": (_I, [_P, _P, _P, _I, _I, _I, _P, _P, _P, _P]),
    "libraspec_confidence_select": (_I, [_P, _P, _P, _P, _I, _I, _I, _P, _P, _P, _P, _SZ, _P]),
    "libraspec_confidence_select_bf16": (_I, [_P, _P, _P, _P, _I, _I, _I, _P, _P, _P, _P, _SZ, _P]),
    "libraspec_select_lengths": (_I, [_P, _P, _I, _I, _P, _P, _SZ, _P]),
    "libraspec_select_alpha": (_I, [_P, _I, _I, _I, _F, _P, _P, _P]),
    "libraspec_verify_attn": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _F, _P, _P, _P, _SZ, _P]),
    "libraspec_verify_attn_layers": (_I, [_P, _P, _P, _I, _P, _P, _I, _I, _I, _I, _I, _I, _F, _P, _P, _P, _SZ, _P]),
    "libraspec_verify_attn_paged_layers": (_I, [_P, _P, _P, _I, _P, _I, _I, _I, _P, _P, _I, _I, _I, _I, _I, _F, _P, _P,
                                                _P, _SZ, _P]),
    "libraspec_verify_attn_tree_layers": (_I, [_P, _P, _P, _I, _P, _P, _P, _I, _I, _I, _I, _I, _I, _F, _P, _P, _P,
                                               _SZ, _P]),
    "libraspec_verify_attn_tree_paged_layers": (_I, [_P, _P, _P, _I, _P, _P, _I, _I, _I, _P, _P, _I, _I, _I, _I, _I,
                                                     _F, _P, _P, _P, _SZ, _P]),
    "libraspec_accept_tree_greedy": (_I, [_P, _P, _P, _P, _I, _I, _I, _P, _P, _P, _P, _SZ, _P]),
    "libraspec_accept_tree_greedy_bf16": (_I, [_P, _P, _P, _P, _I, _I, _I, _P, _P, _P, _P, _SZ, _P]),
    "libraspec_accept_tree": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _U64, _U64, _U32, _P, _P, _P, _P, _SZ, _P]),
    "libraspec_accept_tree_bf16": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _U64, _U64, _U32, _P, _P, _P, _P, _SZ,
                                        _P]),
    "libraspec_verify_round_staged": (_I, [_P] * 18 + [_I, _P] + [_I] * 7 + [_F, _U64, _U64, _U32] + [_P] * 6 +
                                      [_SZ, _P]),
    "libraspec_verify_round_staged_bf16": (_I, [_P] * 18 + [_I, _P] + [_I] * 7 + [_F, _U64, _U64, _U32] + [_P] * 6 +
                                           [_SZ, _P]),
    "libraspec_lm_head_workspace_size": (_SZ, [_I, _I]),
    "libraspec_lm_head_stats": (_I, [_P, _P, _P, _I, _P, _I, _I, _I, _P, _P, _P, _P, _SZ, _P]),
    "libraspec_kv_append": (_I, [_P, _P, _P, _I, _P, _I, _I, _I, _I, _I, _P, _SZ, _P]),
    "libraspec_kv_append_paged": (_I, [_P, _P, _P, _I, _P, _I, _I, _I, _P, _I, _I, _I, _I, _P, _SZ, _P]),
    "libraspec_accept": (_I, [_P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _U64, _U64, _U32, _P, _P, _P, _SZ, _P]),
    "libraspec_accept_bf16": (_I, [_P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _U64, _U64, _U32, _P, _P, _P, _SZ, _P]),
    "libraspec_verify_round": (_I, [_P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _I, _P, _I, _I, _I, _I, _I, _I, _I,
                                    _F, _U64, _U64, _U32, _P, _P, _P, _P, _P, _P, _SZ, _P]),
    "libraspec_verify_round_bf16": (_I, [_P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _I, _P, _I, _I, _I, _I, _I, _I,
                                         _I, _F, _U64, _U64, _U32, _P, _P, _P, _P, _P, _P, _SZ, _P]),
}

_lib = None


class LibraspecError(RuntimeError):
    def __init__(self, what: str, status: int):
        super().__init__("%s failed: %s (%d)" % (what, _status_name(status), status))
        self.status = status


def _status_name(status: int) -> str:
    return {OK: "ok", EINVAL: "invalid argument", EUNSUPPORTED: "unsupported shape", ECUDA: "CUDA error",
            EDEVICE: "device-reported violation"}.get(status, "unknown")


def load() -> ctypes.CDLL:
    """Load libraspec.so (built by build.py); raises if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError("libraspec.so is not built (%s); run `python -m paper_2608_08721_gb300.build` or "
                           "__graft_entry__.build()" % LIB_PATH)
    lib = ctypes.CDLL(LIB_PATH)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _check(rc: int, what: str) -> None:
    if rc != OK:
        raise LibraspecError(what, rc)


def _stream(stream: Optional[torch.cuda.Stream]) -> ctypes.c_void_p:
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _req_dev_or_pinned(t: torch.Tensor, dtype, name: str, shape=None) -> torch.Tensor:
    """_req, or the same checks on a pinned host tensor (read in place by the kernels)."""
    if isinstance(t, torch.Tensor) and not t.is_cuda:
        if not t.is_pinned():
            raise ValueError("%s must be on a CUDA device or in pinned host memory" % name)
        if t.dtype != dtype or not t.is_contiguous() or (shape is not None and tuple(t.shape) != tuple(shape)):
            raise ValueError("%s: dtype %s, contiguous, shape %s required" % (name, dtype, shape))
        return t
    return _req(t, dtype, name, shape)


def _req(t: torch.Tensor, dtype, name: str, shape=None) -> torch.Tensor:
    if not isinstance(t, torch.Tensor):
        raise TypeError("%s must be a torch tensor" % name)
    if t.dtype != dtype:
        raise TypeError("%s must be %s, got %s" % (name, dtype, t.dtype))
    if not t.is_cuda:
        raise ValueError("%s must be on a CUDA device" % name)
    if not t.is_contiguous():
        raise ValueError("%s must be contiguous" % name)
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError("%s must have shape %s, got %s" % (name, tuple(shape), tuple(t.shape)))
    return t


class Workspace:
    """Device scratch for one round's shapes (a zero-filled torch buffer)."""

    def __init__(self, B, K, V, Hq=1, Hkv=1, head_dim=64, S_cap=1, device=None):
        lib = load()
        self.nbytes = int(lib.libraspec_workspace_size(B, K, V, Hq, Hkv, head_dim, S_cap))
        if self.nbytes == 0:
            raise ValueError("invalid workspace shapes")
        dev = torch.device("cuda") if device is None else torch.device(device)
        self.buf = torch.zeros(self.nbytes, dtype=torch.uint8, device=dev)
        if self.buf.data_ptr() % 256:
            raise RuntimeError("workspace allocation is not 256-byte aligned")
        self.shapes = (B, K, V, Hq, Hkv, head_dim, S_cap)

    @property
    def ptr(self) -> int:
        return self.buf.data_ptr()


def libraspec_version() -> str:
    return load().libraspec_version().decode()


def libraspec_workspace_size(B, K, V, Hq, Hkv, head_dim, S_cap) -> int:
    return int(load().libraspec_workspace_size(B, K, V, Hq, Hkv, head_dim, S_cap))


def libraspec_get_status(ws: Workspace, stream=None) -> int:
    out = ctypes.c_int32(0)
    rc = load().libraspec_get_status(ctypes.c_void_p(ws.ptr), _stream(stream), ctypes.byref(out))
    if rc not in (OK, EDEVICE):
        _check(rc, "libraspec_get_status")
    return int(out.value)


def libraspec_selftest_wait(flag, limit_ns: int, ws: Workspace, observed=None, stream=None) -> torch.Tensor:
    """The library's bounded wait on the device word ``flag`` (uint32 stored as int32 [1]) with a limit of
    limit_ns; returns ``observed`` (int32 [1] on the device): 1 if the flag was seen, 0 if the wait gave up
    (LIBRASPEC_ST_TIMEOUT is then set in the workspace's status)."""
    _req(flag, torch.int32, "flag", (1,))
    observed = torch.empty((1,), dtype=torch.int32, device=flag.device) if observed is None else _req(
        observed, torch.int32, "observed", (1,))
    rc = load().libraspec_selftest_wait(_ptr(flag), int(limit_ns), _ptr(observed), ws.ptr, ws.nbytes,
                                        _stream(stream))
    _check(rc, "libraspec_selftest_wait")
    return observed


def libraspec_confidence(draft_logits, draft_tokens, temperature, ws: Workspace, conf=None, dstat=None,
                         stream=None) -> Tuple[torch.Tensor, torch.Tensor]:
    B, K, V = draft_logits.shape
    bf16 = draft_logits.dtype == torch.bfloat16  # libraspec_confidence_bf16
    _req(draft_logits, torch.bfloat16 if bf16 else torch.float32, "draft_logits")
    _req(draft_tokens, torch.int32, "draft_tokens", (B, K))
    _req(temperature, torch.float32, "temperature", (B,))
    dev = draft_logits.device
    conf = torch.empty((B, K), dtype=torch.float32, device=dev) if conf is None else _req(conf, torch.float32,
                                                                                          "conf", (B, K))
    dstat = torch.empty((B, K, 2), dtype=torch.float32, device=dev) if dstat is None else _req(
        dstat, torch.float32, "dstat", (B, K, 2))
    name = "libraspec_confidence_bf16" if bf16 else "libraspec_confidence"
    rc = getattr(load(), name)(_ptr(draft_logits), _ptr(draft_tokens), _ptr(temperature), B, K, V, _ptr(conf),
                               _ptr(dstat), ws.ptr, ws.nbytes, _stream(stream))
    _check(rc, name)
    return conf, dstat


NOALLOC_MAX_ROWS = 4096


def libraspec_confidence_noalloc(draft_logits, draft_tokens, temperature, conf, dstat=None, status=None,
                                 stream=None) -> None:
    """libraspec_confidence with the library's static scratch instead of a
    workspace. Allocates nothing: the outputs (conf [B,K], optional dstat
    [B,K,2], optional status [1] int32) are caller tensors."""
    B, K, V = draft_logits.shape
    _req(draft_logits, torch.float32, "draft_logits")
    _req(draft_tokens, torch.int32, "draft_tokens", (B, K))
    _req(temperature, torch.float32, "temperature", (B,))
    _req(conf, torch.float32, "conf", (B, K))
    if dstat is not None:
        _req(dstat, torch.float32, "dstat", (B, K, 2))
    if status is not None:
        _req(status, torch.int32, "status", (1,))
    if B * K > NOALLOC_MAX_ROWS:
        raise ValueError("libraspec_confidence_noalloc: B*K = %d drafter rows exceeds the static scratch limit "
                         "of %d rows; use libraspec_confidence with a workspace" % (B * K, NOALLOC_MAX_ROWS))
    rc = load().libraspec_confidence_noalloc(_ptr(draft_logits), _ptr(draft_tokens), _ptr(temperature), B, K, V,
                                             _ptr(conf), _ptr(dstat), _ptr(status), _stream(stream))
    _check(rc, "libraspec_confidence_noalloc")


def libraspec_confidence_select(draft_logits, draft_tokens, temperature, cost_table, ws: Workspace, conf=None,
                                dstat=None, L=None, stream=None):
    """Confidence and the Thm. 4 selection in one launch: (conf [B,K], dstat [B,K,2], L [B])."""
    B, K, V = draft_logits.shape
    bf16 = draft_logits.dtype == torch.bfloat16
    _req(draft_logits, torch.bfloat16 if bf16 else torch.float32, "draft_logits")
    _req(draft_tokens, torch.int32, "draft_tokens", (B, K))
    _req(temperature, torch.float32, "temperature", (B,))
    _req(cost_table, torch.float32, "cost_table", (K + 1,))
    dev = draft_logits.device
    conf = torch.empty((B, K), dtype=torch.float32, device=dev) if conf is None else conf
    dstat = torch.empty((B, K, 2), dtype=torch.float32, device=dev) if dstat is None else dstat
    L = torch.empty((B,), dtype=torch.int32, device=dev) if L is None else L
    name = "libraspec_confidence_select_bf16" if bf16 else "libraspec_confidence_select"
    rc = getattr(load(), name)(_ptr(draft_logits), _ptr(draft_tokens), _ptr(temperature), _ptr(cost_table), B, K, V,
                               _ptr(conf), _ptr(dstat), _ptr(L), ws.ptr, ws.nbytes, _stream(stream))
    _check(rc, name)
    return conf, dstat, L


def libraspec_select_lengths(conf, cost_table, ws: Workspace, L=None, stream=None) -> torch.Tensor:
    B, K = conf.shape
    _req(conf, torch.float32, "conf")
    _req(cost_table, torch.float32, "cost_table", (K + 1,))
    L = torch.empty((B,), dtype=torch.int32, device=conf.device) if L is None else _req(L, torch.int32, "L", (B,))
    rc = load().libraspec_select_lengths(_ptr(conf), _ptr(cost_table), B, K, _ptr(L), ws.ptr, ws.nbytes,
                                         _stream(stream))
    _check(rc, "libraspec_select_lengths")
    return L


def libraspec_select_alpha(conf, block_size: int, alpha: float, L=None, n_blocks=None, stream=None):
    """Algorithm 1's alpha-mode search: L[B] and blocks drafted[B] (int32, device)."""
    B, K = conf.shape
    _req(conf, torch.float32, "conf")
    L = torch.empty((B,), dtype=torch.int32, device=conf.device) if L is None else _req(L, torch.int32, "L", (B,))
    if n_blocks is None:
        n_blocks = torch.empty((B,), dtype=torch.int32, device=conf.device)
    else:
        _req(n_blocks, torch.int32, "n_blocks", (B,))
    rc = load().libraspec_select_alpha(_ptr(conf), B, K, int(block_size), float(alpha), _ptr(L), _ptr(n_blocks),
                                       _stream(stream))
    _check(rc, "libraspec_select_alpha")
    return L, n_blocks


def libraspec_verify_attn(Q, Kc, Vc, kv_len, L, ws: Workspace, softmax_scale=None, O=None, lse=None,
                          want_lse=False, stream=None):
    B, K1, Hq, D = Q.shape
    _, Hkv, S_cap, D2 = Kc.shape
    _req(Q, torch.bfloat16, "Q")
    _req(Kc, torch.bfloat16, "Kc", (B, Hkv, S_cap, D))
    _req(Vc, torch.bfloat16, "Vc", (B, Hkv, S_cap, D))
    _req(kv_len, torch.int32, "kv_len", (B,))
    _req(L, torch.int32, "L", (B,))
    if softmax_scale is None:
        softmax_scale = D ** -0.5
    O = torch.empty_like(Q) if O is None else _req(O, torch.bfloat16, "O", Q.shape)
    if want_lse and lse is None:
        lse = torch.empty((B, K1, Hq), dtype=torch.float32, device=Q.device)
    rc = load().libraspec_verify_attn(_ptr(Q), _ptr(Kc), _ptr(Vc), _ptr(kv_len), _ptr(L), B, K1 - 1, Hq, Hkv, D,
                                      S_cap, float(softmax_scale), _ptr(O), _ptr(lse), ws.ptr, ws.nbytes,
                                      _stream(stream))
    _check(rc, "libraspec_verify_attn")
    return O, lse


def libraspec_verify_attn_layers(layers, kv_len, L, ws: Workspace, softmax_scale=None, want_lse=False,
                                 stream=None):
    """layers: sequence of dicts with Q, Kc, Vc (and optionally O, lse). Returns (O list, lse list or None)."""
    return _attn_layers(layers, None, kv_len, L, ws, softmax_scale, want_lse, stream)


def libraspec_verify_attn_tree_layers(layers, parent, kv_len, L, ws: Workspace, softmax_scale=None, want_lse=False,
                                      stream=None):
    """Draft-tree verify attention; parent [B, K+1] int32 (parent[b, t] < t). As libraspec_verify_attn_layers."""
    return _attn_layers(layers, parent, kv_len, L, ws, softmax_scale, want_lse, stream)


def _check_parent(parent, B, K1):
    _req(parent, torch.int32, "parent", (B, K1))


def _attn_layers(layers, parent, kv_len, L, ws, softmax_scale, want_lse, stream):
    n = len(layers)
    if n == 0:
        return [], None
    B, K1, Hq, D = layers[0]["Q"].shape
    _, Hkv, S_cap, _ = layers[0]["Kc"].shape
    for i, lay in enumerate(layers):
        _req(lay["Q"], torch.bfloat16, "Q[%d]" % i, (B, K1, Hq, D))
        _req(lay["Kc"], torch.bfloat16, "Kc[%d]" % i, (B, Hkv, S_cap, D))
        _req(lay["Vc"], torch.bfloat16, "Vc[%d]" % i, (B, Hkv, S_cap, D))
    _req(kv_len, torch.int32, "kv_len", (B,))
    _req(L, torch.int32, "L", (B,))
    if parent is not None:
        _check_parent(parent, B, K1)
    if softmax_scale is None:
        softmax_scale = D ** -0.5
    outs = [lay.get("O") if lay.get("O") is not None else torch.empty_like(lay["Q"]) for lay in layers]
    lses = None
    if want_lse:
        lses = [lay.get("lse") if lay.get("lse") is not None else
                torch.empty((B, K1, Hq), dtype=torch.float32, device=layers[0]["Q"].device) for lay in layers]
    args = [_ptr_array([l["Q"] for l in layers]), _ptr_array([l["Kc"] for l in layers]),
            _ptr_array([l["Vc"] for l in layers]), n]
    name = "libraspec_verify_attn_layers"
    if parent is not None:
        args.append(_ptr(parent))
        name = "libraspec_verify_attn_tree_layers"
    rc = getattr(load(), name)(
        *args, _ptr(kv_len), _ptr(L), B, K1 - 1, Hq, Hkv, D, S_cap, float(softmax_scale), _ptr_array(outs),
        _ptr_array(lses) if lses is not None else None, ws.ptr, ws.nbytes, _stream(stream))
    _check(rc, name)
    return outs, lses


def libraspec_verify_attn_paged_layers(layers, block_table, kv_len, L, ws: Workspace, softmax_scale=None,
                                       want_lse=False, stream=None):
    """layers: dicts with Q [B,K+1,Hq,d] and page pools Kp, Vp [n_pages,Hkv,page_size,d] (optionally O,
    lse); block_table [B, max_pages] int32. Returns (O list, lse list or None)."""
    return _attn_paged_layers(layers, None, block_table, kv_len, L, ws, softmax_scale, want_lse, stream)


def libraspec_verify_attn_tree_paged_layers(layers, parent, block_table, kv_len, L, ws: Workspace,
                                            softmax_scale=None, want_lse=False, stream=None):
    """Draft-tree verify attention over a paged cache; parent [B, K+1] int32."""
    return _attn_paged_layers(layers, parent, block_table, kv_len, L, ws, softmax_scale, want_lse, stream)


def _attn_paged_layers(layers, parent, block_table, kv_len, L, ws, softmax_scale, want_lse, stream):
    n = len(layers)
    if n == 0:
        return [], None
    B, K1, Hq, D = layers[0]["Q"].shape
    n_pages, Hkv, page_size, _ = layers[0]["Kp"].shape
    for i, lay in enumerate(layers):
        _req(lay["Q"], torch.bfloat16, "Q[%d]" % i, (B, K1, Hq, D))
        _req(lay["Kp"], torch.bfloat16, "Kp[%d]" % i, (n_pages, Hkv, page_size, D))
        _req(lay["Vp"], torch.bfloat16, "Vp[%d]" % i, (n_pages, Hkv, page_size, D))
    _req(block_table, torch.int32, "block_table")
    if block_table.dim() != 2 or block_table.shape[0] != B:
        raise ValueError("block_table must be [B, max_pages]")
    max_pages = block_table.shape[1]
    _req(kv_len, torch.int32, "kv_len", (B,))
    _req(L, torch.int32, "L", (B,))
    if parent is not None:
        _check_parent(parent, B, K1)
    if softmax_scale is None:
        softmax_scale = D ** -0.5
    outs = [lay.get("O") if lay.get("O") is not None else torch.empty_like(lay["Q"]) for lay in layers]
    lses = None
    if want_lse:
        lses = [lay.get("lse") if lay.get("lse") is not None else
                torch.empty((B, K1, Hq), dtype=torch.float32, device=layers[0]["Q"].device) for lay in layers]
    args = [_ptr_array([l["Q"] for l in layers]), _ptr_array([l["Kp"] for l in layers]),
            _ptr_array([l["Vp"] for l in layers]), n]
    name = "libraspec_verify_attn_paged_layers"
    if parent is not None:
        args.append(_ptr(parent))
        name = "libraspec_verify_attn_tree_paged_layers"
    rc = getattr(load(), name)(
        *args, _ptr(block_table), max_pages, page_size, n_pages, _ptr(kv_len), _ptr(L), B, K1 - 1, Hq, Hkv, D,
        float(softmax_scale), _ptr_array(outs), _ptr_array(lses) if lses is not None else None, ws.ptr, ws.nbytes,
        _stream(stream))
    _check(rc, name)
    return outs, lses


def libraspec_accept(target_logits, draft_logits, draft_tokens, conf, dstat, L, temperature, seed: int,
                     ws: Workspace, round_offset: int = 0, seq_offset: int = 0, n_accepted=None, bonus_token=None,
                     stream=None):
    B, K1, V = target_logits.shape
    K = K1 - 1
    bf16 = target_logits.dtype == torch.bfloat16  # libraspec_accept_bf16: both logit tensors bf16
    ldt = torch.bfloat16 if bf16 else torch.float32
    _req(target_logits, ldt, "target_logits")
    _req(draft_logits, ldt, "draft_logits", (B, K, V))
    _req(draft_tokens, torch.int32, "draft_tokens", (B, K))
    if conf is not None:
        _req(conf, torch.float32, "conf", (B, K))
    if dstat is not None:
        _req(dstat, torch.float32, "dstat", (B, K, 2))
    _req(L, torch.int32, "L", (B,))
    _req(temperature, torch.float32, "temperature", (B,))
    dev = target_logits.device
    n_accepted = torch.empty((B,), dtype=torch.int32, device=dev) if n_accepted is None else n_accepted
    bonus_token = torch.empty((B,), dtype=torch.int32, device=dev) if bonus_token is None else bonus_token
    name = "libraspec_accept_bf16" if bf16 else "libraspec_accept"
    rc = getattr(load(), name)(_ptr(target_logits), _ptr(draft_logits), _ptr(draft_tokens), _ptr(conf), _ptr(dstat),
                               _ptr(L), _ptr(temperature), B, K, V, int(seed) & (2**64 - 1), int(round_offset),
                               int(seq_offset), _ptr(n_accepted), _ptr(bonus_token), ws.ptr, ws.nbytes,
                               _stream(stream))
    _check(rc, name)
    return n_accepted, bonus_token


def libraspec_accept_tree_greedy(target_logits, draft_tokens, parent, L, ws: Workspace, n_accepted=None,
                                 last_node=None, bonus_token=None, stream=None):
    """Greedy walk of a draft tree. Returns (n_accepted, last_node, bonus_token), int32 [B] each."""
    B, K1, V = target_logits.shape
    K = K1 - 1
    bf16 = target_logits.dtype == torch.bfloat16
    _req(target_logits, torch.bfloat16 if bf16 else torch.float32, "target_logits")
    _req(draft_tokens, torch.int32, "draft_tokens", (B, K))
    _check_parent(parent, B, K1)
    _req(L, torch.int32, "L", (B,))
    dev = target_logits.device
    n_accepted = torch.empty((B,), dtype=torch.int32, device=dev) if n_accepted is None else n_accepted
    last_node = torch.empty((B,), dtype=torch.int32, device=dev) if last_node is None else last_node
    bonus_token = torch.empty((B,), dtype=torch.int32, device=dev) if bonus_token is None else bonus_token
    name = "libraspec_accept_tree_greedy_bf16" if bf16 else "libraspec_accept_tree_greedy"
    rc = getattr(load(), name)(_ptr(target_logits), _ptr(draft_tokens), _ptr(parent), _ptr(L), B, K, V,
                               _ptr(n_accepted), _ptr(last_node), _ptr(bonus_token), ws.ptr, ws.nbytes,
                               _stream(stream))
    _check(rc, name)
    return n_accepted, last_node, bonus_token


def libraspec_accept_tree(target_logits, draft_tokens, parent, L, temperature, seed: int, ws: Workspace,
                          round_offset: int = 0, seq_offset: int = 0, n_accepted=None, last_node=None,
                          bonus_token=None, stream=None):
    """Walk of a draft tree drawing the target's token at each node (greedy where temperature is 0).
    Returns (n_accepted, last_node, bonus_token), int32 [B] each."""
    B, K1, V = target_logits.shape
    K = K1 - 1
    bf16 = target_logits.dtype == torch.bfloat16
    _req(target_logits, torch.bfloat16 if bf16 else torch.float32, "target_logits")
    _req(draft_tokens, torch.int32, "draft_tokens", (B, K))
    _check_parent(parent, B, K1)
    _req(L, torch.int32, "L", (B,))
    _req(temperature, torch.float32, "temperature", (B,))
    dev = target_logits.device
    n_accepted = torch.empty((B,), dtype=torch.int32, device=dev) if n_accepted is None else n_accepted
    last_node = torch.empty((B,), dtype=torch.int32, device=dev) if last_node is None else last_node
    bonus_token = torch.empty((B,), dtype=torch.int32, device=dev) if bonus_token is None else bonus_token
    name = "libraspec_accept_tree_bf16" if bf16 else "libraspec_accept_tree"
    rc = getattr(load(), name)(_ptr(target_logits), _ptr(draft_tokens), _ptr(parent), _ptr(L), _ptr(temperature), B,
                               K, V, int(seed) & (2**64 - 1), int(round_offset), int(seq_offset), _ptr(n_accepted),
                               _ptr(last_node), _ptr(bonus_token), ws.ptr, ws.nbytes, _stream(stream))
    _check(rc, name)
    return n_accepted, last_node, bonus_token


def libraspec_kv_append(kv_new, caches, kv_len, ws: Workspace, block_table=None, stream=None) -> None:
    """kv_new [n_layers, 2, B, Hkv, T, d] bf16; caches: per layer {"Kc", "Vc"} (dense [B,Hkv,S_cap,d]) or
    {"Kp", "Vp"} (page pools [n_pages,Hkv,page_size,d], with block_table [B, max_pages])."""
    n_layers, two, B, Hkv, T, d = kv_new.shape
    if two != 2 or len(caches) != n_layers:
        raise ValueError("kv_new must be [n_layers, 2, B, Hkv, T, d] with one cache per layer")
    _req(kv_new, torch.bfloat16, "kv_new")
    _req(kv_len, torch.int32, "kv_len", (B,))
    if block_table is None:
        S_cap = caches[0]["Kc"].shape[2] if n_layers else 1
        for i, c in enumerate(caches):
            _req(c["Kc"], torch.bfloat16, "Kc[%d]" % i, (B, Hkv, S_cap, d))
            _req(c["Vc"], torch.bfloat16, "Vc[%d]" % i, (B, Hkv, S_cap, d))
        rc = load().libraspec_kv_append(_ptr(kv_new), _ptr_array([c["Kc"] for c in caches]),
                                        _ptr_array([c["Vc"] for c in caches]), n_layers, _ptr(kv_len), B, T, Hkv,
                                        d, S_cap, ws.ptr, ws.nbytes, _stream(stream))
        _check(rc, "libraspec_kv_append")
        return
    _req(block_table, torch.int32, "block_table")
    n_pages, _, page_size, _ = caches[0]["Kp"].shape
    for i, c in enumerate(caches):
        _req(c["Kp"], torch.bfloat16, "Kp[%d]" % i, (n_pages, Hkv, page_size, d))
        _req(c["Vp"], torch.bfloat16, "Vp[%d]" % i, (n_pages, Hkv, page_size, d))
    rc = load().libraspec_kv_append_paged(_ptr(kv_new), _ptr_array([c["Kp"] for c in caches]),
                                          _ptr_array([c["Vp"] for c in caches]), n_layers, _ptr(block_table),
                                          block_table.shape[1], page_size, n_pages, _ptr(kv_len), B, T, Hkv, d,
                                          ws.ptr, ws.nbytes, _stream(stream))
    _check(rc, "libraspec_kv_append_paged")


class LmHeadWorkspace:
    """Device scratch of libraspec_lm_head_stats for M rows and a vocabulary of V."""

    def __init__(self, M, V, device=None):
        self.nbytes = int(load().libraspec_lm_head_workspace_size(M, V))
        if self.nbytes == 0:
            raise ValueError("invalid LM-head workspace shapes")
        dev = torch.device("cuda") if device is None else torch.device(device)
        self.buf = torch.zeros(self.nbytes, dtype=torch.uint8, device=dev)

    @property
    def ptr(self) -> int:
        return self.buf.data_ptr()


def libraspec_lm_head_stats(H, W, ws: "LmHeadWorkspace", temperature=None, rows_per_seq: int = 1, tokens=None,
                            row_stat=None, row_argmax=None, token_prob=None, stream=None):
    """Row statistics of H @ W^T without storing it: (row_stat [M,2], row_argmax [M], token_prob [M] or None)."""
    M, Dm = H.shape
    V = W.shape[0]
    _req(H, torch.bfloat16, "H")
    _req(W, torch.bfloat16, "W", (V, Dm))
    if temperature is not None:
        _req(temperature, torch.float32, "temperature")
        if temperature.numel() * rows_per_seq < M:
            raise ValueError("temperature needs one entry per sequence of rows_per_seq rows")
    if tokens is not None:
        _req(tokens, torch.int32, "tokens", (M,))
    dev = H.device
    row_stat = torch.empty((M, 2), dtype=torch.float32, device=dev) if row_stat is None else row_stat
    row_argmax = torch.empty((M,), dtype=torch.int32, device=dev) if row_argmax is None else row_argmax
    if tokens is not None and token_prob is None:
        token_prob = torch.empty((M,), dtype=torch.float32, device=dev)
    rc = load().libraspec_lm_head_stats(_ptr(H), _ptr(W), _ptr(temperature), int(rows_per_seq), _ptr(tokens), M, V,
                                        Dm, _ptr(row_stat), _ptr(row_argmax), _ptr(token_prob), ws.ptr, ws.nbytes,
                                        _stream(stream))
    _check(rc, "libraspec_lm_head_stats")
    return row_stat, row_argmax, token_prob


def _ptr_array(tensors: Sequence[Optional[torch.Tensor]]):
    arr = (ctypes.c_void_p * max(1, len(tensors)))()
    for i, t in enumerate(tensors):
        arr[i] = None if t is None else t.data_ptr()
    return arr


class RoundOutputs:
    def __init__(self, conf, dstat, L, n_accepted, bonus_token, O, lse):
        self.conf, self.dstat, self.L = conf, dstat, L
        self.n_accepted, self.bonus_token = n_accepted, bonus_token
        self.O, self.lse = O, lse


def libraspec_verify_round(draft_logits, draft_tokens, temperature, cost_table, target_logits, layers, kv_len,
                           seed: int, ws: Workspace, round_offset: int = 0, seq_offset: int = 0,
                           softmax_scale=None, outputs: Optional[RoundOutputs] = None, want_lse=False,
                           stream=None) -> RoundOutputs:
    """layers: sequence of dicts with Q, Kc, Vc (and optionally O)."""
    B, K, V = draft_logits.shape
    bf16 = draft_logits.dtype == torch.bfloat16  # libraspec_verify_round_bf16: both logit tensors bf16
    ldt = torch.bfloat16 if bf16 else torch.float32
    _req(draft_logits, ldt, "draft_logits")
    _req(target_logits, ldt, "target_logits", (B, K + 1, V))
    _req(draft_tokens, torch.int32, "draft_tokens", (B, K))
    _req(temperature, torch.float32, "temperature", (B,))
    _req(cost_table, torch.float32, "cost_table", (K + 1,))
    _req(kv_len, torch.int32, "kv_len", (B,))
    n_layers = len(layers)
    Hq, D = (layers[0]["Q"].shape[2], layers[0]["Q"].shape[3]) if n_layers else (1, 64)
    Hkv, S_cap = (layers[0]["Kc"].shape[1], layers[0]["Kc"].shape[2]) if n_layers else (1, 1)
    for i, lay in enumerate(layers):
        _req(lay["Q"], torch.bfloat16, "Q[%d]" % i, (B, K + 1, Hq, D))
        _req(lay["Kc"], torch.bfloat16, "Kc[%d]" % i, (B, Hkv, S_cap, D))
        _req(lay["Vc"], torch.bfloat16, "Vc[%d]" % i, (B, Hkv, S_cap, D))
    dev = draft_logits.device
    if outputs is None:
        outputs = RoundOutputs(
            torch.empty((B, K), dtype=torch.float32, device=dev), torch.empty((B, K, 2), dtype=torch.float32, device=dev),
            torch.empty((B,), dtype=torch.int32, device=dev), torch.empty((B,), dtype=torch.int32, device=dev),
            torch.empty((B,), dtype=torch.int32, device=dev),
            [lay.get("O") if lay.get("O") is not None else torch.empty_like(lay["Q"]) for lay in layers],
            [torch.empty((B, K + 1, Hq), dtype=torch.float32, device=dev) for _ in layers] if want_lse else None)
    if softmax_scale is None:
        softmax_scale = D ** -0.5
    qa = _ptr_array([lay["Q"] for lay in layers])
    ka = _ptr_array([lay["Kc"] for lay in layers])
    va = _ptr_array([lay["Vc"] for lay in layers])
    oa = _ptr_array(outputs.O)
    la = _ptr_array(outputs.lse) if outputs.lse is not None else None
    name = "libraspec_verify_round_bf16" if bf16 else "libraspec_verify_round"
    rc = getattr(load(), name)(
        _ptr(draft_logits), _ptr(draft_tokens), _ptr(temperature), _ptr(cost_table), _ptr(target_logits), qa, ka, va,
        oa, la, n_layers, _ptr(kv_len), B, K, V, Hq, Hkv, D, S_cap, float(softmax_scale), int(seed) & (2**64 - 1),
        int(round_offset), int(seq_offset), _ptr(outputs.conf), _ptr(outputs.dstat), _ptr(outputs.L),
        _ptr(outputs.n_accepted), _ptr(outputs.bonus_token), ws.ptr, ws.nbytes, _stream(stream))
    _check(rc, name)
    return outputs


class StagedRound:
    """Marshalled arguments of libraspec_verify_round_staged for fixed buffers: built (and checked)
    once, then each call enqueues one round.

    host_parts / dev_parts: three (pinned host, device) uint8 tensors, the drafter part, the layers
    part and the target part; the typed inputs (draft_logits ... target_logits, each layer's Q,
    kv_new) are device tensors inside dev_parts; layers: per layer {"Q", "Kc", "Vc"};
    outputs: RoundOutputs; n_host / bonus_host: pinned int32 [B] tensors."""

    def __init__(self, host_parts, dev_parts, kv_new, n_host, bonus_host, draft_logits, draft_tokens, temperature,
                 cost_table, target_logits, layers, kv_len, outputs: "RoundOutputs", ws: Workspace,
                 rng_host, rng_dev, softmax_scale=None, copy_stream=None, copy_parts=(True, True, True)):
        """copy_parts[i] False: part i is not copied; its typed inputs (and kv_new / rng_dev when they
        lie in it) are then pinned host tensors that the kernels read in place (a pinned allocation's
        address is valid on the device under unified addressing)."""
        B, K, V = draft_logits.shape
        bf16 = draft_logits.dtype == torch.bfloat16
        ldt = torch.bfloat16 if bf16 else torch.float32
        req = _req_dev_or_pinned
        req(draft_logits, ldt, "draft_logits")
        req(target_logits, ldt, "target_logits", (B, K + 1, V))
        req(draft_tokens, torch.int32, "draft_tokens", (B, K))
        req(temperature, torch.float32, "temperature", (B,))
        req(cost_table, torch.float32, "cost_table", (K + 1,))
        _req(kv_len, torch.int32, "kv_len", (B,))
        n_layers = len(layers)
        Hq, D = layers[0]["Q"].shape[2], layers[0]["Q"].shape[3]
        Hkv, S_cap = layers[0]["Kc"].shape[1], layers[0]["Kc"].shape[2]
        for i, lay in enumerate(layers):
            _req(lay["Q"], torch.bfloat16, "Q[%d]" % i, (B, K + 1, Hq, D))
            _req(lay["Kc"], torch.bfloat16, "Kc[%d]" % i, (B, Hkv, S_cap, D))
            _req(lay["Vc"], torch.bfloat16, "Vc[%d]" % i, (B, Hkv, S_cap, D))
        req(kv_new, torch.bfloat16, "kv_new", (n_layers, 2, B, Hkv, K + 1, D))
        if len(host_parts) != 3 or len(dev_parts) != 3:
            raise ValueError("three host and three device parts")
        for h, d in zip(host_parts, dev_parts):
            if not h.is_pinned() or h.numel() != d.numel() or not d.is_cuda:
                raise ValueError("each part: a pinned host tensor and a device tensor of the same size")
        req(rng_dev, torch.int64, "rng_dev", (3,))
        if (not isinstance(rng_host, torch.Tensor) or rng_host.dtype != torch.int64 or rng_host.numel() != 3
                or not rng_host.is_pinned()):
            raise ValueError("rng_host must be 3 int64 of pinned host memory inside host part 2")
        if softmax_scale is None:
            softmax_scale = D ** -0.5
        self._keep = (host_parts, dev_parts, layers, outputs, n_host, bonus_host, rng_host, rng_dev)
        self._hp = (ctypes.c_void_p * 3)(*[h.data_ptr() for h in host_parts])
        self._dp = (ctypes.c_void_p * 3)(*[d.data_ptr() for d in dev_parts])
        self._nb = (ctypes.c_size_t * 3)(*[h.numel() * h.element_size() if c else 0
                                           for h, c in zip(host_parts, copy_parts)])
        self._copy = copy_stream if copy_stream is not None else torch.cuda.Stream(device=kv_len.device)
        self._qa = _ptr_array([l["Q"] for l in layers])
        self._ka = _ptr_array([l["Kc"] for l in layers])
        self._va = _ptr_array([l["Vc"] for l in layers])
        self._oa = _ptr_array(outputs.O)
        self._name = "libraspec_verify_round_staged_bf16" if bf16 else "libraspec_verify_round_staged"
        self._fn = getattr(load(), self._name)
        self._pre = (self._hp, self._dp, self._nb, ctypes.c_void_p(self._copy.cuda_stream), _ptr(kv_new),
                     _ptr(rng_host), _ptr(rng_dev), _ptr(n_host), _ptr(bonus_host), _ptr(draft_logits), _ptr(draft_tokens), _ptr(temperature),
                     _ptr(cost_table), _ptr(target_logits), self._qa, self._ka, self._va, self._oa, n_layers,
                     _ptr(kv_len), B, K, V, Hq, Hkv, D, S_cap, float(softmax_scale))
        self._post = (_ptr(outputs.conf), _ptr(outputs.dstat), _ptr(outputs.L), _ptr(outputs.n_accepted),
                      _ptr(outputs.bonus_token), ws.ptr, ws.nbytes)

    def __call__(self, seed: int, round_offset: int = 0, seq_offset: int = 0, stream=None) -> None:
        rc = self._fn(*self._pre, int(seed) & (2**64 - 1), int(round_offset), int(seq_offset), *self._post,
                      _stream(stream))
        _check(rc, self._name)


def libraspec_verify_round_staged(host_parts, dev_parts, kv_new, n_host, bonus_host, draft_logits, draft_tokens,
                                  temperature, cost_table, target_logits, layers, kv_len, outputs, ws, rng_host,
                                  rng_dev, seed: int, round_offset: int = 0, seq_offset: int = 0, softmax_scale=None,
                                  copy_stream=None, stream=None) -> None:
    """One staged round (see StagedRound); returns after enqueuing."""
    StagedRound(host_parts, dev_parts, kv_new, n_host, bonus_host, draft_logits, draft_tokens, temperature,
                cost_table, target_logits, layers, kv_len, outputs, ws, rng_host, rng_dev, softmax_scale,
                copy_stream)(
        seed, round_offset, seq_offset, stream)

