"""Public API: a verify round over device-resident state, fed from host buffers.

``VerifyRound`` owns the device buffers of one round's shapes (per-round
inputs, outputs, workspace) and runs the whole round through
``libraspec_verify_round``. The KV caches are model state and stay on the
device; the per-round inputs (logits, drafts, temperatures, cost table, the
verified block's queries and its new K/V rows) can be passed as pinned host
tensors, in which case they are copied in on the round's stream and the
accepted counts and bonus tokens are copied back.
"""
from __future__ import annotations

from typing import Dict, List, Optional

import numpy as np
import torch

from . import binding


class VerifyRound:
    def __init__(self, B: int, K: int, V: int, Hq: int, Hkv: int, head_dim: int, S_cap: int,
                 caches: List[Dict[str, torch.Tensor]], kv_len: torch.Tensor, device=None,
                 logits_dtype=torch.float32):
        """caches: per layer {"Kc", "Vc"} bf16 [B,Hkv,S_cap,d] on the device;
        logits_dtype: float32 or bfloat16 drafter and target logits."""
        if logits_dtype not in (torch.float32, torch.bfloat16):
            raise ValueError("logits_dtype must be torch.float32 or torch.bfloat16")
        self.B, self.K, self.V, self.Hq, self.Hkv, self.d, self.S_cap = B, K, V, Hq, Hkv, head_dim, S_cap
        self.device = torch.device("cuda") if device is None else torch.device(device)
        dev = self.device
        self.caches = caches
        self.n_layers = len(caches)
        self.ws = binding.Workspace(B, K, V, Hq, Hkv, head_dim, S_cap, device=dev)
        self.kv_len = kv_len.to(dev, torch.int32).contiguous()
        self.kv_len_host = [int(x) for x in kv_len.cpu()]
        f32, i32, bf = torch.float32, torch.int32, torch.bfloat16
        self.draft_logits = torch.empty((B, K, V), dtype=logits_dtype, device=dev)
        self.target_logits = torch.empty((B, K + 1, V), dtype=logits_dtype, device=dev)
        self.draft_tokens = torch.empty((B, K), dtype=i32, device=dev)
        self.temperature = torch.empty((B,), dtype=f32, device=dev)
        self.cost_table = torch.empty((K + 1,), dtype=f32, device=dev)
        self.layers = [{"Q": torch.empty((B, K + 1, Hq, head_dim), dtype=bf, device=dev),
                        "Kc": c["Kc"], "Vc": c["Vc"]} for c in caches]
        self.out = binding.RoundOutputs(
            torch.empty((B, K), dtype=f32, device=dev), torch.empty((B, K, 2), dtype=f32, device=dev),
            torch.empty((B,), dtype=i32, device=dev), torch.empty((B,), dtype=i32, device=dev),
            torch.empty((B,), dtype=i32, device=dev),
            [torch.empty((B, K + 1, Hq, head_dim), dtype=bf, device=dev) for _ in caches], None)
        self.result_host = torch.empty((2, B), dtype=i32, pin_memory=True)

    def run_device(self, seed: int, round_offset: int = 0, seq_offset: int = 0, stream=None):
        """The round on inputs already resident in this object's device buffers."""
        return binding.libraspec_verify_round(
            self.draft_logits, self.draft_tokens, self.temperature, self.cost_table, self.target_logits,
            self.layers, self.kv_len, seed, self.ws, round_offset=round_offset, seq_offset=seq_offset,
            outputs=self.out, stream=stream)

    def h2d_bytes(self) -> int:
        per_layer = self.B * (self.K + 1) * self.Hq * self.d * 2 + 2 * self.B * self.Hkv * (self.K + 1) * self.d * 2
        lb = self.draft_logits.element_size()
        return (self.draft_logits.numel() * lb + self.target_logits.numel() * lb + self.draft_tokens.numel() * 4 +
                self.temperature.numel() * 4 + self.cost_table.numel() * 4 + self.n_layers * per_layer)

    def d2h_bytes(self) -> int:
        return self.result_host.numel() * 4

    def run_host(self, host: Dict, seed: int, round_offset: int = 0, seq_offset: int = 0):
        """Copy one round's host inputs in, run the round, copy the results out.

        host: draft_logits, target_logits, draft_tokens, temperature, cost_table
        (pinned CPU tensors) and "layers": per layer {"Q", "K_new", "V_new"}
        with K_new / V_new [B,Hkv,K+1,d], the verified block's keys and values,
        written into the caches at kv_len_b .. kv_len_b + K.
        Returns (n_accepted, bonus_token) as numpy arrays."""
        nb = True
        self.draft_logits.copy_(host["draft_logits"], non_blocking=nb)
        self.target_logits.copy_(host["target_logits"], non_blocking=nb)
        self.draft_tokens.copy_(host["draft_tokens"], non_blocking=nb)
        self.temperature.copy_(host["temperature"], non_blocking=nb)
        self.cost_table.copy_(host["cost_table"], non_blocking=nb)
        K1 = self.K + 1
        for l, hl in enumerate(host["layers"]):
            self.layers[l]["Q"].copy_(hl["Q"], non_blocking=nb)
            for b in range(self.B):
                kv = self.kv_len_host[b]
                self.layers[l]["Kc"][b, :, kv:kv + K1].copy_(hl["K_new"][b], non_blocking=nb)
                self.layers[l]["Vc"][b, :, kv:kv + K1].copy_(hl["V_new"][b], non_blocking=nb)
        self.run_device(seed, round_offset, seq_offset)
        self.result_host[0].copy_(self.out.n_accepted, non_blocking=nb)
        self.result_host[1].copy_(self.out.bonus_token, non_blocking=nb)
        torch.cuda.current_stream().synchronize()
        return self.result_host[0].numpy().copy(), self.result_host[1].numpy().copy()
