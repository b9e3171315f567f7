"""Public API: a verify round over device-resident state, fed from host buffers.

``VerifyRound`` owns the device buffers of one round's shapes and runs the
whole round through ``libraspec_verify_round``. The KV caches are model state
and stay on the device. Every per-round input (drafter and target logits,
draft tokens, temperatures, the cost table, each layer's queries and the
verified block's new keys and values) lives in ONE pinned host buffer, laid
out in the order the round needs them: the drafter block (confidence and
selection), the layers' queries and new keys/values (``libraspec_kv_append``,
then attention), the target rows (acceptance).

By default the kernels read the inputs in place, over the host link: a
pinned allocation's address is valid on the device (unified addressing), and
a verify round reads most of its inputs once, or not at all (acceptance reads
only the verified target rows), so only the bytes the round uses cross the
link. The layers' queries, which the attention kernel's TMA loads, are copied
in on a side stream while the confidence streams the drafter block. With
``inputs_in_place=False`` the three parts are copied to a device mirror
instead, each step starting once its part has landed. Either way the accepted
counts and bonus tokens come back into pinned memory (8 bytes per sequence).
"""
from __future__ import annotations

from typing import Dict, List

import torch

from . import binding


def _layout(regions):
    """Byte offsets of the regions, each 256-byte aligned; returns (offsets, total)."""
    offs, off = {}, 0
    for name, shape, dtype in regions:
        offs[name] = off
        n = 1
        for s in shape:
            n *= s
        off += (n * torch.empty((), dtype=dtype).element_size() + 255) // 256 * 256
    return offs, off


class VerifyRound:
    def __init__(self, B: int, K: int, V: int, Hq: int, Hkv: int, head_dim: int, S_cap: int,
                 caches: List[Dict[str, torch.Tensor]], kv_len: torch.Tensor, device=None,
                 logits_dtype=torch.float32, inputs_in_place: bool = True):
        """caches: per layer {"Kc", "Vc"} bf16 [B,Hkv,S_cap,d] on the device;
        logits_dtype: float32 or bfloat16 drafter and target logits; inputs_in_place: the kernels read
        the pinned inputs over the host link (only the queries are copied), else every part is copied."""
        if logits_dtype not in (torch.float32, torch.bfloat16):
            raise ValueError("logits_dtype must be torch.float32 or torch.bfloat16")
        self.B, self.K, self.V, self.Hq, self.Hkv, self.d, self.S_cap = B, K, V, Hq, Hkv, head_dim, S_cap
        self.device = torch.device("cuda") if device is None else torch.device(device)
        dev = self.device
        self.caches = caches
        self.n_layers = n = len(caches)
        self.ws = binding.Workspace(B, K, V, Hq, Hkv, head_dim, S_cap, device=dev)
        self.kv_len = kv_len.to(dev, torch.int32).contiguous()
        f32, i32, bf = torch.float32, torch.int32, torch.bfloat16
        K1 = K + 1
        regions = [("draft_logits", (B, K, V), logits_dtype), ("draft_tokens", (B, K), i32),
                   ("temperature", (B,), f32), ("cost_table", (K1,), f32),
                   ("Q", (n, B, K1, Hq, head_dim), bf), ("kv_new", (n, 2, B, Hkv, K1, head_dim), bf),
                   ("target_logits", (B, K1, V), logits_dtype), ("rng", (3,), torch.int64)]
        offs, total = _layout(regions)
        # the three parts a round copies in, in the order its steps need them
        self._parts = [(0, offs["Q"]), (offs["Q"], offs["target_logits"]), (offs["target_logits"], total)]
        self._host_stage = torch.empty(total, dtype=torch.uint8, pin_memory=True)
        self._dev_stage = torch.empty(total, dtype=torch.uint8, device=dev)

        def views(buf):
            out = {}
            for name, shape, dtype in regions:
                nbytes = torch.empty((), dtype=dtype).element_size()
                for s in shape:
                    nbytes *= s
                out[name] = buf[offs[name]:offs[name] + nbytes].view(dtype).view(shape)
            return out

        self._host = views(self._host_stage)
        self._dev = views(self._dev_stage)
        self.in_place = bool(inputs_in_place)
        # in place: everything but the queries is read from the pinned buffer (part 1 is copied up to
        # the new keys and values, i.e. the queries only)
        d = dict(self._dev)
        copy_parts = (True, True, True)
        if self.in_place:
            for name in ("draft_logits", "draft_tokens", "temperature", "cost_table", "kv_new", "target_logits",
                         "rng"):
                d[name] = self._host[name]
            self._parts[1] = (offs["Q"], offs["kv_new"])
            copy_parts = (False, True, False)
        self._copied = sum(b - a for (a, b), c in zip(self._parts, copy_parts) if c)
        self.draft_logits, self.target_logits = d["draft_logits"], d["target_logits"]
        self.draft_tokens, self.temperature, self.cost_table = d["draft_tokens"], d["temperature"], d["cost_table"]
        self.layers = [{"Q": self._dev["Q"][l], "Kc": c["Kc"], "Vc": c["Vc"]} for l, c in enumerate(caches)]
        self.out = binding.RoundOutputs(
            torch.empty((B, K), dtype=f32, device=dev), torch.empty((B, K, 2), dtype=f32, device=dev),
            torch.empty((B,), dtype=i32, device=dev), torch.empty((B,), dtype=i32, device=dev),
            torch.empty((B,), dtype=i32, device=dev),
            [torch.empty((B, K1, Hq, head_dim), dtype=bf, device=dev) for _ in caches], None)
        self.result_host = torch.empty((2, B), dtype=i32, pin_memory=True)
        # the staged round runs on its own stream (a graph cannot be captured on the legacy default one)
        self._stream = torch.cuda.Stream(device=dev)
        self._staged = binding.StagedRound(
            [self._host_stage[a:b] for a, b in self._parts], [self._dev_stage[a:b] for a, b in self._parts],
            d["kv_new"], self.result_host[0], self.result_host[1], self.draft_logits, self.draft_tokens,
            self.temperature, self.cost_table, self.target_logits, self.layers, self.kv_len, self.out, self.ws,
            self._host["rng"], d["rng"], copy_parts=copy_parts)
        self._dims = (B, K, V, n, Hq, Hkv, head_dim, torch.empty((), dtype=logits_dtype).element_size())

    def host_inputs(self) -> Dict[str, torch.Tensor]:
        """Pinned host views to fill before ``run_staged``: draft_logits [B,K,V], target_logits [B,K+1,V],
        draft_tokens [B,K], temperature [B], cost_table [K+1], Q [n_layers,B,K+1,Hq,d] and kv_new
        [n_layers,2,B,Hkv,K+1,d] (layer l's new keys [l,0] and values [l,1] of the verified block)."""
        return {k: v for k, v in self._host.items() if k != "rng"}

    def run_device(self, seed: int, round_offset: int = 0, seq_offset: int = 0, stream=None):
        """The round on inputs resident in this object's device buffers (the new keys and values already
        in the caches). Reading in place, the host buffer is first copied to the device buffers."""
        if self.in_place:
            self._dev_stage.copy_(self._host_stage, non_blocking=True)
        d = self._dev
        return binding.libraspec_verify_round(
            d["draft_logits"], d["draft_tokens"], d["temperature"], d["cost_table"], d["target_logits"],
            [{"Q": d["Q"][l], "Kc": c["Kc"], "Vc": c["Vc"]} for l, c in enumerate(self.caches)], self.kv_len, seed,
            self.ws, round_offset=round_offset, seq_offset=seq_offset, outputs=self.out, stream=stream)

    def h2d_bytes(self, L=None, n_accepted=None, temperature=None) -> int:
        """Bytes that move host -> device per round. Copying every part: the whole pinned buffer. In
        place: the copied queries, plus what the kernels read over the link: the drafter block, the
        new keys and values, and the target rows acceptance reads given the round's lengths L,
        accepted counts and temperatures (rows 0..L_b, and a rejected sampling sequence's target and
        drafter rows at the rejection once more); without them, every target row."""
        if not self.in_place:
            return self._host_stage.numel()
        B, K, V, n, Hq, Hkv, d, eb = self._dims
        h = self._host
        small = sum(h[k].numel() * h[k].element_size() for k in ("draft_tokens", "temperature", "cost_table", "rng"))
        drafter = B * K * V * eb
        kv_new = h["kv_new"].numel() * h["kv_new"].element_size()
        if L is None:
            target = B * (K + 1) * V * eb
        else:
            import numpy as np

            L = np.asarray(L)
            rows = int(np.sum(L + 1))
            if n_accepted is not None and temperature is not None:
                rows += 2 * int(np.sum((np.asarray(n_accepted) < L) & (np.asarray(temperature) > 0)))
            target = rows * V * eb
        return self._copied + drafter + small + kv_new + target

    def d2h_bytes(self) -> int:
        return self.result_host.numel() * 4

    def run_staged(self, seed: int, round_offset: int = 0, seq_offset: int = 0):
        """One round from the pinned host inputs (``host_inputs``), by libraspec_verify_round_staged: the
        three parts are copied in on a side stream; confidence and selection start once the drafter
        part has landed, the key/value append and the attention layers once the layer part has,
        acceptance once the target rows have; the results come back into pinned memory. Returns
        (n_accepted, bonus_token) numpy arrays."""
        self._stream.wait_stream(torch.cuda.current_stream(self.device))
        self._staged(seed, round_offset, seq_offset, stream=self._stream)
        self._stream.synchronize()
        return self.result_host[0].numpy().copy(), self.result_host[1].numpy().copy()

    def run_host(self, host: Dict, seed: int, round_offset: int = 0, seq_offset: int = 0):
        """``run_staged`` from separate host tensors: draft_logits, target_logits, draft_tokens,
        temperature, cost_table and "layers": per layer {"Q", "K_new", "V_new"} (K_new / V_new
        [B,Hkv,K+1,d]), first gathered into the pinned buffer on the host."""
        h = self._host
        for name in ("draft_logits", "target_logits", "draft_tokens", "temperature", "cost_table"):
            h[name].copy_(host[name])
        for l, hl in enumerate(host["layers"]):
            h["Q"][l].copy_(hl["Q"])
            h["kv_new"][l, 0].copy_(hl["K_new"])
            h["kv_new"][l, 1].copy_(hl["V_new"])
        return self.run_staged(seed, round_offset, seq_offset)
