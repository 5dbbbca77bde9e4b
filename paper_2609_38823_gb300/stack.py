"""Attention-free decoder stack over the C ABI: the layer schedule of a
DecoMoE prefill (Algorithm 2) without attention.

Each layer computes h <- h + MoE_l(RMSNorm(h)) with its own prefix length K_l.
At the entrance of the exit layer (the first text-only layer, where SAVB
triggers) the contiguous visual block leaves the hidden state and every layer
slice of the K and V caches (Section 3.2); later layers run on the text rows
only. Every step is a library call; this module only sequences them and owns
the buffers.
"""
from __future__ import annotations

from typing import List, Optional, Sequence

import torch

from . import (DECOMOE_BF16, DECOMOE_F32, decomoe_drop_visual_block, decomoe_moe_layer,
               decomoe_moe_layer_workspace_bytes, decomoe_rmsnorm, workspace)


class StackLayer:
    """Device weights of one layer (gate/up already in the fused layout)."""

    def __init__(self, w_r, bias, w_gate_up, w_down):
        self.w_r = w_r
        self.bias = bias
        self.w_gate_up = w_gate_up
        self.w_down = w_down


class Stack:
    def __init__(self, layers: Sequence[StackLayer], K_sched: Sequence[int], k: int, exit_layer: Optional[int],
                 v0: int, nv: int, T: int, eps: float = 1e-6):
        assert len(K_sched) == len(layers)
        self.layers = list(layers)
        self.K = [int(v) for v in K_sched]
        self.k = k
        self.exit = exit_layer
        self.v0, self.nv, self.T = v0, nv, T
        self.eps = eps
        w0 = layers[0]
        self.d = w0.w_r.shape[1]
        self.E = w0.w_r.shape[0]
        self.m = w0.w_down.shape[2]
        self.dtype = w0.w_r.dtype
        dev = w0.w_r.device
        dt = DECOMOE_BF16 if self.dtype == torch.bfloat16 else DECOMOE_F32
        self.ws = workspace(decomoe_moe_layer_workspace_bytes(T, self.d, self.E, k, self.m, dt), dev)
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)
        Tt = T - (nv if exit_layer is not None else 0)
        # ping-pong hidden buffers for the full and the text-only sequence
        self.hf = [torch.empty(T, self.d, dtype=self.dtype, device=dev) for _ in range(2)]
        self.ht = [torch.empty(Tt, self.d, dtype=self.dtype, device=dev) for _ in range(2)]
        self.xn_f = torch.empty(T, self.d, dtype=self.dtype, device=dev)
        self.xn_t = torch.empty(Tt, self.d, dtype=self.dtype, device=dev)

    def forward(self, h0: torch.Tensor, kv: Optional[List[torch.Tensor]] = None,
                kv_out: Optional[List[torch.Tensor]] = None) -> torch.Tensor:
        """Run every layer on h0 [T, d]; returns the final hidden state (text
        rows only when the exit layer is inside the stack). kv: K and V caches
        [L, T, w]; kv_out: their compacted destinations [L, T - nv, w]."""
        cur = self.hf[0]
        cur.copy_(h0)
        bufs, xn, nxt = self.hf, self.xn_f, 1
        for l, Lw in enumerate(self.layers):
            if self.exit is not None and l == self.exit:
                dst = self.ht[0]
                decomoe_drop_visual_block(cur, dst, self.v0, self.nv)
                if kv is not None:
                    for src, out in zip(kv, kv_out):
                        decomoe_drop_visual_block(src, out, self.v0, self.nv)
                cur, bufs, xn, nxt = dst, self.ht, self.xn_t, 1
            decomoe_rmsnorm(cur, xn, self.eps)
            out = bufs[nxt]
            decomoe_moe_layer(xn, Lw.w_r, Lw.bias, Lw.w_gate_up, Lw.w_down, self.k, out, self.ws,
                              K_fixed=self.K[l], p=0.0, residual=cur, status=self.status)
            cur, nxt = out, 1 - nxt
        return cur
