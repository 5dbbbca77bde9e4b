"""Attention-free decoder stack over the C ABI: the layer schedule of a
DecoMoE prefill (Algorithm 2) without attention.

Each layer computes h <- h + MoE_l(RMSNorm(h)). Before the visual exit every
layer runs on the full sequence with its K_l (the full pool in the paper);
from the exit on, layers run on the text rows only, with either a fixed K_l
or the prefix selected from the activated mass with fraction p (Eq. 12, on
the device). The exit is either a fixed layer (the first text-only layer) or
decided by the SAVB gate (Eqs. 2-3): at each candidate layer l the gate reads
the output of layer l, and when it fires the visual block leaves the hidden
state and every layer slice of the K and V caches before layer l + 1 (the
zero-based trigger convention of the paper's appendix). Every step is a
library call; this module only sequences them and owns the buffers.
"""
from __future__ import annotations

from typing import Dict, List, Optional, Sequence, Tuple

import torch

from . import (DECOMOE_BF16, DECOMOE_F32, decomoe_drop_visual_block, decomoe_drop_visual_block_if, decomoe_moe_layer,
               decomoe_moe_layer_workspace_bytes, decomoe_rmsnorm, decomoe_savb_gate,
               decomoe_savb_gate_workspace_bytes, workspace)


class StackLayer:
    """Device weights of one layer (gate/up already in the fused layout)."""

    def __init__(self, w_r, bias, w_gate_up, w_down):
        self.w_r = w_r
        self.bias = bias
        self.w_gate_up = w_gate_up
        self.w_down = w_down


class SavbGate:
    """Per-candidate-layer gate parameters (the paper trains an independent
    two-class MLP at each candidate position): {layer: (w1 [H, 2d], b1 [H],
    w2 [2, H], b2 [2])}, fp32 on the device, and the threshold theta."""

    def __init__(self, params: Dict[int, Tuple[torch.Tensor, ...]], theta: float = 0.5):
        self.params = dict(params)
        self.theta = float(theta)


class Stack:
    def __init__(self, layers: Sequence[StackLayer], K_sched: Sequence[int], k: int, exit_layer: Optional[int],
                 v0: int, nv: int, T: int, eps: float = 1e-6, gate: Optional[SavbGate] = None,
                 p_after_exit: Optional[float] = None, select_on_host: bool = False):
        assert len(K_sched) == len(layers)
        assert exit_layer is None or gate is None, "a fixed exit layer or a gate, not both"
        self.layers = list(layers)
        self.K = [int(v) for v in K_sched]
        self.k = k
        self.exit = exit_layer
        self.gate = gate
        self.p = p_after_exit
        self.select_on_host = select_on_host  # Eq. 12 in host C after a sync, instead of on the device
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
        Tt = T - nv
        # ping-pong hidden buffers for the full and the text-only sequence
        self.hf = [torch.empty(T, self.d, dtype=self.dtype, device=dev) for _ in range(2)]
        self.ht = [torch.empty(Tt, self.d, dtype=self.dtype, device=dev) for _ in range(2)]
        self.xn_f = torch.empty(T, self.d, dtype=self.dtype, device=dev)
        self.xn_t = torch.empty(Tt, self.d, dtype=self.dtype, device=dev)
        if gate is not None:
            H = max(p[0].shape[0] for p in gate.params.values())
            self.gate_ws = workspace(decomoe_savb_gate_workspace_bytes(self.d, H), dev)
            self.p_exit = torch.zeros(len(layers), dtype=torch.float32, device=dev)
            self.exit_flag = torch.zeros(len(layers), dtype=torch.int32, device=dev)
        self.exit_taken: Optional[int] = None  # first text-only layer of the last forward

    def _compact(self, cur, kv, kv_out, flag=None):
        """Remove the visual block from the hidden state (into ht[0]) and the
        KV caches; with flag (the gate's device-side decision) only when it
        holds 1."""
        dst = self.ht[0]
        if flag is None:
            decomoe_drop_visual_block(cur, dst, self.v0, self.nv)
        else:
            decomoe_drop_visual_block_if(flag, cur, dst, self.v0, self.nv)
        if kv is not None:
            for src, out in zip(kv, kv_out):
                if flag is None:
                    decomoe_drop_visual_block(src, out, self.v0, self.nv)
                else:
                    decomoe_drop_visual_block_if(flag, src, out, self.v0, self.nv)
        return dst

    def forward(self, h0: torch.Tensor, kv: Optional[List[torch.Tensor]] = None,
                kv_out: Optional[List[torch.Tensor]] = None, trace=None) -> torch.Tensor:
        """Run every layer on h0 [T, d]; returns the final hidden state (text
        rows only once the visual block has left). kv: K and V caches
        [L, T, w]; kv_out: their compacted destinations [L, T - nv, w]. With a
        gate, each candidate layer's decision is read back to the host (one
        4-byte copy) because the exit changes the shapes of later launches.
        trace, if given, is called after each layer's launches are queued as
        trace(l, layer_input, normed_input, layer_output, workspace), so a
        caller can inspect any layer's inputs and results (the buffers are
        reused by later layers)."""
        cur = self.hf[0]
        cur.copy_(h0)
        bufs, xn, nxt = self.hf, self.xn_f, 1
        exited = False
        self.exit_taken = None
        for l, Lw in enumerate(self.layers):
            if not exited and self.exit is not None and l == self.exit:
                cur = self._compact(cur, kv, kv_out)
                bufs, xn, nxt, exited = self.ht, self.xn_t, 1, True
                self.exit_taken = l
            decomoe_rmsnorm(cur, xn, self.eps)
            out = bufs[nxt]
            if exited and self.p is not None:
                decomoe_moe_layer(xn, Lw.w_r, Lw.bias, Lw.w_gate_up, Lw.w_down, self.k, out, self.ws,
                                  K_fixed=0 if self.select_on_host else -1, p=self.p, residual=cur,
                                  status=self.status)
            else:
                decomoe_moe_layer(xn, Lw.w_r, Lw.bias, Lw.w_gate_up, Lw.w_down, self.k, out, self.ws,
                                  K_fixed=self.K[l], p=0.0, residual=cur, status=self.status)
            if trace is not None:
                trace(l, cur, xn, out, self.ws)
            cur, nxt = out, 1 - nxt
            if self.gate is not None and not exited and l in self.gate.params and l + 1 < len(self.layers):
                w1, b1, w2, b2 = self.gate.params[l]
                flag = self.exit_flag[l:l + 1]
                decomoe_savb_gate(cur, self.v0, self.nv, w1, b1, w2, b2, self.gate.theta, self.p_exit[l:l + 1],
                                  flag, self.gate_ws)
                # the removal is queued behind the gate and reads its decision
                # on the device; the host reads the decision afterwards (the
                # later launches' shapes depend on it)
                dst = self._compact(cur, kv, kv_out, flag)
                if int(flag.item()) == 1:
                    cur = dst
                    bufs, xn, nxt, exited = self.ht, self.xn_t, 1, True
                    self.exit_taken = l + 1
        return cur
