"""Seeded synthetic inputs for the prefix-MoE layer workloads.

This module only draws random numbers and rounds them to the storage dtype. It
holds none of the layer's arithmetic (no routing, no expert math), so both the
CPU oracle side and the CUDA side may take their inputs from it.

The shapes and distributions stand in for a Qwen3-VL-30B-A3B-class MoE decoder
(48 layers, E=128 experts, top-8 routing, hidden 2048, expert FFN width 768,
4 KV heads x 128 dims), as the DecoMoE paper's FLOPs replay states them
(Appendix "Analytical FLOPs Accounting"). The paper's benchmarks and trained
weights are not used: every tensor here is random with a fixed seed.

Per-tensor seed streams: ``seed*1000003 + workload_id*1009 + layer*97 + tensor_id``.
Each stream drives one ``torch.Generator`` on the device the tensor is made on,
so a given (seed, workload, layer, tensor) is reproducible on that device.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional

import torch

# tensor ids inside a layer's seed space
TID_X = 1
TID_WR = 2
TID_WG = 3
TID_WU = 4
TID_WD = 5
TID_LOGITS = 6
TID_KV = 7
TID_KSCHED = 8
TID_RESID = 9


@dataclasses.dataclass(frozen=True)
class Workload:
    """One workload shape. ``K_list`` are prefix lengths (number of retained experts)."""

    name: str
    wid: int            # workload id used in the seed streams
    T: int              # tokens in the invocation
    d: int              # hidden size
    E: int              # experts in the (reordered) pool
    k: int              # top-k routing width
    m: int              # expert FFN width
    dtype: str          # "bf16" or "f32" storage of activations and weights
    x_std: float        # hidden ~ N(0, x_std)
    wr_std: float       # router weight ~ N(0, wr_std)
    w_std: float        # expert weights ~ N(0, w_std)
    bias_kind: str      # "linear" (+1 .. -1) or "zipf" (-s*ln(e+1))
    zipf_s: float       # Zipf exponent for "zipf" bias
    K_list: tuple       # prefix lengths this workload is run at
    v0: int             # visual block start row
    nv: int             # visual block length
    layers: int = 1
    exit_layer: Optional[int] = None
    kv_width: int = 512

    @property
    def torch_dtype(self):
        return torch.bfloat16 if self.dtype == "bf16" else torch.float32


def _bias(wl: Workload, E: Optional[int] = None) -> torch.Tensor:
    """Per-expert router logit bias of the workload recipe (fp32)."""
    E = wl.E if E is None else E
    e = torch.arange(E, dtype=torch.float64)
    if wl.bias_kind == "linear":
        b = 1.0 - 2.0 * e / (E - 1)
    elif wl.bias_kind == "zipf":
        b = -wl.zipf_s * torch.log(e + 1.0)
    elif wl.bias_kind == "none":
        b = torch.zeros(E, dtype=torch.float64)
    else:
        raise ValueError(wl.bias_kind)
    return b.to(torch.float32)


# The five workloads: tiny fp32 correctness layer, T=2048 prefill layer,
# decode-size layers, the 48-layer stack, and the T=16384 prefill sweep.
TINY = Workload("tiny_fp32_T64", 1, T=64, d=256, E=16, k=2, m=128, dtype="f32",
                x_std=1.0, wr_std=0.05, w_std=0.02, bias_kind="linear", zipf_s=0.0,
                K_list=(10, 16, 2), v0=8, nv=48)
PREFILL = Workload("prefill_T2048", 2, T=2048, d=2048, E=128, k=8, m=768, dtype="bf16",
                   x_std=1.0, wr_std=0.02, w_std=0.02, bias_kind="zipf", zipf_s=1.1,
                   K_list=(128, 96, 64, 40), v0=0, nv=1792)
DECODE = Workload("decode_K64", 3, T=1, d=2048, E=128, k=8, m=768, dtype="bf16",
                  x_std=1.0, wr_std=0.02, w_std=0.02, bias_kind="zipf", zipf_s=1.1,
                  K_list=(64,), v0=0, nv=0)
DECODE_T = (1, 8, 32, 128)
STACK = Workload("stack48_T1552_exit20", 4, T=1552, d=2048, E=128, k=8, m=768, dtype="bf16",
                 x_std=1.0, wr_std=0.02, w_std=0.02, bias_kind="zipf", zipf_s=1.1,
                 K_list=(128,), v0=16, nv=1280, layers=48, exit_layer=20)
LARGE = Workload("large_T16384_exit12", 5, T=16384, d=2048, E=128, k=8, m=768, dtype="bf16",
                 x_std=1.0, wr_std=0.02, w_std=0.02, bias_kind="zipf", zipf_s=0.8,
                 K_list=(128, 96, 64, 39), v0=0, nv=14336, layers=48, exit_layer=12)
LARGE_FRACTIONS = (1.0, 0.75, 0.5, 0.3)
LARGE_ZIPF = (0.8, 1.2)

WORKLOADS: Dict[str, Workload] = {w.name: w for w in (TINY, PREFILL, DECODE, STACK, LARGE)}


def with_(wl: Workload, **kw) -> Workload:
    """A copy of a workload with some fields replaced (e.g. T, zipf_s, sizes)."""
    return dataclasses.replace(wl, **kw)


def stream(seed: int, wid: int, layer: int, tensor_id: int) -> int:
    return seed * 1000003 + wid * 1009 + layer * 97 + tensor_id


def _gen(device, s: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(s)
    return g


def _normal(shape, std, dtype, device, s):
    """N(0, std) draws in fp32, then rounded to the storage dtype (RNE for bf16)."""
    g = _gen(device, s)
    t = torch.randn(*shape, generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        t.mul_(std)
    return t.to(dtype)


def make_layer(wl: Workload, layer: int = 0, seed: int = 0, device="cpu",
               T: Optional[int] = None, with_x: bool = True) -> Dict[str, torch.Tensor]:
    """Inputs of one MoE layer in the paper's plain (unfused) layout.

    x      [T, d]    hidden states (storage dtype)
    w_r    [E, d]    router weights (storage dtype), rows already in reordered expert order
    bias   [E]       router logit bias (fp32), the workload's skew over reordered index
    w_gate [E, m, d] gate projection per expert
    w_up   [E, m, d] up projection per expert
    w_down [E, d, m] down projection per expert
    """
    T = wl.T if T is None else T
    dt = wl.torch_dtype
    out = {}
    if with_x:
        out["x"] = _normal((T, wl.d), wl.x_std, dt, device, stream(seed, wl.wid, layer, TID_X))
    out["w_r"] = _normal((wl.E, wl.d), wl.wr_std, dt, device, stream(seed, wl.wid, layer, TID_WR))
    out["bias"] = _bias(wl).to(device)
    out["w_gate"] = _normal((wl.E, wl.m, wl.d), wl.w_std, dt, device, stream(seed, wl.wid, layer, TID_WG))
    out["w_up"] = _normal((wl.E, wl.m, wl.d), wl.w_std, dt, device, stream(seed, wl.wid, layer, TID_WU))
    out["w_down"] = _normal((wl.E, wl.d, wl.m), wl.w_std, dt, device, stream(seed, wl.wid, layer, TID_WD))
    return out


def make_x(wl: Workload, T: Optional[int] = None, layer: int = 0, seed: int = 0, device="cpu",
           tensor_id: int = TID_X) -> torch.Tensor:
    T = wl.T if T is None else T
    return _normal((T, wl.d), wl.x_std, wl.torch_dtype, device, stream(seed, wl.wid, layer, tensor_id))


def make_logits(T: int, E: int, std: float = 0.9, bias: Optional[torch.Tensor] = None,
                seed: int = 0, wid: int = 0, layer: int = 0, device="cpu") -> torch.Tensor:
    """fp32 router logits drawn directly: N(0, std) per entry plus a per-expert bias.

    std=0.9 matches the spread of x.W_r for x~N(0,1), W_r~N(0,0.02), d=2048.
    """
    g = _gen(device, stream(seed, wid, layer, TID_LOGITS))
    a = torch.randn(T, E, generator=g, device=device, dtype=torch.float32) * std
    if bias is not None:
        a = a + bias.to(device=device, dtype=torch.float32)[None, :]
    return a


def make_kv(wl: Workload, seed: int = 0, device="cpu", T: Optional[int] = None,
            layers: Optional[int] = None) -> torch.Tensor:
    """Per-layer KV buffer [L, T, kv_width] in bf16 (K or V, one of the two)."""
    T = wl.T if T is None else T
    L = wl.layers if layers is None else layers
    return _normal((L, T, wl.kv_width), 1.0, torch.bfloat16, device,
                   stream(seed, wl.wid, 0, TID_KV))


def stack_K_schedule(wl: Workload, seed: int = 0) -> List[int]:
    """Prefix length per layer of the 48-layer stack.

    Layers before the exit layer run the full pool (K=E). Layers from the exit
    layer on draw K_l uniformly from the integers 32..96 (inclusive).
    """
    import numpy as np

    rng = np.random.default_rng(stream(seed, wl.wid, 0, TID_KSCHED))
    n_after = wl.layers - wl.exit_layer
    ks = rng.integers(32, 97, size=n_after).tolist()
    return [wl.E] * wl.exit_layer + [int(v) for v in ks]


def large_K(fraction: float, E: int = 128) -> int:
    """Prefix length for a retained fraction f of the pool: ceil(f*E) (0.3*128 -> 39)."""
    return int(math.ceil(fraction * E - 1e-9))


def make_gate_params(d: int, H: int, candidates, fire_at: Optional[int], seed: int = 0, device="cpu",
                     margin: float = 8.0):
    """Synthetic SAVB gate parameters for each candidate layer (the trained
    checkpoint is not available): W1 ~ N(0, 1/(2d)), b1 ~ N(0, 0.1),
    W2 ~ N(0, 1/H), and an output bias b2 = (+margin, -margin) at every
    candidate except ``fire_at``, where it is (-margin, +margin), so the gate
    computes its full MLP everywhere and fires at that candidate.
    Returns {layer: (w1 [H, 2d], b1 [H], w2 [2, H], b2 [2])} fp32."""
    out = {}
    for l in candidates:
        g = _gen("cpu", stream(seed, 90, l, 0))
        w1 = torch.randn(H, 2 * d, generator=g) / (2 * d) ** 0.5
        b1 = torch.randn(H, generator=g) * 0.1
        w2 = torch.randn(2, H, generator=g) / H ** 0.5
        b2 = torch.tensor([-margin, margin] if l == fire_at else [margin, -margin])
        out[l] = tuple(t.to(device=device, dtype=torch.float32).contiguous() for t in (w1, b1, w2, b2))
    return out
