"""Python binding of libdecomoe (the DecoMoE prefix-MoE hot path on GB300).

Argument marshalling only: every function here forwards torch tensors' device
pointers, sizes and the current CUDA stream to the C ABI of include/decomoe.h,
and raises DecomoeError on a non-zero status. No step of the computation runs
in Python or in PyTorch ops; PyTorch provides device memory and streams.

The shared library is built in-tree (``__graft_entry__.build()`` or
``python paper_2609_38823_gb300/_build.py``). Importing this package does not
need a GPU; calling a device function without the library or without a GPU
raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libdecomoe.so")

DECOMOE_OK = 0
DECOMOE_ERR_INVALID_ARG = 1
DECOMOE_ERR_CUDA = 2
DECOMOE_ERR_TIMEOUT = 3
DECOMOE_ERR_UNSUPPORTED = 4
DECOMOE_ERR_WORKSPACE = 5
DECOMOE_ERR_BAD_INPUT = 6
DECOMOE_BF16 = 0
DECOMOE_F32 = 1
GU_BLOCK = 64

# name -> (restype, argtypes)
_P = ctypes.c_void_p
_I = ctypes.c_int
_L = ctypes.c_int64
_S = ctypes.c_size_t
_D = ctypes.c_double
_F = ctypes.c_float
SIGNATURES = {
    "decomoe_last_error": (ctypes.c_char_p, []),
    "decomoe_version": (_I, []),
    "decomoe_device_info": (_I, [_P, _P, _P]),
    "decomoe_router_logits": (_I, [_P, _P, _P, _L, _I, _I, _I, _P, _P, _P]),
    "decomoe_router_logits_ws_bytes": (_S, [_L, _I, _I]),
    "decomoe_router_logits_ws": (_I, [_P, _P, _P, _L, _I, _I, _I, _P, _P, _S, _P, _P]),
    "decomoe_route_workspace_bytes": (_S, [_L, _I]),
    "decomoe_route_prefix": (_I, [_P, _L, _I, _L, _I, _I, _P, _P, _P, _P, _S, _P]),
    "decomoe_select_prefix": (_I, [_P, _I, _I, _D, _P]),
    "decomoe_select_prefix_device": (_I, [_P, _I, _I, _D, _P, _P]),
    "decomoe_route_prefix_dk": (_I, [_P, _L, _I, _L, _P, _I, _P, _P, _P]),
    "decomoe_dispatch_workspace_bytes": (_S, [_L, _I, _I]),
    "decomoe_route_dispatch_workspace_bytes": (_S, [_L, _I, _I]),
    "decomoe_route_dispatch": (_I, [_P, _L, _I, _I, _I, _D, _P, _P, _P, _P, _P, _I, _I, _P, _P, _P, _P, _P, _P, _S,
                                    _P, _P]),
    "decomoe_expert_swiglu_ready_ints": (_S, [_L, _I]),
    "decomoe_expert_swiglu_fused": (_I, [_P, _P, _L, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P]),
    "decomoe_gather_rows": (_I, [_P, _P, _P, _I, _L, _I, _I, _P, _P]),
    "decomoe_attention_workspace_bytes": (_S, [_L, _L, _I, _I, _I]),
    "decomoe_attention": (_I, [_P, _L, _P, _P, _L, _I, _I, _I, _F, _P, _P, _S, _P, _P]),
    "decomoe_expert_swiglu_fused_gather": (_I, [_P, _L, _P, _P, _L, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P,
                                                _P]),
    "decomoe_router_route_dispatch_workspace_bytes": (_S, [_L, _I, _I, _I]),
    "decomoe_router_route_dispatch": (_I, [_P, _P, _P, _L, _I, _I, _I, _I, _I, _D, _P, _P, _P, _P, _P, _P, _P, _P, _P,
                                           _P, _P, _S, _P, _P]),
    "decomoe_savb_gate_workspace_bytes": (_S, [_I, _I]),
    "decomoe_savb_gate": (_I, [_P, _L, _I, _I, _L, _L, _P, _P, _P, _P, _I, _F, _P, _P, _P, _S, _P]),
    "decomoe_calib_workspace_bytes": (_S, [_L, _I]),
    "decomoe_calib_case_mass": (_I, [_P, _L, _I, _L, _I, _L, _L, _P, _P, _S, _P]),
    "decomoe_mean_mass_order": (_I, [_P, _I, _I, _P, _P, _P, _P]),
    "decomoe_permute_experts": (_I, [_P, _P, _P, _I, _L, _P, _P]),
    "decomoe_dispatch": (_I, [_P, _L, _I, _I, _P, _I, _I, _P, _P, _P, _P, _P, _P, _S, _P, _P]),
    "decomoe_dispatch_noalloc": (_I, [_P, _L, _I, _I, _P, _I, _I, _P, _P, _P, _P, _P, _P, _P]),
    "decomoe_weight_layout": (_I, [_P, _P, _P, _I, _I, _I, _I, _P]),
    "decomoe_expert_swiglu": (_I, [_P, _P, _L, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P]),
    "decomoe_expert_gate_up": (_I, [_P, _P, _L, _I, _I, _I, _I, _P, _P, _P, _P, _P]),
    "decomoe_expert_down": (_I, [_P, _P, _L, _I, _I, _I, _I, _P, _P, _P, _P, _P]),
    "decomoe_expert_gate_up_gather": (_I, [_P, _L, _P, _P, _L, _I, _I, _I, _I, _P, _P, _P, _P, _P]),
    "decomoe_expert_swiglu_gather": (_I, [_P, _L, _P, _P, _L, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P]),
    "decomoe_expert_swiglu_ref": (_I, [_P, _P, _L, _I, _I, _I, _P, _P, _P, _P, _P]),
    "decomoe_combine": (_I, [_P, _P, _P, _L, _I, _I, _I, _P, _P, _P]),
    "decomoe_combine_drop_visual_block": (_I, [_P, _P, _P, _L, _I, _I, _I, _P, _P, _P, _L, _L, _P]),
    "decomoe_drop_visual_block": (_I, [_P, _P, _L, _L, _L, _L, _L, _L, _L, _P]),
    "decomoe_drop_visual_block_if": (_I, [_P, _P, _P, _L, _L, _L, _L, _L, _L, _L, _P]),
    "decomoe_rmsnorm": (_I, [_P, _P, _L, _I, _F, _I, _P]),
    "decomoe_moe_layer_workspace_bytes": (_S, [_L, _I, _I, _I, _I, _I]),
    "decomoe_moe_layer": (_I, [_P, _P, _P, _P, _P, _L, _I, _I, _I, _I, _I, _I, _D, _P, _P, _P, _P,
                               _P, _S, _P, _P]),
    "decomoe_moe_layer_exit": (_I, [_P, _P, _P, _P, _P, _L, _I, _I, _I, _I, _I, _I, _D, _P, _P, _P, _L, _L, _P,
                                    _P, _P, _S, _P, _P]),
    "decomoe_moe_layer_workspace_layout": (_I, [_L, _I, _I, _I, _I, _I, _P]),
    "decomoe_read_status": (_I, [_P, _P, _P]),
    "decomoe_set_wait_limit_ns": (_I, [_L]),
    "decomoe_set_discard_scratch": (_I, [_I]),
    "decomoe_set_pdl": (_I, [_I]),
    "decomoe_selftest_wait": (_I, [_P, _L, _P]),
}


class DecomoeError(RuntimeError):
    def __init__(self, name, code, msg):
        super().__init__(f"{name} failed with status {code}: {msg}")
        self.code = code


_lib = None


def lib() -> ctypes.CDLL:
    """Load libdecomoe.so (raises if it was not built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(
                f"{LIB_PATH} is missing: build it with __graft_entry__.build() "
                "(the CUDA library is required; there is no fallback)")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def _check(name, code):
    if code != DECOMOE_OK:
        msg = lib().decomoe_last_error()
        raise DecomoeError(name, code, msg.decode() if msg else "")


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dt(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return DECOMOE_BF16
    if t.dtype == torch.float32:
        return DECOMOE_F32
    raise TypeError(f"unsupported dtype {t.dtype}")


def _need_cuda(*ts):
    for t in ts:
        if t is not None:
            if not t.is_cuda:
                raise ValueError("device tensors expected")
            if not t.is_contiguous():
                raise ValueError("contiguous tensors expected")


# ----------------------------------------------------------------- host-only calls

def decomoe_version() -> int:
    return lib().decomoe_version()


def decomoe_select_prefix(mass, k: int, p: float) -> int:
    """Eq. 12 on the host (plain C): shortest prefix covering mass fraction p."""
    import numpy as np

    m = np.ascontiguousarray(np.asarray(mass, dtype=np.float64))
    out = ctypes.c_int(0)
    _check("decomoe_select_prefix",
           lib().decomoe_select_prefix(m.ctypes.data_as(ctypes.c_void_p), int(m.shape[0]), int(k),
                                       float(p), ctypes.byref(out)))
    return out.value


def decomoe_route_workspace_bytes(T: int, E: int) -> int:
    return lib().decomoe_route_workspace_bytes(T, E)


def decomoe_dispatch_workspace_bytes(T: int, k: int, K: int) -> int:
    return lib().decomoe_dispatch_workspace_bytes(T, k, K)


def decomoe_moe_layer_workspace_bytes(T, d, E, k, m, dtype) -> int:
    return lib().decomoe_moe_layer_workspace_bytes(T, d, E, k, m, dtype)


def decomoe_moe_layer_workspace_layout(T, d, E, k, m, dtype):
    offs = (ctypes.c_size_t * 12)()
    _check("decomoe_moe_layer_workspace_layout",
           lib().decomoe_moe_layer_workspace_layout(T, d, E, k, m, dtype, offs))
    return list(offs)


def decomoe_set_wait_limit_ns(limit_ns: int):
    _check("decomoe_set_wait_limit_ns", lib().decomoe_set_wait_limit_ns(int(limit_ns)))


def decomoe_set_discard_scratch(on: bool):
    _check("decomoe_set_discard_scratch", lib().decomoe_set_discard_scratch(1 if on else 0))


def decomoe_set_pdl(on: bool):
    _check("decomoe_set_pdl", lib().decomoe_set_pdl(1 if on else 0))


def decomoe_device_info():
    a, b, c = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    _check("decomoe_device_info", lib().decomoe_device_info(ctypes.byref(a), ctypes.byref(b), ctypes.byref(c)))
    return a.value, b.value, c.value


# ----------------------------------------------------------------- device calls

def decomoe_router_logits(x, w_r, bias, logits, status=None, stream=None):
    _need_cuda(x, w_r, bias, logits, status)
    T, d = x.shape
    E = w_r.shape[0]
    _check("decomoe_router_logits",
           lib().decomoe_router_logits(_ptr(x), _ptr(w_r), _ptr(bias), T, d, E, _dt(x), _ptr(logits),
                                       _ptr(status), _stream(stream)))


def decomoe_router_logits_ws_bytes(T, d, E):
    return int(lib().decomoe_router_logits_ws_bytes(T, d, E))


def decomoe_router_logits_ws(x, w_r, bias, logits, ws, status=None, stream=None):
    """Router logits with a workspace (k-split tensor-core path at large T)."""
    _need_cuda(x, w_r, bias, logits, ws, status)
    T, d = x.shape
    E = w_r.shape[0]
    _check("decomoe_router_logits_ws",
           lib().decomoe_router_logits_ws(_ptr(x), _ptr(w_r), _ptr(bias), T, d, E, _dt(x), _ptr(logits), _ptr(ws),
                                          0 if ws is None else ws.numel() * ws.element_size(), _ptr(status),
                                          _stream(stream)))


def decomoe_route_prefix(logits, K, k, topk_idx=None, topk_w=None, mass_out=None, ws=None, E=None,
                         stream=None):
    _need_cuda(logits, topk_idx, topk_w, mass_out, ws)
    T, ld = logits.shape
    E = ld if E is None else E
    ws_bytes = 0 if ws is None else ws.numel() * ws.element_size()
    _check("decomoe_route_prefix",
           lib().decomoe_route_prefix(_ptr(logits), T, E, ld, K, k, _ptr(topk_idx), _ptr(topk_w),
                                      _ptr(mass_out), _ptr(ws), ws_bytes, _stream(stream)))


def decomoe_select_prefix_device(mass, k, p, K_dev, stream=None):
    _need_cuda(mass, K_dev)
    _check("decomoe_select_prefix_device",
           lib().decomoe_select_prefix_device(_ptr(mass), mass.shape[0], k, float(p), _ptr(K_dev), _stream(stream)))


def decomoe_route_prefix_dk(logits, K_dev, k, topk_idx, topk_w, stream=None):
    _need_cuda(logits, K_dev, topk_idx, topk_w)
    T, E = logits.shape
    _check("decomoe_route_prefix_dk",
           lib().decomoe_route_prefix_dk(_ptr(logits), T, E, E, _ptr(K_dev), k, _ptr(topk_idx), _ptr(topk_w),
                                         _stream(stream)))


def decomoe_route_dispatch_workspace_bytes(T, k, E):
    return int(lib().decomoe_route_dispatch_workspace_bytes(T, k, E))


def decomoe_route_dispatch(logits, K, k, topk_idx, topk_w, x, counts, offsets, perm_token, inv_slot, x_perm, ws,
                           p=0.0, mass_out=None, K_dev=None, status=None, stream=None):
    """Routing and dispatch in one call: K >= k a fixed prefix (mass_out
    optional), K = -1 the prefix selected on the device from p (mass_out and
    K_dev required; dispatch then runs over all E groups)."""
    _need_cuda(logits, topk_idx, topk_w, x, counts, offsets, perm_token, inv_slot, x_perm, ws, mass_out, K_dev,
               status)
    T, E = logits.shape
    d = x.shape[1] if x is not None else 0
    dtype = _dt(x) if x is not None else DECOMOE_BF16
    _check("decomoe_route_dispatch",
           lib().decomoe_route_dispatch(_ptr(logits), T, E, K, k, float(p), _ptr(topk_idx), _ptr(topk_w),
                                        _ptr(mass_out), _ptr(K_dev), _ptr(x), d, dtype, _ptr(counts), _ptr(offsets),
                                        _ptr(perm_token), _ptr(inv_slot), _ptr(x_perm), _ptr(ws),
                                        0 if ws is None else ws.numel() * ws.element_size(), _ptr(status),
                                        _stream(stream)))


def decomoe_router_route_dispatch_workspace_bytes(T, d, E, k):
    return int(lib().decomoe_router_route_dispatch_workspace_bytes(T, d, E, k))


def decomoe_router_route_dispatch(x, w_r, bias, logits, K, k, topk_idx, topk_w, counts, offsets, perm_token,
                                  inv_slot, x_perm, ws, p=0.0, mass_out=None, K_dev=None, status=None, stream=None):
    """Router logits, routing and dispatch in one call (the same results as
    decomoe_router_logits_ws followed by decomoe_route_dispatch)."""
    _need_cuda(x, w_r, bias, logits, topk_idx, topk_w, counts, offsets, perm_token, inv_slot, x_perm, ws, mass_out,
               K_dev, status)
    T, d = x.shape
    E = w_r.shape[0]
    _check("decomoe_router_route_dispatch",
           lib().decomoe_router_route_dispatch(_ptr(x), _ptr(w_r), _ptr(bias), T, d, E, _dt(x), K, k, float(p),
                                               _ptr(logits), _ptr(topk_idx), _ptr(topk_w), _ptr(mass_out),
                                               _ptr(K_dev), _ptr(counts), _ptr(offsets), _ptr(perm_token),
                                               _ptr(inv_slot), _ptr(x_perm), _ptr(ws),
                                               0 if ws is None else ws.numel() * ws.element_size(), _ptr(status),
                                               _stream(stream)))


def decomoe_dispatch(topk_idx, K, x, counts, offsets, perm_token, inv_slot, x_perm, ws, status=None,
                     stream=None):
    _need_cuda(topk_idx, x, counts, offsets, perm_token, inv_slot, x_perm, ws, status)
    T, k = topk_idx.shape
    d = x.shape[1] if x is not None else 0
    dtype = _dt(x) if x is not None else DECOMOE_BF16
    _check("decomoe_dispatch",
           lib().decomoe_dispatch(_ptr(topk_idx), T, k, K, _ptr(x), d, dtype, _ptr(counts), _ptr(offsets),
                                  _ptr(perm_token), _ptr(inv_slot), _ptr(x_perm), _ptr(ws),
                                  ws.numel() * ws.element_size(), _ptr(status), _stream(stream)))


def decomoe_dispatch_noalloc(topk_idx, K, x, counts, offsets, perm_token, inv_slot, x_perm, status=None,
                             stream=None):
    """decomoe_dispatch without a workspace: for callers that cannot allocate
    device memory; its scratch is a fixed array inside the library (see the
    header for the size limit and the rule that overlapping calls race)."""
    _need_cuda(topk_idx, x, counts, offsets, perm_token, inv_slot, x_perm, status)
    T, k = topk_idx.shape
    d = x.shape[1] if x is not None else 0
    dtype = _dt(x) if x is not None else DECOMOE_BF16
    _check("decomoe_dispatch_noalloc",
           lib().decomoe_dispatch_noalloc(_ptr(topk_idx), T, k, K, _ptr(x), d, dtype, _ptr(counts), _ptr(offsets),
                                          _ptr(perm_token), _ptr(inv_slot), _ptr(x_perm), _ptr(status),
                                          _stream(stream)))


# ----------------------------------------------------------------- SAVB gate and RCEP calibration

def decomoe_savb_gate_workspace_bytes(d, H):
    return int(lib().decomoe_savb_gate_workspace_bytes(d, H))


def decomoe_savb_gate(h, v0, nv, w1, b1, w2, b2, theta, p_exit, exit_flag, ws, stream=None):
    """SAVB exit gate on hidden h [T, d] (Eqs. 2-3); writes p_exit [1] fp32 and
    exit_flag [1] int32 on the device."""
    _need_cuda(h, w1, b1, w2, b2, p_exit, exit_flag, ws)
    T, d = h.shape
    H = w1.shape[0]
    _check("decomoe_savb_gate",
           lib().decomoe_savb_gate(_ptr(h), T, d, _dt(h), v0, nv, _ptr(w1), _ptr(b1), _ptr(w2), _ptr(b2), H,
                                   float(theta), _ptr(p_exit), _ptr(exit_flag), _ptr(ws),
                                   ws.numel() * ws.element_size(), _stream(stream)))


def decomoe_calib_workspace_bytes(T, E):
    return int(lib().decomoe_calib_workspace_bytes(T, E))


def decomoe_calib_case_mass(logits, k, v0, nv, accum, ws, E=None, stream=None):
    """accum [E] fp64 += the case's text-token routed mass (Eq. 9)."""
    _need_cuda(logits, accum, ws)
    T, ld = logits.shape
    E = ld if E is None else E
    _check("decomoe_calib_case_mass",
           lib().decomoe_calib_case_mass(_ptr(logits), T, E, ld, k, v0, nv, _ptr(accum), _ptr(ws),
                                         ws.numel() * ws.element_size(), _stream(stream)))


def decomoe_mean_mass_order(accum, n_cases, pi, mean_out=None, status=None, stream=None):
    """Eq. 8: pi [E] int32 = experts by descending case-mean routed mass."""
    _need_cuda(accum, pi, mean_out, status)
    _check("decomoe_mean_mass_order",
           lib().decomoe_mean_mass_order(_ptr(accum), accum.shape[0], n_cases, _ptr(pi), _ptr(mean_out),
                                         _ptr(status), _stream(stream)))


def decomoe_permute_experts(src, dst, pi, status=None, stream=None):
    """dst[i] = src[pi[i]] over the leading (expert) dimension, out of place."""
    _need_cuda(src, dst, pi, status)
    E = src.shape[0]
    if dst.shape != src.shape or dst.dtype != src.dtype or pi.shape[0] != E:
        raise ValueError("src, dst and pi must agree in shape")
    _check("decomoe_permute_experts",
           lib().decomoe_permute_experts(_ptr(src), _ptr(dst), _ptr(pi), E, src[0].numel() * src.element_size()
                                         if E > 0 else 0, _ptr(status), _stream(stream)))


def decomoe_weight_layout(w_gate, w_up, w_gate_up, stream=None):
    _need_cuda(w_gate, w_up, w_gate_up)
    E, m, d = w_gate.shape
    _check("decomoe_weight_layout",
           lib().decomoe_weight_layout(_ptr(w_gate), _ptr(w_up), _ptr(w_gate_up), E, d, m, _dt(w_gate),
                                       _stream(stream)))


def decomoe_expert_swiglu(x_perm, offsets, K, w_gate_up, w_down, h_ws, y_perm, status=None, sched=None,
                          stream=None):
    _need_cuda(x_perm, offsets, w_gate_up, w_down, h_ws, y_perm, status, sched)
    rows, d = x_perm.shape
    m = w_down.shape[2]
    _check("decomoe_expert_swiglu",
           lib().decomoe_expert_swiglu(_ptr(x_perm), _ptr(offsets), rows, K, d, m, _dt(x_perm),
                                       _ptr(w_gate_up), _ptr(w_down), _ptr(h_ws), _ptr(y_perm),
                                       _ptr(status), _ptr(sched), _stream(stream)))


def decomoe_expert_swiglu_ready_ints(rows, K):
    return int(lib().decomoe_expert_swiglu_ready_ints(rows, K))


def decomoe_expert_swiglu_fused(x_perm, offsets, K, w_gate_up, w_down, h, y_perm, ready, status=None, stream=None):
    """Both expert GEMMs, in one launch where that is faster; ready: int32
    counters, zero at the call (decomoe_expert_swiglu_ready_ints)."""
    _need_cuda(x_perm, offsets, w_gate_up, w_down, h, y_perm, ready, status)
    rows, d = x_perm.shape
    m = h.shape[1]
    _check("decomoe_expert_swiglu_fused",
           lib().decomoe_expert_swiglu_fused(_ptr(x_perm), _ptr(offsets), rows, K, d, m, _dt(x_perm),
                                             _ptr(w_gate_up), _ptr(w_down), _ptr(h), _ptr(y_perm), _ptr(ready),
                                             _ptr(status), _stream(stream)))


def decomoe_attention_workspace_bytes(n, C, Hq, Hkv, D=128):
    return int(lib().decomoe_attention_workspace_bytes(n, C, Hq, Hkv, D))


def decomoe_attention(q, k_cache, v_cache, out, ws, scale=0.0, status=None, stream=None):
    """Causal grouped-head attention of the last n positions over a
    (compacted) sequence: q [n, Hq, D], k_cache / v_cache [C, Hkv, D], out
    [n, Hq, D], bf16."""
    _need_cuda(q, k_cache, v_cache, out, ws, status)
    n, Hq, D = q.shape
    C, Hkv, _ = k_cache.shape
    _check("decomoe_attention",
           lib().decomoe_attention(_ptr(q), n, _ptr(k_cache), _ptr(v_cache), C, Hq, Hkv, D, float(scale), _ptr(out),
                                   _ptr(ws), 0 if ws is None else ws.numel() * ws.element_size(), _ptr(status),
                                   _stream(stream)))


def decomoe_gather_rows(x, perm_token, offsets, K, x_perm, stream=None):
    """The dispatch's row gather alone: x_perm[r] = x[perm_token[r]] for the
    offsets[K] rows on the device."""
    _need_cuda(x, perm_token, offsets, x_perm)
    d = x.shape[1]
    _check("decomoe_gather_rows",
           lib().decomoe_gather_rows(_ptr(x), _ptr(perm_token), _ptr(offsets), K, x_perm.shape[0], d, _dt(x),
                                     _ptr(x_perm), _stream(stream)))


def decomoe_expert_swiglu_fused_gather(x, perm_token, offsets, K, w_gate_up, w_down, x_perm, h, y_perm, ready,
                                       status=None, stream=None):
    """The one-launch expert FFN as the layer runs it from 8192 routed rows:
    it gathers x_perm[r] = x[perm_token[r]] itself (dispatch called without
    x_perm); ready: int32 counters, zero at the call."""
    _need_cuda(x, perm_token, offsets, w_gate_up, w_down, x_perm, h, y_perm, ready, status)
    T, d = x.shape
    rows = x_perm.shape[0]
    m = h.shape[1]
    _check("decomoe_expert_swiglu_fused_gather",
           lib().decomoe_expert_swiglu_fused_gather(_ptr(x), T, _ptr(perm_token), _ptr(offsets), rows, K, d, m,
                                                    _dt(x), _ptr(w_gate_up), _ptr(w_down), _ptr(x_perm), _ptr(h),
                                                    _ptr(y_perm), _ptr(ready), _ptr(status), _stream(stream)))


def decomoe_expert_gate_up(x_perm, offsets, K, w_gate_up, h, status=None, sched=None, stream=None):
    _need_cuda(x_perm, offsets, w_gate_up, h, status, sched)
    rows, d = x_perm.shape
    m = h.shape[1]
    _check("decomoe_expert_gate_up",
           lib().decomoe_expert_gate_up(_ptr(x_perm), _ptr(offsets), rows, K, d, m, _dt(x_perm), _ptr(w_gate_up),
                                        _ptr(h), _ptr(status), _ptr(sched), _stream(stream)))


def decomoe_expert_down(h, offsets, K, w_down, y_perm, status=None, sched=None, stream=None):
    _need_cuda(h, offsets, w_down, y_perm, status, sched)
    rows, m = h.shape
    d = y_perm.shape[1]
    _check("decomoe_expert_down",
           lib().decomoe_expert_down(_ptr(h), _ptr(offsets), rows, K, d, m, _dt(h), _ptr(w_down), _ptr(y_perm),
                                     _ptr(status), _ptr(sched), _stream(stream)))


def decomoe_expert_gate_up_gather(x, perm_token, offsets, K, w_gate_up, h, status=None, stream=None):
    _need_cuda(x, perm_token, offsets, w_gate_up, h, status)
    T, d = x.shape
    rows = perm_token.shape[0]
    m = h.shape[1]
    _check("decomoe_expert_gate_up_gather",
           lib().decomoe_expert_gate_up_gather(_ptr(x), T, _ptr(perm_token), _ptr(offsets), rows, K, d, m, _dt(x),
                                               _ptr(w_gate_up), _ptr(h), _ptr(status), None, _stream(stream)))


def decomoe_expert_swiglu_gather(x, perm_token, offsets, K, w_gate_up, w_down, h_ws, y_perm, status=None,
                                 stream=None):
    _need_cuda(x, perm_token, offsets, w_gate_up, w_down, h_ws, y_perm, status)
    T, d = x.shape
    rows = perm_token.shape[0]
    m = w_down.shape[2]
    _check("decomoe_expert_swiglu_gather",
           lib().decomoe_expert_swiglu_gather(_ptr(x), T, _ptr(perm_token), _ptr(offsets), rows, K, d, m, _dt(x),
                                              _ptr(w_gate_up), _ptr(w_down), _ptr(h_ws), _ptr(y_perm),
                                              _ptr(status), None, _stream(stream)))


def decomoe_expert_swiglu_ref(x_perm, offsets, K, w_gate_up, w_down, h_ws, y_perm, stream=None):
    _need_cuda(x_perm, offsets, w_gate_up, w_down, h_ws, y_perm)
    rows, d = x_perm.shape
    m = w_down.shape[2]
    _check("decomoe_expert_swiglu_ref",
           lib().decomoe_expert_swiglu_ref(_ptr(x_perm), _ptr(offsets), rows, K, d, m, _ptr(w_gate_up),
                                           _ptr(w_down), _ptr(h_ws), _ptr(y_perm), _stream(stream)))


def decomoe_combine(y_perm, inv_slot, topk_w, out, residual=None, stream=None):
    _need_cuda(y_perm, inv_slot, topk_w, out, residual)
    T, k = topk_w.shape
    d = out.shape[1]
    _check("decomoe_combine",
           lib().decomoe_combine(_ptr(y_perm), _ptr(inv_slot), _ptr(topk_w), T, k, d, _dt(out),
                                 _ptr(residual), _ptr(out), _stream(stream)))


def decomoe_combine_drop_visual_block(y_perm, inv_slot, topk_w, out, text_out, v0, nv, residual=None, stream=None):
    """Combine, and the output's text rows (outside [v0, v0 + nv)) also
    stored to text_out [T - nv, d] in the same launch."""
    _need_cuda(y_perm, inv_slot, topk_w, out, text_out, residual)
    T, k = topk_w.shape
    d = out.shape[1]
    _check("decomoe_combine_drop_visual_block",
           lib().decomoe_combine_drop_visual_block(_ptr(y_perm), _ptr(inv_slot), _ptr(topk_w), T, k, d, _dt(out),
                                                   _ptr(residual), _ptr(out), _ptr(text_out), v0, nv,
                                                   _stream(stream)))


def _drop_geometry(src, dst, nv):
    if src.dim() >= 3:
        nbatch, rows = src.shape[0], src.shape[1]
        row_bytes = src[0, 0].numel() * src.element_size()
        sstride = src.stride(0) * src.element_size()
        dstride = dst.stride(0) * dst.element_size()
    else:
        nbatch, rows = 1, src.shape[0]
        row_bytes = (src.numel() // max(rows, 1)) * src.element_size() if rows else src.element_size()
        sstride = rows * row_bytes
        dstride = (rows - nv) * row_bytes
    return nbatch, rows, row_bytes, sstride, dstride


def decomoe_drop_visual_block(src, dst, v0, nv, stream=None):
    """src: [rows, ...] or [nbatch, rows, ...] contiguous; dst the compacted shape."""
    _need_cuda(src, dst)
    nbatch, rows, row_bytes, sstride, dstride = _drop_geometry(src, dst, nv)
    _check("decomoe_drop_visual_block",
           lib().decomoe_drop_visual_block(_ptr(src), _ptr(dst), rows, row_bytes, v0, nv, nbatch, sstride,
                                           dstride, _stream(stream)))


def decomoe_drop_visual_block_if(exit_flag, src, dst, v0, nv, stream=None):
    """decomoe_drop_visual_block when the device int32 exit_flag holds 1 (the
    SAVB gate's decision); otherwise dst is left as it is."""
    _need_cuda(exit_flag, src, dst)
    nbatch, rows, row_bytes, sstride, dstride = _drop_geometry(src, dst, nv)
    _check("decomoe_drop_visual_block_if",
           lib().decomoe_drop_visual_block_if(_ptr(exit_flag), _ptr(src), _ptr(dst), rows, row_bytes, v0, nv, nbatch,
                                              sstride, dstride, _stream(stream)))


def decomoe_rmsnorm(x, y, eps=1e-6, stream=None):
    _need_cuda(x, y)
    T, d = x.shape
    _check("decomoe_rmsnorm", lib().decomoe_rmsnorm(_ptr(x), _ptr(y), T, d, float(eps), _dt(x), _stream(stream)))


def decomoe_moe_layer(x, w_r, bias, w_gate_up, w_down, k, out, ws, K_fixed=0, p=0.0, residual=None,
                      status=None, stream=None, text_out=None, v0=0, nv=0):
    """One RCEP MoE invocation. Returns (K_used, K_selected or None). With
    text_out, the exit layer: the output's text rows (outside [v0, v0 + nv))
    are also stored, compacted, to text_out."""
    _need_cuda(x, w_r, bias, w_gate_up, w_down, out, ws, residual, status, text_out)
    T, d = x.shape
    E = w_r.shape[0]
    m = w_down.shape[2]
    Ku, Ks = ctypes.c_int(0), ctypes.c_int(-1)
    if text_out is None:
        _check("decomoe_moe_layer",
               lib().decomoe_moe_layer(_ptr(x), _ptr(w_r), _ptr(bias), _ptr(w_gate_up), _ptr(w_down), T, d, E,
                                       k, m, _dt(x), int(K_fixed), float(p), _ptr(residual), _ptr(out),
                                       ctypes.byref(Ku), ctypes.byref(Ks), _ptr(ws),
                                       ws.numel() * ws.element_size(), _ptr(status), _stream(stream)))
    else:
        _check("decomoe_moe_layer_exit",
               lib().decomoe_moe_layer_exit(_ptr(x), _ptr(w_r), _ptr(bias), _ptr(w_gate_up), _ptr(w_down), T, d,
                                            E, k, m, _dt(x), int(K_fixed), float(p), _ptr(residual), _ptr(out),
                                            _ptr(text_out), int(v0), int(nv), ctypes.byref(Ku), ctypes.byref(Ks),
                                            _ptr(ws), ws.numel() * ws.element_size(), _ptr(status),
                                            _stream(stream)))
    return Ku.value, (Ks.value if Ks.value >= 0 else None)


def decomoe_read_status(status, stream=None) -> int:
    code = ctypes.c_int32(0)
    _check("decomoe_read_status", lib().decomoe_read_status(_ptr(status), ctypes.byref(code), _stream(stream)))
    return code.value


def decomoe_selftest_wait(status, limit_ns, stream=None):
    _check("decomoe_selftest_wait", lib().decomoe_selftest_wait(_ptr(status), int(limit_ns), _stream(stream)))


# ----------------------------------------------------------------- helpers

def fuse_gate_up(w_gate: torch.Tensor, w_up: torch.Tensor) -> torch.Tensor:
    """Interleaved gate/up weights [E, 2m, d] made on the device by the library."""
    E, m, d = w_gate.shape
    out = torch.empty((E, 2 * m, d), dtype=w_gate.dtype, device=w_gate.device)
    decomoe_weight_layout(w_gate, w_up, out)
    return out


def capture_graph(fn, warmup: int = 1) -> "torch.cuda.CUDAGraph":
    """Capture fn() (a sequence of the calls above with fixed sizes, e.g. one
    fixed-K MoE layer) into a CUDA graph; replay it with g.replay(). Calls
    that synchronise (decomoe_moe_layer with K_fixed == 0, decomoe_read_status)
    cannot be captured."""
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        for _ in range(warmup):
            fn()
    torch.cuda.current_stream().wait_stream(side)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        fn()
    return g


def workspace(nbytes: int, device) -> torch.Tensor:
    """A caller-owned device workspace of at least nbytes (256-byte aligned)."""
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)
