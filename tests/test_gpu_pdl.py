"""Programmatic dependent launch changes when kernels start, never what they
compute: the layer's output and its routing/dispatch intermediates are
bit-identical with it on (the default) and off (decomoe_set_pdl(0)), at
prefill and decode sizes, over several graph replays. A kernel that read its
predecessor's output before griddepcontrol.wait would show up here as a
mismatch.
"""
import pytest
import torch

import paper_2609_38823_gb300 as dm
import workloads as W

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda")


def _run():
    res = {}
    for T, K in ((2048, 64), (8, 64), (1, -1)):
        wl = W.with_(W.PREFILL, T=T)
        g = W.make_layer(wl, device="cuda", seed=5)
        wgu = dm.fuse_gate_up(g["w_gate"], g["w_up"])
        out = torch.empty_like(g["x"])
        ws = dm.workspace(dm.decomoe_moe_layer_workspace_bytes(T, wl.d, wl.E, wl.k, wl.m, 0), DEV)
        ws.zero_()  # padding between sub-buffers compares equal too
        st = torch.zeros(1, dtype=torch.int32, device=DEV)
        fn = lambda: dm.decomoe_moe_layer(g["x"], g["w_r"], g["bias"], wgu, g["w_down"], wl.k, out, ws, K_fixed=K,
                                          p=0.7, residual=g["x"], status=st)
        gr = dm.capture_graph(fn)
        for _ in range(5):
            gr.replay()
        torch.cuda.synchronize()
        assert dm.decomoe_read_status(st) == 0
        res[f"{T}_{K}_out"] = out.cpu().clone()
        res[f"{T}_{K}_ws"] = ws[: dm.decomoe_moe_layer_workspace_layout(T, wl.d, wl.E, wl.k, wl.m, 0)[8]].cpu().clone()
        del gr
    return res


def test_pdl_on_and_off_give_identical_bits():
    import __graft_entry__

    __graft_entry__.build()
    on = _run()
    dm.decomoe_set_pdl(False)
    try:
        off = _run()
    finally:
        dm.decomoe_set_pdl(True)
    assert on.keys() == off.keys()
    for key in on:
        a, b = on[key], off[key]
        if a.dtype == torch.bfloat16:
            a, b = a.view(torch.int16), b.view(torch.int16)
        assert torch.equal(a, b), key
