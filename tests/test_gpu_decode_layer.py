"""The decode-size layer as one launch (router, routing, dispatch, experts and
combine in a single persistent kernel, 1 <= T <= 32 tokens).

Its counters live in the layer workspace and must reset themselves: these
tests start from a workspace full of garbage or zeros (no signature: the
launch initialises the block), replay several CUDA graphs that share one
workspace with different inputs in a rotating order (also after the
workspace was zeroed between replays), and compare every output with a
fresh eager call. The combine done inside the kernel must
equal, bit for bit, decomoe_combine run on the kernel's own expert outputs;
the oracle comparison of the same layer sits in test_gpu_layer.py.
"""
import numpy as np
import pytest
import torch

import paper_2609_38823_gb300 as dm
import workloads as W
from oracle import decomoe_oracle as O
from tests.helpers import BF16_MAX_ABS, BF16_REL_L2, assert_close_out, f64

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__

    __graft_entry__.build()
    dm.lib()


@pytest.fixture(scope="module")
def layer():
    wl = W.PREFILL
    g = W.make_layer(wl, device="cuda", with_x=False, seed=3)
    g["w_gu"] = dm.fuse_gate_up(g["w_gate"], g["w_up"])
    return wl, g


def _ws(wl, T):
    return dm.workspace(dm.decomoe_moe_layer_workspace_bytes(T, wl.d, wl.E, wl.k, wl.m, dm.DECOMOE_BF16), DEV)


def _call(wl, g, x, out, ws, K, p=0.7, residual=None, status=None):
    return dm.decomoe_moe_layer(x, g["w_r"], g["bias"], g["w_gu"], g["w_down"], wl.k, out, ws, K_fixed=K, p=p,
                                residual=residual, status=status)


def _bits(t):
    return t.view(torch.int16)


class _Experts:
    """float64 host copies of the experts a test touches, made on first use."""

    def __init__(self, t):
        self.t, self.c = t, {}

    def __getitem__(self, e):
        if e not in self.c:
            self.c[e] = self.t[e].double().cpu().numpy()
        return self.c[e]


@pytest.mark.parametrize("T,K", [(1, 64), (2, 64), (5, 8), (16, 128), (12, -1), (3, -1), (32, 64), (1, -1)])
def test_garbage_workspace_first_call(layer, T, K):
    wl, g = layer
    x = W.make_x(W.DECODE, T=T, device="cuda", seed=T)
    ref = torch.empty_like(x)
    ws0 = _ws(wl, T)
    ws0.zero_()
    _call(wl, g, x, ref, ws0, K)
    ws = _ws(wl, T)
    ws.copy_(torch.randint(0, 256, ws.shape, dtype=torch.uint8, generator=torch.Generator().manual_seed(T)).to(DEV))
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    out = torch.empty_like(x)
    for _ in range(3):  # the first call clears the counters, the next ones find them reset
        out.fill_(7.0)
        _call(wl, g, x, out, ws, K, status=st)
        torch.cuda.synchronize()
        assert dm.decomoe_read_status(st) == 0
        assert torch.equal(_bits(out), _bits(ref))


@pytest.mark.parametrize("T,K", [(1, 64), (2, 64), (8, 64), (32, 40), (8, -1), (13, 64)])
def test_rotating_graph_replays_share_one_workspace(layer, T, K):
    """The counters must be back at zero after every launch, and the launch
    counter one number further, for the next replay (of the same or another
    graph) to be right; a zeroed workspace (no signature) between two replays
    is initialised again by the next one."""
    wl, g = layer
    xs = [W.make_x(W.DECODE, T=T, device="cuda", seed=10 + i) for i in range(3)]
    res = torch.zeros_like(xs[0])
    refs = []
    for x in xs:
        o = torch.empty_like(x)
        _call(wl, g, x, o, _ws(wl, T), K, residual=res)
        refs.append(o)
    ws = _ws(wl, T)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    outs = [torch.empty_like(x) for x in xs]
    graphs = [dm.capture_graph(lambda i=i: _call(wl, g, xs[i], outs[i], ws, K, residual=res, status=st))
              for i in range(3)]
    for n, i in enumerate((0, 1, 2, 0, 0, 1, 2, 2, 1, 0, 1, 2, 0)):
        if n in (5, 11):
            ws.zero_()
        outs[i].fill_(-3.0)
        graphs[i].replay()
        torch.cuda.synchronize()
        assert torch.equal(_bits(outs[i]), _bits(refs[i])), f"replay {n} of graph {i}"
    assert dm.decomoe_read_status(st) == 0


@pytest.mark.parametrize("T,K,resid", [(2, 64, False), (7, 64, True), (32, 96, True), (12, -1, False),
                                        (20, 64, True)])
def test_in_kernel_combine_equals_combine_call(layer, T, K, resid):
    wl, g = layer
    x = W.make_x(W.DECODE, T=T, device="cuda", seed=100 + T)
    r = W.make_x(W.DECODE, T=T, device="cuda", seed=200 + T, tensor_id=W.TID_RESID) if resid else None
    ws = _ws(wl, T)
    out = torch.empty_like(x)
    dm.decomoe_set_discard_scratch(False)
    try:
        _call(wl, g, x, out, ws, K, residual=r)
        torch.cuda.synchronize()
    finally:
        dm.decomoe_set_discard_scratch(True)
    offs = dm.decomoe_moe_layer_workspace_layout(T, wl.d, wl.E, wl.k, wl.m, dm.DECOMOE_BF16)
    k = wl.k
    w = ws[offs[2]:offs[2] + T * k * 4].view(torch.float32).view(T, k)
    inv = ws[offs[7]:offs[7] + T * k * 4].view(torch.int32)
    y = ws[offs[10]:offs[10] + T * k * wl.d * 2].view(torch.bfloat16).view(T * k, wl.d)
    out2 = torch.empty_like(x)
    dm.decomoe_combine(y, inv, w, out2, residual=r)
    torch.cuda.synchronize()
    assert torch.equal(_bits(out), _bits(out2))


@pytest.mark.parametrize("T,K,p", [(2, 8, 0.7), (4, 128, 0.0), (2, -1, 1.0), (32, 8, 0.0), (9, -1, 0.05),
                                   (25, 64, 0.7)])
def test_edge_prefixes_against_oracle(layer, T, K, p):
    """K = k (the prefix is exactly the top-k), the full span, p = 1 and a
    tiny p on the device, no mass pass (p = 0): routing, mass and output
    against the oracle on the layer's own fp32 logits."""
    wl, g = layer
    x = W.make_x(W.DECODE, T=T, device="cuda", seed=300 + T)
    ws = _ws(wl, T)
    out = torch.empty_like(x)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    _call(wl, g, x, out, ws, K, p=p, status=st)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(st) == 0
    offs = dm.decomoe_moe_layer_workspace_layout(T, wl.d, wl.E, wl.k, wl.m, dm.DECOMOE_BF16)
    E, k = wl.E, wl.k
    logits = f64(ws[offs[0]:offs[0] + T * E * 4].view(torch.float32).view(T, E))
    idx = ws[offs[1]:offs[1] + T * k * 4].view(torch.int32).view(T, k).cpu().numpy()
    wts = ws[offs[2]:offs[2] + T * k * 4].view(torch.float32).view(T, k).cpu().numpy()
    if K == -1:
        mass = ws[offs[3]:offs[3] + E * 8].view(torch.float64).cpu().numpy()
        s_ref = O.activated_mass(logits.astype(np.float32), k)
        assert np.allclose(mass, s_ref, rtol=4e-6, atol=1e-5)
        Kd = int(ws[offs[11]:offs[11] + 4].view(torch.int32).cpu())
        assert Kd == O.select_prefix(mass, p, k)
        Ku = Kd
    else:
        Ku = K
    ref_idx, ref_w = O.route_prefix(logits.astype(np.float32), Ku, k)
    keep = O.prefix_margin(logits.astype(np.float32), Ku, k) > 1e-6
    assert np.array_equal(idx[keep], ref_idx[keep])
    assert np.abs(wts[keep] - ref_w[keep]).max(initial=0.0) <= 1e-6
    wg, wu, wd = (_Experts(g[n]) for n in ("w_gate", "w_up", "w_down"))
    ref = np.stack([O.moe_token(f64(x[t]), logits[t].astype(np.float32), wg, wu, wd, Ku, k)[0] for t in range(T)])
    assert_close_out(f64(out)[keep], ref[keep], BF16_REL_L2, BF16_MAX_ABS, "decode layer output")


@pytest.mark.parametrize("T,K,p", [(1, 64, 0.7), (5, 64, 0.7), (8, -1, 0.7), (16, 64, 0.7), (3, 40, 0.0),
                                   (24, 64, 0.0)])
def test_tied_logits_take_the_lower_index(layer, T, K, p):
    """A router whose rows come in identical pairs gives every logit twice:
    the one-launch routing (a bitonic top-8 network for E <= 128, k <= 8)
    must order equal logits by index exactly as the routing kernel's arg-max
    rounds do, picks and weights bit for bit, on the layer's own logits."""
    wl, g = layer
    w_r = g["w_r"].clone()
    w_r[1::2] = w_r[0::2]
    bias = None
    if g["bias"] is not None:
        bias = g["bias"].clone()
        bias[1::2] = bias[0::2]
    x = W.make_x(W.DECODE, T=T, device="cuda", seed=400 + T)
    ws = _ws(wl, T)
    out = torch.empty_like(x)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    dm.decomoe_moe_layer(x, w_r, bias, g["w_gu"], g["w_down"], wl.k, out, ws, K_fixed=K, p=p, status=st)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(st) == 0
    offs = dm.decomoe_moe_layer_workspace_layout(T, wl.d, wl.E, wl.k, wl.m, dm.DECOMOE_BF16)
    E, k = wl.E, wl.k
    logits = ws[offs[0]:offs[0] + T * E * 4].view(torch.float32).view(T, E).clone()
    assert torch.equal(logits[:, 0::2].view(torch.int32), logits[:, 1::2].view(torch.int32))
    idx = ws[offs[1]:offs[1] + T * k * 4].view(torch.int32).view(T, k).clone()
    wts = ws[offs[2]:offs[2] + T * k * 4].view(torch.float32).view(T, k).clone()
    Ku = int(ws[offs[11]:offs[11] + 4].view(torch.int32).cpu()) if K == -1 else K
    ri = torch.empty(T, k, dtype=torch.int32, device=DEV)
    rw = torch.empty(T, k, dtype=torch.float32, device=DEV)
    dm.decomoe_route_prefix(logits, Ku, k, topk_idx=ri, topk_w=rw)
    torch.cuda.synchronize()
    assert torch.equal(idx, ri)
    assert torch.equal(wts.view(torch.int32), rw.view(torch.int32))
    oi, _ = O.route_prefix(logits.cpu().numpy(), Ku, k)
    assert np.array_equal(idx.cpu().numpy(), oi)


@pytest.mark.parametrize("E,k,T,K,p", [(256, 16, 1, 200, 0.7), (256, 16, 4, -1, 0.7), (256, 16, 13, 240, 0.7),
                                       (256, 16, 16, 64, 0.0), (64, 4, 8, 32, 0.7), (64, 4, 32, 48, 0.7)])
def test_other_pool_shapes_against_oracle(E, k, T, K, p):
    """Pools other than 128 experts with k = 8: 256 experts (eight key slots
    per lane in the routing rounds) with k = 16, where up to 16 tokens fill
    the 256 routed rows and 13 or more tokens take the per-CTA routing with
    its exchanged picks, and 64 experts with k = 4. Routing, mass and the
    device-selected prefix against the oracle on the layer's own logits;
    outputs within the bf16 tolerance."""
    wl = W.with_(W.PREFILL, E=E, k=k, d=256, m=128)
    g = W.make_layer(wl, device="cuda", with_x=False, seed=5)
    x = W.make_x(wl, T=T, device="cuda", seed=600 + T)
    ws = _ws(wl, T)
    out = torch.empty_like(x)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    dm.decomoe_moe_layer(x, g["w_r"], g["bias"], dm.fuse_gate_up(g["w_gate"], g["w_up"]), g["w_down"], k, out, ws,
                         K_fixed=K, p=p, status=st)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(st) == 0
    offs = dm.decomoe_moe_layer_workspace_layout(T, wl.d, E, k, wl.m, dm.DECOMOE_BF16)
    logits = f64(ws[offs[0]:offs[0] + T * E * 4].view(torch.float32).view(T, E))
    idx = ws[offs[1]:offs[1] + T * k * 4].view(torch.int32).view(T, k).cpu().numpy()
    wts = ws[offs[2]:offs[2] + T * k * 4].view(torch.float32).view(T, k).cpu().numpy()
    if K == -1:
        mass = ws[offs[3]:offs[3] + E * 8].view(torch.float64).cpu().numpy()
        assert np.allclose(mass, O.activated_mass(logits.astype(np.float32), k), rtol=4e-6, atol=1e-5)
        Ku = int(ws[offs[11]:offs[11] + 4].view(torch.int32).cpu())
        assert Ku == O.select_prefix(mass, p, k)
    else:
        Ku = K
    ref_idx, ref_w = O.route_prefix(logits.astype(np.float32), Ku, k)
    keep = O.prefix_margin(logits.astype(np.float32), Ku, k) > 1e-6
    assert np.array_equal(idx[keep], ref_idx[keep])
    assert np.abs(wts[keep] - ref_w[keep]).max(initial=0.0) <= 1e-6
    wg, wu, wd = (_Experts(g[n]) for n in ("w_gate", "w_up", "w_down"))
    ref = np.stack([O.moe_token(f64(x[t]), logits[t].astype(np.float32), wg, wu, wd, Ku, k)[0] for t in range(T)])
    assert_close_out(f64(out)[keep], ref[keep], BF16_REL_L2, BF16_MAX_ABS, f"decode layer E={E} k={k} T={T}")
