"""Whole-layer parity (router -> mass -> prefix routing -> dispatch -> experts
-> combine through decomoe_moe_layer) on the workloads' shapes.

The router logits of the two sides differ by fp32 rounding. Each logit is
checked against a rigorous bound. A token whose oracle prefix margin is larger
than twice its own largest bound must get exactly the oracle's experts. For a
near-tie token several expert sets are correct: the GPU's set is checked to be
one that logits within the bounds rank first, and its weights and output are
compared with the oracle evaluated on that set. Every sampled token is thus
compared; the near-tie count is printed and bounded.
"""
import numpy as np
import pytest
import torch

import paper_2609_38823_gb300 as dm
import workloads as W
from oracle import decomoe_oracle as O
from tests.helpers import (BF16_MAX_ABS, BF16_REL_L2, F32_MAX_ABS, F32_REL_L2, MASS_P_BAND, MASS_REL, W_ABS,
                           Experts, check_layer_tokens, f64)

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__

    __graft_entry__.build()
    dm.lib()


class ExpertView:
    """Per-expert float64 view of a (device or host) weight tensor."""

    def __init__(self, t):
        self.t = t

    def __getitem__(self, e):
        return self.t[e].double().cpu().numpy()


def _run_layer(g, k, T, K_fixed=0, p=0.0, residual=None):
    d = g["x"].shape[1]
    E = g["w_r"].shape[0]
    m = g["w_down"].shape[2]
    dt = dm.DECOMOE_BF16 if g["x"].dtype == torch.bfloat16 else dm.DECOMOE_F32
    w_gu = g.get("w_gu")
    if w_gu is None:
        w_gu = dm.fuse_gate_up(g["w_gate"], g["w_up"])
        g["w_gu"] = w_gu
    out = torch.empty_like(g["x"])
    nbytes = dm.decomoe_moe_layer_workspace_bytes(T, d, E, k, m, dt)
    ws = dm.workspace(nbytes, DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    Ku, Ks = dm.decomoe_moe_layer(g["x"], g["w_r"], g["bias"], w_gu, g["w_down"], k, out, ws, K_fixed=K_fixed,
                                  p=p, residual=residual, status=status)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(status) == 0
    offs = dm.decomoe_moe_layer_workspace_layout(T, d, E, k, m, dt)
    logits = ws[offs[0]:offs[0] + T * E * 4].view(torch.float32).view(T, E)
    idx = ws[offs[1]:offs[1] + T * k * 4].view(torch.int32).view(T, k)
    w = ws[offs[2]:offs[2] + T * k * 4].view(torch.float32).view(T, k)
    mass = ws[offs[3]:offs[3] + E * 8].view(torch.float64)
    return out, Ku, Ks, logits.cpu(), idx.cpu().numpy(), w.cpu().numpy(), mass.cpu().numpy()


def _compare(g_cpu, out, logits, idx, w, K, k, sample, tol, residual=None):
    """The sampled tokens' routing and output against the oracle (rule in
    tests.helpers.check_layer_tokens). Returns the near-tie count."""
    return check_layer_tokens(f64(g_cpu["x"][sample]), f64(g_cpu["w_r"]), g_cpu["bias"].numpy().astype(np.float64),
                              Experts(g_cpu["w_gate"]), Experts(g_cpu["w_up"]), Experts(g_cpu["w_down"]),
                              f64(logits[sample]), idx[sample], w[sample], f64(out[sample]), K, k,
                              residual64=None if residual is None else f64(residual[sample]), tol=tol,
                              label="layer parity")


# ----------------------------------------------------------------- tiny fp32 layer (all tokens)

@pytest.mark.parametrize("K", [10, 16, 2])
def test_layer_tiny_fp32(K):
    wl = W.TINY
    g_cpu = W.make_layer(wl, device="cpu")
    g = {n: t.to(DEV) for n, t in g_cpu.items()}
    out, Ku, _, logits, idx, w, mass = _run_layer(g, wl.k, wl.T, K_fixed=K, p=0.7)
    assert Ku == K
    _compare(g_cpu, out, logits, idx, w, K, wl.k, np.arange(wl.T), (F32_REL_L2, F32_MAX_ABS))
    ref_mass = O.activated_mass(O.router_logits(f64(g_cpu["x"]), f64(g_cpu["w_r"]), g_cpu["bias"].numpy()), wl.k)
    assert (np.abs(mass - ref_mass) <= MASS_REL * ref_mass + 1e-5).all()


def test_layer_tiny_fp32_mass_selected_prefix():
    wl = W.TINY
    g_cpu = W.make_layer(wl, device="cpu")
    g = {n: t.to(DEV) for n, t in g_cpu.items()}
    a = O.router_logits(f64(g_cpu["x"]), f64(g_cpu["w_r"]), g_cpu["bias"].numpy())
    s = O.activated_mass(a, wl.k)
    for p in (0.3, 0.7, 0.95, 1.0):
        K_ref = O.select_prefix(s, p, wl.k)
        out, Ku, Ks, logits, idx, w, mass = _run_layer(g, wl.k, wl.T, K_fixed=0, p=p)
        cum = np.cumsum(s) / s.sum()
        if p < 1.0 and np.abs(cum - p).min() < MASS_P_BAND:
            continue  # selection within rounding of p: reported, not compared
        assert Ku == Ks == K_ref
        _compare(g_cpu, out, logits, idx, w, Ku, wl.k, np.arange(wl.T), (F32_REL_L2, F32_MAX_ABS))


def test_layer_tiny_fp32_residual():
    wl = W.TINY
    g_cpu = W.make_layer(wl, device="cpu")
    g = {n: t.to(DEV) for n, t in g_cpu.items()}
    res = W.make_x(wl, tensor_id=W.TID_RESID)
    out, _, _, logits, idx, w, _ = _run_layer(g, wl.k, wl.T, K_fixed=10, residual=res.to(DEV))
    _compare(g_cpu, out, logits, idx, w, 10, wl.k, np.arange(wl.T), (F32_REL_L2, F32_MAX_ABS), residual=res)


# ----------------------------------------------------------------- prefill T=2048 at full size

@pytest.fixture(scope="module")
def prefill_layer():
    wl = W.PREFILL
    g = W.make_layer(wl, device="cuda")
    g_cpu = {"x": g["x"].cpu(), "w_r": g["w_r"].cpu(), "bias": g["bias"].cpu(), "w_gate": g["w_gate"],
             "w_up": g["w_up"], "w_down": g["w_down"]}
    return wl, g, g_cpu


@pytest.mark.parametrize("K", [128, 96, 64, 40])
def test_layer_prefill_bf16_sampled(prefill_layer, K):
    wl, g, g_cpu = prefill_layer
    out, Ku, _, logits, idx, w, mass = _run_layer(g, wl.k, wl.T, K_fixed=K, p=0.7)
    r = np.random.default_rng(K)
    sample = np.unique(np.concatenate([[0, wl.T - 1], r.choice(wl.T, 62, replace=False)]))
    _compare(g_cpu, out, logits, idx, w, K, wl.k, sample, (BF16_REL_L2, BF16_MAX_ABS))
    # properties over every token
    assert ((idx >= 0) & (idx < K)).all()
    assert np.abs(w.sum(-1) - 1).max() <= W_ABS
    assert torch.isfinite(out.float()).all()
    assert abs(mass.sum() - wl.T) <= MASS_REL * wl.T


# ----------------------------------------------------------------- decode sizes (all tokens)

@pytest.mark.parametrize("T", [1, 8, 32, 128])
def test_layer_decode_bf16(prefill_layer, T):
    wl, g, g_cpu = prefill_layer
    x = W.make_x(W.DECODE, T=T, device="cuda")
    gd = dict(g, x=x)
    gc = dict(g_cpu, x=x.cpu())
    out, Ku, _, logits, idx, w, _ = _run_layer(gd, wl.k, T, K_fixed=64, p=0.7)
    _compare(gc, out, logits, idx, w, 64, wl.k, np.arange(T), (BF16_REL_L2, BF16_MAX_ABS))


# ----------------------------------------------------------------- prefix selected on the device

def test_select_prefix_device_matches_host_c():
    r = np.random.default_rng(11)
    for trial in range(60):
        E = int(r.choice([8, 16, 128, 256]))
        k = int(r.integers(1, min(E, 32) + 1))
        s = (1.0 / (np.arange(E) + 1.0) ** r.uniform(0.0, 2.0)) * r.uniform(0.0, 2.0, E) * r.uniform(1, 3000)
        if trial % 7 == 0:
            s[r.integers(0, E, size=E // 2)] = 0.0
        if trial % 11 == 0:
            s[:] = 0.0
        md = torch.from_numpy(s).to(DEV)
        Kd = torch.zeros(1, dtype=torch.int32, device=DEV)
        for p in (0.05, 0.3, 0.7, 0.9, 1.0):
            dm.decomoe_select_prefix_device(md, k, p, Kd)
            torch.cuda.synchronize()
            assert int(Kd) == dm.decomoe_select_prefix(s, k, p) == O.select_prefix(s, p, k)


@pytest.mark.parametrize("which", ["tiny", "prefill"])
def test_layer_device_selected_prefix_equals_host_selected(which, prefill_layer):
    if which == "tiny":
        wl = W.TINY
        g_cpu = W.make_layer(wl, device="cpu")
        g = {n: t.to(DEV) for n, t in g_cpu.items()}
    else:
        wl, g, g_cpu = prefill_layer
    p = 0.9 if which == "prefill" else 0.7
    out_h, Ku, Ks, logits, idx, w, mass = _run_layer(g, wl.k, wl.T, K_fixed=0, p=p)
    out_d, Kud, Ksd, logits_d, idx_d, w_d, mass_d = _run_layer(g, wl.k, wl.T, K_fixed=-1, p=p)
    assert Kud == -1 and Ksd is None
    assert torch.equal(out_h, out_d)
    assert np.array_equal(idx, idx_d) and np.array_equal(w, w_d)
    assert np.array_equal(mass, mass_d)


def test_layer_device_selected_prefix_in_cuda_graph(prefill_layer):
    wl, g, _ = prefill_layer
    T, d, E, k, m = wl.T, wl.d, wl.E, wl.k, wl.m
    w_gu = g.get("w_gu")
    if w_gu is None:
        w_gu = dm.fuse_gate_up(g["w_gate"], g["w_up"])
        g["w_gu"] = w_gu
    ws = dm.workspace(dm.decomoe_moe_layer_workspace_bytes(T, d, E, k, m, dm.DECOMOE_BF16), DEV)
    out_e = torch.empty_like(g["x"])
    dm.decomoe_moe_layer(g["x"], g["w_r"], g["bias"], w_gu, g["w_down"], k, out_e, ws, K_fixed=-1, p=0.8)
    torch.cuda.synchronize()
    out_g = torch.zeros_like(g["x"])
    graph = dm.capture_graph(lambda: dm.decomoe_moe_layer(g["x"], g["w_r"], g["bias"], w_gu, g["w_down"], k, out_g,
                                                          ws, K_fixed=-1, p=0.8))
    out_g.zero_()
    graph.replay()
    torch.cuda.synchronize()
    assert torch.equal(out_e, out_g)
    offs = dm.decomoe_moe_layer_workspace_layout(T, d, E, k, m, dm.DECOMOE_BF16)
    Kdev = int(ws[offs[11]:offs[11] + 4].view(torch.int32))
    mass = ws[offs[3]:offs[3] + E * 8].view(torch.float64).cpu().numpy()
    assert Kdev == dm.decomoe_select_prefix(mass, k, 0.8)


@pytest.mark.parametrize("T,K_fixed,p", [(1, 64, 0.7), (2, 64, 0.7), (6, 64, 0.7), (7, 64, 0.7), (8, 64, 0.7),
                                         (32, 40, 0.0), (100, 128, 0.7),
                                         (256, 96, 0.7), (1, -1, 0.7), (8, -1, 0.5), (129, -1, 0.9), (256, -1, 1.0),
                                         (1100, 40, 0.7), (2048, 64, 0.7), (2048, -1, 0.7)])
def test_layer_intermediates_equal_separate_calls(T, K_fixed, p):
    """The layer's routing, mass, prefix and dispatch intermediates and its
    expert outputs h and y (left in its workspace) equal, bit for bit, the
    separate C-ABI calls on the same router logits, for fixed and
    device-selected prefixes, at decode sizes (one expert launch from 16 rows)
    and prefill sizes (from 8192 routed rows the expert launch gathers x_perm
    itself: the gathered rows are compared too)."""
    wl = W.with_(W.PREFILL, T=T)
    E, k, d, m = wl.E, wl.k, wl.d, wl.m
    g = W.make_layer(wl, device="cuda", seed=T)
    w_gu = dm.fuse_gate_up(g["w_gate"], g["w_up"])
    out = torch.empty_like(g["x"])
    ws = dm.workspace(dm.decomoe_moe_layer_workspace_bytes(T, d, E, k, m, dm.DECOMOE_BF16), DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    # by default the combine drops the y rows from L2 after reading them: the
    # output must not depend on it; the run that keeps them is inspected below
    dm.decomoe_moe_layer(g["x"], g["w_r"], g["bias"], w_gu, g["w_down"], k, out, ws, K_fixed=K_fixed, p=p,
                         status=st)
    torch.cuda.synchronize()
    out_discard = out.clone()
    dm.decomoe_set_discard_scratch(False)
    try:
        dm.decomoe_moe_layer(g["x"], g["w_r"], g["bias"], w_gu, g["w_down"], k, out, ws, K_fixed=K_fixed, p=p,
                             status=st)
        torch.cuda.synchronize()
    finally:
        dm.decomoe_set_discard_scratch(True)
    assert dm.decomoe_read_status(st) == 0
    assert torch.equal(out.view(torch.int16), out_discard.view(torch.int16))
    offs = dm.decomoe_moe_layer_workspace_layout(T, d, E, k, m, dm.DECOMOE_BF16)
    view = lambda i, n, dt: ws[offs[i]:offs[i] + n * torch.tensor([], dtype=dt).element_size()].view(dt)
    logits = view(0, T * E, torch.float32).view(T, E).clone()
    Kd = E if K_fixed == -1 else K_fixed
    got = dict(idx=view(1, T * k, torch.int32).cpu(), w=view(2, T * k, torch.float32).cpu(),
               counts=view(4, Kd, torch.int32).cpu(), offsets=view(5, Kd + 1, torch.int32).cpu(),
               perm=view(6, T * k, torch.int32).cpu(), inv=view(7, T * k, torch.int32).cpu(),
               xp=view(8, T * k * d, torch.bfloat16).view(T * k, d).clone())
    mass_l = view(3, E, torch.float64).cpu()
    # separate calls on the same logits
    mass = torch.empty(E, dtype=torch.float64, device=DEV)
    rws = dm.workspace(dm.decomoe_route_workspace_bytes(T, E), DEV)
    idx = torch.empty(T, k, dtype=torch.int32, device=DEV)
    w = torch.empty(T, k, dtype=torch.float32, device=DEV)
    if K_fixed == -1:
        Kdev = torch.empty(1, dtype=torch.int32, device=DEV)
        dm.decomoe_route_prefix(logits, E, k, None, None, mass, rws)
        dm.decomoe_select_prefix_device(mass, k, p, Kdev)
        dm.decomoe_route_prefix_dk(logits, Kdev, k, idx, w)
        assert int(Kdev) == int(view(11, 1, torch.int32).cpu())
    else:
        dm.decomoe_route_prefix(logits, K_fixed, k, idx, w, mass if p > 0 else None, rws)
    counts = torch.empty(Kd, dtype=torch.int32, device=DEV)
    offsets = torch.empty(Kd + 1, dtype=torch.int32, device=DEV)
    perm = torch.empty(T * k, dtype=torch.int32, device=DEV)
    inv = torch.empty(T * k, dtype=torch.int32, device=DEV)
    xp = torch.empty(T * k, d, dtype=torch.bfloat16, device=DEV)
    dws = dm.workspace(dm.decomoe_dispatch_workspace_bytes(T, k, Kd), DEV)
    dm.decomoe_dispatch(idx, Kd, g["x"], counts, offsets, perm, inv, xp, dws)
    torch.cuda.synchronize()
    assert torch.equal(got["idx"], idx.view(-1).cpu())
    assert torch.equal(got["w"].view(torch.int32), w.view(-1).cpu().view(torch.int32))
    for n, t in (("counts", counts), ("offsets", offsets), ("perm", perm), ("inv", inv)):
        assert torch.equal(got[n], t.cpu()), n
    assert torch.equal(got["xp"].view(torch.int16), xp.view(torch.int16))
    if K_fixed == -1 or p > 0:
        assert torch.equal(mass_l.view(torch.int64), mass.cpu().view(torch.int64))
    # the layer's expert launch (both GEMMs in one launch where it fuses them)
    # writes the same h and y as the two separate expert calls
    h_l = view(9, T * k * m, torch.bfloat16).view(T * k, m)
    y_l = view(10, T * k * d, torch.bfloat16).view(T * k, d)
    h2 = torch.empty(T * k, m, dtype=torch.bfloat16, device=DEV)
    y2 = torch.empty(T * k, d, dtype=torch.bfloat16, device=DEV)
    dm.decomoe_expert_gate_up(xp, offsets, Kd, w_gu, h2, st)
    dm.decomoe_expert_down(h2, offsets, Kd, g["w_down"], y2, st)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(st) == 0
    assert torch.equal(h_l.view(torch.int16), h2.view(torch.int16))
    assert torch.equal(y_l.view(torch.int16), y2.view(torch.int16))


@pytest.mark.parametrize("T,K_fixed,v0,nv", [(2048, 64, 0, 1792), (300, -1, 16, 200), (8, 64, 7, 1), (64, 40, 0, 64)])
def test_layer_exit_equals_layer_then_removal(prefill_layer, T, K_fixed, v0, nv):
    """decomoe_moe_layer_exit writes the same layer output as
    decomoe_moe_layer and the same compacted text rows as a
    decomoe_drop_visual_block of that output, bit for bit."""
    wl, g, _ = prefill_layer
    x = g["x"][:T].contiguous()
    w_gu = dm.fuse_gate_up(g["w_gate"], g["w_up"])
    d, E, k, m = wl.d, wl.E, wl.k, wl.m
    ws1 = dm.workspace(dm.decomoe_moe_layer_workspace_bytes(T, d, E, k, m, dm.DECOMOE_BF16), DEV)
    ws2 = dm.workspace(dm.decomoe_moe_layer_workspace_bytes(T, d, E, k, m, dm.DECOMOE_BF16), DEV)
    out1, out2 = torch.empty_like(x), torch.empty_like(x)
    text1 = torch.full((T - nv, d), 5.0, dtype=x.dtype, device=DEV)
    text2 = torch.full((T - nv, d), -5.0, dtype=x.dtype, device=DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    dm.decomoe_moe_layer(x, g["w_r"], g["bias"], w_gu, g["w_down"], k, out1, ws1, K_fixed=K_fixed, p=0.7,
                         status=st, text_out=text1, v0=v0, nv=nv)
    dm.decomoe_moe_layer(x, g["w_r"], g["bias"], w_gu, g["w_down"], k, out2, ws2, K_fixed=K_fixed, p=0.7,
                         status=st)
    if T - nv > 0:
        dm.decomoe_drop_visual_block(out2, text2, v0, nv)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(st) == 0
    assert torch.equal(out1.view(torch.int16), out2.view(torch.int16))
    assert torch.equal(text1.view(torch.int16), text2.view(torch.int16))
