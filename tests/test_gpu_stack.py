"""The attention-free layer stack (RMSNorm -> prefix MoE + residual, visual
block removed from the hidden state and the KV caches at the exit layer) and
the T=16384 prefill layer, against the oracle.

Tokens are independent once every layer's prefix K_l is fixed (no attention),
so the oracle follows sampled tokens through the layers one by one
(stack_token). Tokens whose routing margin at some layer is too small for the
two sides' rounding are counted and left out of the output comparison.
"""
import numpy as np
import pytest
import torch

import paper_2609_38823_gb300 as dm
import workloads as W
from oracle import decomoe_oracle as O
from paper_2609_38823_gb300.stack import Stack, StackLayer
from tests.helpers import MASS_P_BAND, Experts, assert_close_out, bf16_round, check_layer_tokens, f64

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__

    __graft_entry__.build()
    dm.lib()


class ExpertView:
    def __init__(self, t):
        self.t = t

    def __getitem__(self, e):
        return self.t[e].double().cpu().numpy()


def _layers(wl, n, device, first=0):
    out_dev, out_ref = [], []
    for l in range(first, first + n):
        g = W.make_layer(wl, layer=l, device=device, with_x=False)
        w_gu = dm.fuse_gate_up(g["w_gate"].to(DEV), g["w_up"].to(DEV))
        out_dev.append(StackLayer(g["w_r"].to(DEV), g["bias"].to(DEV), w_gu, g["w_down"].to(DEV)))
        out_ref.append(dict(w_r=f64(g["w_r"]).astype(np.float32) if wl.dtype == "f32" else f64(g["w_r"]),
                            bias=g["bias"].cpu().numpy(), w_gate=ExpertView(g["w_gate"]),
                            w_up=ExpertView(g["w_up"]), w_down=ExpertView(g["w_down"])))
    return out_dev, out_ref


def _trajectories(h0, ref_layers, K_sched, k, rows, round_fn):
    outs, margins = [], []
    for t in rows:
        h, mg = O.stack_token(h0[t], ref_layers, K_sched, k, round_bf16=round_fn)
        outs.append(h)
        margins.append(min(mg))
    return np.stack(outs), np.array(margins)


def test_small_fp32_stack_with_exit():
    wl = W.with_(W.TINY, layers=6, exit_layer=3)
    L, R = _layers(wl, 6, "cpu")
    K_sched = [16, 16, 16, 10, 6, 12]
    h0 = W.make_x(wl)
    st = Stack(L, K_sched, wl.k, exit_layer=3, v0=wl.v0, nv=wl.nv, T=wl.T)
    kv = [torch.randn(6, wl.T, 64, generator=torch.Generator().manual_seed(s)).to(DEV) for s in (1, 2)]
    kv_out = [torch.empty(6, wl.T - wl.nv, 64, device=DEV) for _ in range(2)]
    out = st.forward(h0.to(DEV), kv, kv_out)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(st.status) == 0
    text = [t for t in range(wl.T) if not (wl.v0 <= t < wl.v0 + wl.nv)]
    assert out.shape == (len(text), wl.d)
    ref, margins = _trajectories(f64(h0), R, K_sched, wl.k, text, None)
    keep = margins > 1e-4
    assert keep.mean() > 0.8
    assert_close_out(f64(out)[keep], ref[keep], 1e-4, 1e-4, "fp32 stack output")
    for src, dst in zip(kv, kv_out):
        ref_kv = np.stack([O.drop_visual_block(src[l].cpu().numpy(), wl.v0, wl.nv) for l in range(6)])
        assert np.array_equal(dst.cpu().numpy(), ref_kv)


@pytest.fixture(scope="module")
def stack48():
    wl = W.STACK
    L, R = _layers(wl, wl.layers, "cuda")
    return wl, L, R


def test_stack48_teacher_forced_every_layer(stack48):
    """The 48-layer stack at its real size (1552 rows, exit at layer 20,
    K_l drawn from 32..96 after it): every layer is checked against the
    oracle from the GPU's own bf16 input to that layer (teacher forcing: bf16
    drift over 48 layers would otherwise flip near-tie routing), on 16
    sampled text tokens (4 system rows, 12 trailing text rows) followed
    through all 48 layers, plus the KV compaction bit-exact. The RMSNorm
    output is compared with the oracle's on the same layer input. The
    end-to-end relative L2 of the oracle's own trajectory is printed, not
    gated."""
    wl, L, R = stack48
    d, E, k, m = wl.d, wl.E, wl.k, wl.m
    K_sched = W.stack_K_schedule(wl)
    assert K_sched[:20] == [128] * 20 and all(32 <= v <= 96 for v in K_sched[20:])
    h0 = W.make_x(wl, device="cuda")
    kv = [W.make_kv(wl, device="cuda", seed=s) for s in (0, 1)]
    kv_out = [torch.empty(wl.layers, wl.T - wl.nv, wl.kv_width, dtype=torch.bfloat16, device=DEV) for _ in range(2)]
    r = np.random.default_rng(7)
    rows = sorted(r.choice(wl.v0, 4, replace=False).tolist() +
                  r.choice(np.arange(wl.v0 + wl.nv, wl.T), 12, replace=False).tolist())
    rows_after = [t if t < wl.v0 else t - wl.nv for t in rows]
    rec = {}

    def trace(l, cur, xn, out, ws):
        Tc = cur.shape[0]
        idx = torch.tensor(rows if Tc == wl.T else rows_after, device=DEV)
        o = dm.decomoe_moe_layer_workspace_layout(Tc, d, E, k, m, dm.DECOMOE_BF16)
        lg = ws[o[0]:o[0] + Tc * E * 4].view(torch.float32).view(Tc, E)
        ti = ws[o[1]:o[1] + Tc * k * 4].view(torch.int32).view(Tc, k)
        tw = ws[o[2]:o[2] + Tc * k * 4].view(torch.float32).view(Tc, k)
        rec[l] = tuple(t[idx].cpu() for t in (cur, xn, out, lg, ti, tw))

    st = Stack(L, K_sched, k, exit_layer=wl.exit_layer, v0=wl.v0, nv=wl.nv, T=wl.T)
    out = st.forward(h0, kv, kv_out, trace=trace)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(st.status) == 0
    assert out.shape == (wl.T - wl.nv, d) and torch.isfinite(out.float()).all()
    for src, dst in zip(kv, kv_out):
        for l in (0, 19, 20, 47):
            ref = O.drop_visual_block(src[l].view(torch.int16).cpu().numpy(), wl.v0, wl.nv)
            assert np.array_equal(dst[l].view(torch.int16).cpu().numpy(), ref)
    assert sorted(rec) == list(range(wl.layers))
    h_ref = f64(h0[torch.tensor(rows, device=DEV)])
    ties = 0
    for l in range(wl.layers):
        cur, xn, o, lg, ti, tw = rec[l]
        wg, wu, wd = Experts(R[l]["w_gate"].t), Experts(R[l]["w_up"].t), Experts(R[l]["w_down"].t)
        wr64, b64 = R[l]["w_r"], R[l]["bias"].astype(np.float64)
        # RMSNorm of the layer input (stored in bf16)
        assert_close_out(f64(xn), O.rmsnorm(f64(cur)), 5e-3, 2e-2, f"layer {l} rmsnorm")
        # the layer from the GPU's own normed input, residual = its input
        ties += check_layer_tokens(f64(xn), wr64, b64, wg, wu, wd, f64(lg), ti.numpy(), tw.numpy(), f64(o),
                                   K_sched[l], k, residual64=f64(cur), label=f"stack layer {l}")
        # the oracle's own trajectory (bf16 storage between layers), reported
        xr = bf16_round(O.rmsnorm(h_ref))
        h_ref = bf16_round(h_ref + O.moe_layer(xr, wr64, b64, wg, wu, wd, k=k, K=K_sched[l])["out"])
    got = f64(out[torch.tensor(rows_after, device=DEV)])
    rel = np.linalg.norm(got - h_ref) / np.linalg.norm(h_ref)
    print(f"[stack48] {ties} near-tie token-layers of {16 * wl.layers}; end-to-end rel-L2 of the oracle's own "
          f"trajectory vs the GPU output after 48 layers: {rel:.3e} (reported, not gated)")


@pytest.mark.parametrize("K,zipf", [(39, 1.2), (128, 0.8)])
def test_large_T16384_layer_sampled_and_compaction(K, zipf):
    wl = W.with_(W.LARGE, zipf_s=zipf)
    g = W.make_layer(wl, device="cuda")
    w_gu = dm.fuse_gate_up(g["w_gate"], g["w_up"])
    out = torch.empty_like(g["x"])
    ws = dm.workspace(dm.decomoe_moe_layer_workspace_bytes(wl.T, wl.d, wl.E, wl.k, wl.m, dm.DECOMOE_BF16), DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    dm.decomoe_moe_layer(g["x"], g["w_r"], g["bias"], w_gu, g["w_down"], wl.k, out, ws, K_fixed=K, p=0.7, status=st)
    text = torch.empty(wl.T - wl.nv, wl.d, dtype=torch.bfloat16, device=DEV)
    dm.decomoe_drop_visual_block(out, text, wl.v0, wl.nv)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(st) == 0
    # compaction of the layer output: bit-exact against the oracle
    ref_text = O.drop_visual_block(out.view(torch.int16).cpu().numpy(), wl.v0, wl.nv)
    assert np.array_equal(text.view(torch.int16).cpu().numpy(), ref_text)
    # sampled tokens through the layer
    r = np.random.default_rng(K)
    sample = np.sort(r.choice(wl.T, 24, replace=False))
    x64 = f64(g["x"][torch.from_numpy(sample).to(DEV)])
    wr64 = f64(g["w_r"])
    b64 = g["bias"].cpu().numpy().astype(np.float64)
    from tests.helpers import logit_error_bound
    bound = logit_error_bound(x64, wr64, b64)
    a = O.router_logits(x64, wr64, b64).astype(np.float64)
    keep = O.prefix_margin(a, K, wl.k) > 2 * bound.max()
    ref = O.moe_layer(x64, wr64, b64, ExpertView(g["w_gate"]), ExpertView(g["w_up"]), ExpertView(g["w_down"]),
                      k=wl.k, K=K)
    assert_close_out(f64(out[torch.from_numpy(sample).to(DEV)])[keep], ref["out"][keep], 5e-3, 2e-2,
                     "T=16384 layer output")


def _gate_dev(wl, candidates, fire_at, H=64, seed=0):
    from paper_2609_38823_gb300.stack import SavbGate

    prm = W.make_gate_params(wl.d, H, candidates, fire_at, seed=seed, device="cuda")
    return SavbGate(prm, theta=0.5), prm


def test_gate_driven_exit_equals_fixed_exit_and_gate_parity():
    """Algorithm 2 with the SAVB gate: candidates 1 and 3; the synthetic gate
    fires at 3, so the visual block leaves before layer 4. The output and the
    compacted KV equal the fixed-exit stack's bit for bit, and the gate's
    p_exit at each candidate matches the oracle gate on that layer's output."""
    wl = W.with_(W.TINY, layers=6)
    L, _ = _layers(wl, 6, "cpu")
    K_sched = [16, 16, 16, 16, 10, 6]
    h0 = W.make_x(wl).to(DEV)
    gate, prm = _gate_dev(wl, [1, 3], fire_at=3)
    kvs = [torch.randn(6, wl.T, 64, generator=torch.Generator().manual_seed(s)).to(DEV) for s in (1, 2)]
    outs = []
    for kind in ("gate", "fixed"):
        kv_out = [torch.empty(6, wl.T - wl.nv, 64, device=DEV) for _ in range(2)]
        if kind == "gate":
            st = Stack(L, K_sched, wl.k, exit_layer=None, v0=wl.v0, nv=wl.nv, T=wl.T, gate=gate)
        else:
            st = Stack(L, K_sched, wl.k, exit_layer=4, v0=wl.v0, nv=wl.nv, T=wl.T)
        out = st.forward(h0, kvs, kv_out).clone()
        torch.cuda.synchronize()
        assert dm.decomoe_read_status(st.status) == 0
        assert st.exit_taken == 4
        outs.append((out, [t.clone() for t in kv_out], st))
    assert torch.equal(outs[0][0], outs[1][0])
    for a, b in zip(outs[0][1], outs[1][1]):
        assert torch.equal(a, b)
    gst = outs[0][2]
    assert gst.exit_flag.cpu().tolist()[1] == 0 and gst.exit_flag.cpu().tolist()[3] == 1
    # teacher-forced gate parity: hidden after layers 0..l from a window stack
    for l in (1, 3):
        win = Stack(L[:l + 1], K_sched[:l + 1], wl.k, exit_layer=None, v0=wl.v0, nv=wl.nv, T=wl.T)
        hl = win.forward(h0)
        torch.cuda.synchronize()
        w1, b1, w2, b2 = (t.cpu().numpy() for t in prm[l])
        p_ref = O.gate_exit_prob(O.gate_logits(O.gate_feature(f64(hl), wl.v0, wl.nv), w1, b1, w2, b2))
        assert abs(float(gst.p_exit[l]) - p_ref) <= 2e-5


def test_mass_selected_prefix_after_exit_device_equals_host():
    """After the exit, each layer's prefix is selected from its activated mass
    (Eq. 12 with p); the device selection gives the same output bits as the
    host selection, and the first post-exit layer matches the oracle run with
    the oracle's own K."""
    wl = W.with_(W.TINY, layers=5)
    L, R = _layers(wl, 5, "cpu")
    K_sched = [16] * 5
    h0 = W.make_x(wl).to(DEV)
    res = []
    for host in (False, True):
        st = Stack(L, K_sched, wl.k, exit_layer=2, v0=wl.v0, nv=wl.nv, T=wl.T, p_after_exit=0.7,
                   select_on_host=host)
        res.append(st.forward(h0).clone())
        torch.cuda.synchronize()
        assert dm.decomoe_read_status(st.status) == 0
    assert torch.equal(res[0], res[1])
    # layer 2 (first text-only layer) from the GPU's own input, K by the oracle
    pre = Stack(L[:2], K_sched[:2], wl.k, exit_layer=None, v0=wl.v0, nv=wl.nv, T=wl.T)
    h2 = O.drop_visual_block(f64(pre.forward(h0)), wl.v0, wl.nv)
    # already text-only (nv = 0): the mass-selected branch from its first layer
    one = Stack(L[2:3], [16], wl.k, exit_layer=0, v0=0, nv=0, T=h2.shape[0], p_after_exit=0.7)
    got = one.forward(torch.from_numpy(h2).to(DEV, torch.float32))
    torch.cuda.synchronize()
    xn = O.rmsnorm(h2)
    a = O.router_logits(xn, R[2]["w_r"], R[2]["bias"]).astype(np.float64)
    s_ref = O.activated_mass(a, wl.k)
    cum = np.cumsum(s_ref) / s_ref.sum()
    if np.abs(cum - 0.7).min() < MASS_P_BAND:
        pytest.skip("mass ratio within rounding of p: K is reported, not compared")
    K = O.select_prefix(s_ref, 0.7, wl.k)
    keep = O.prefix_margin(a, K, wl.k) > 1e-4
    ref = O.moe_layer(xn, R[2]["w_r"], R[2]["bias"], R[2]["w_gate"], R[2]["w_up"], R[2]["w_down"], k=wl.k,
                      K=K)["out"] + h2
    assert_close_out(f64(got)[keep], ref[keep], 1e-4, 1e-4, "mass-selected layer")
