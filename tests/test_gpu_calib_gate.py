"""GPU parity of the offline RCEP calibration (Eqs. 8-9, Algorithm 1) and of
the SAVB exit gate (Eqs. 2-3) against the oracle.

Calibration: the per-case routed mass within the activated-mass tolerance;
the Mean-Mass order bit-exact against the oracle's order of the GPU's own case
masses (same fp64 sums); the permutation gather byte-exact; and the reordered
layer with every expert kept (K = E) bit-identical to the original layer.
Gate: p_exit within an fp32 bound of the oracle's fp64 value on the same
hidden state, and the same decision wherever p_exit is not within that bound
of the threshold.
"""
import numpy as np
import pytest
import torch

import paper_2609_38823_gb300 as dm
import workloads as W
from oracle import decomoe_oracle as O
from tests.helpers import MASS_REL, f64

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__

    __graft_entry__.build()
    torch.cuda.set_device(0)
    dm.lib()


def _shuffled_bias(E, s, seed):
    """Zipf-skewed router bias in a shuffled expert order: the calibration
    has an order to find."""
    b = -s * np.log(np.arange(E) + 1.0)
    sigma = np.random.default_rng(seed).permutation(E)
    return torch.tensor(b[sigma], dtype=torch.float32), sigma


# ----------------------------------------------------------------- calibration

@pytest.mark.parametrize("E,k,cases", [
    (16, 2, [(64, 8, 48), (30, 0, 0), (20, 3, 16)]),               # tiny, ragged text spans
    (128, 8, [(1552, 16, 1280), (600, 0, 500), (300, 100, 150)]),  # text around a visual block
    (256, 32, [(129, 0, 0), (77, 76, 0)]),
])
def test_case_mass_and_mean_mass_order(E, k, cases):
    bias, _ = _shuffled_bias(E, 1.1, seed=E)
    accum = torch.zeros(E, dtype=torch.float64, device=DEV)
    per_case = []
    ref_cases = []
    for ci, (T, v0, nv) in enumerate(cases):
        a = W.make_logits(T, E, std=0.9, bias=bias, seed=ci, wid=50 + E)
        ad = a.to(DEV)
        ws = dm.workspace(dm.decomoe_calib_workspace_bytes(T, E), DEV)
        one = torch.zeros(E, dtype=torch.float64, device=DEV)
        dm.decomoe_calib_case_mass(ad, k, v0, nv, one, ws)
        dm.decomoe_calib_case_mass(ad, k, v0, nv, accum, ws)
        torch.cuda.synchronize()
        M_gpu = one.cpu().numpy()
        M_ref = O.text_routed_mass(O.drop_visual_block(a.numpy(), v0, nv), k)
        assert (np.abs(M_gpu - M_ref) <= MASS_REL * M_ref + 1e-30).all()
        assert abs(M_gpu.sum() - 1.0) <= MASS_REL
        per_case.append(M_gpu)
        ref_cases.append(M_ref)
    # accum is the case sum in call order: the oracle's sum of the GPU's case masses
    acc = accum.cpu().numpy()
    assert np.array_equal(acc, _ordered_sum(per_case))
    pi = torch.empty(E, dtype=torch.int32, device=DEV)
    mean = torch.empty(E, dtype=torch.float64, device=DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    dm.decomoe_mean_mass_order(accum, len(cases), pi, mean, st)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(st) == 0
    pi_ref, mean_ref = O.mean_mass_order(np.stack(per_case))
    assert np.array_equal(mean.cpu().numpy(), mean_ref)
    assert np.array_equal(pi.cpu().numpy(), pi_ref)
    # against the oracle's own masses: same order wherever the means are apart
    pi_o, mean_o = O.mean_mass_order(np.stack(ref_cases))
    srt = mean_o[pi_o]
    gaps = np.abs(np.diff(srt)) > 4 * MASS_REL * np.maximum(srt[:-1], 1e-300)
    # positions whose neighbours on both sides are clearly separated must agree
    sep = np.ones(E, bool)
    sep[:-1] &= gaps
    sep[1:] &= gaps
    assert np.array_equal(pi.cpu().numpy()[sep], pi_o[sep])


def _ordered_sum(ms):
    acc = np.zeros_like(ms[0])
    for m in ms:
        acc = acc + m
    return acc


def test_mean_mass_order_ties_and_bad_input():
    accum = torch.tensor([0.2, 0.4, 0.2, 0.2, 0.0, 0.4], dtype=torch.float64, device=DEV)
    pi = torch.empty(6, dtype=torch.int32, device=DEV)
    dm.decomoe_mean_mass_order(accum, 2, pi)
    assert pi.cpu().tolist() == [1, 5, 0, 2, 3, 4]
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    accum[2] = float("nan")
    dm.decomoe_mean_mass_order(accum, 2, pi, None, st)
    assert dm.decomoe_read_status(st) == dm.DECOMOE_ERR_BAD_INPUT


@pytest.mark.parametrize("shape,dtype", [((128, 2048), torch.bfloat16), ((128,), torch.float32),
                                         ((16, 2 * 128, 256), torch.bfloat16), ((16, 256, 128), torch.bfloat16),
                                         ((5, 3), torch.int16)])
def test_permute_experts_bit_exact(shape, dtype):
    E = shape[0]
    src = (torch.randn(shape, generator=torch.Generator().manual_seed(E)) * 100).to(dtype).to(DEV)
    dst = torch.empty_like(src)
    pi = np.random.default_rng(E).permutation(E)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    dm.decomoe_permute_experts(src, dst, torch.from_numpy(pi.astype(np.int32)).to(DEV), st)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(st) == 0
    ref = src.cpu()[torch.from_numpy(pi)]
    assert torch.equal(dst.cpu().view(torch.uint8) if dtype != torch.float32 else dst.cpu(),
                       ref.view(torch.uint8) if dtype != torch.float32 else ref)


def test_permute_experts_flags_bad_index():
    src = torch.arange(8 * 4, dtype=torch.float32, device=DEV).view(8, 4)
    dst = torch.zeros_like(src)
    pi = torch.tensor([1, 0, 2, 3, 4, 5, 6, 9], dtype=torch.int32, device=DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    dm.decomoe_permute_experts(src, dst, pi, st)
    assert dm.decomoe_read_status(st) == dm.DECOMOE_ERR_BAD_INPUT
    assert torch.equal(dst[:7], src[[1, 0, 2, 3, 4, 5, 6]]) and (dst[7] == 0).all()


@pytest.mark.parametrize("wl_name", ["tiny", "prefill"])
def test_calibrate_reorder_end_to_end(wl_name):
    """Calibrate a layer whose experts are stored in a shuffled order, apply
    the order to all four tensors on the GPU, and check: the unsliced layer
    (K = E) is bit-identical before and after; the calibration mass is
    non-increasing in the new order; the order recovers the shuffle where the
    oracle's means are clearly apart."""
    base = W.TINY if wl_name == "tiny" else W.with_(W.PREFILL, T=512)
    E, k, d, m = base.E, base.k, base.d, base.m
    bias, sigma = _shuffled_bias(E, 1.1, seed=3)
    g = W.make_layer(base, device="cuda")
    g["bias"] = bias.to(DEV)
    dt = g["x"].dtype
    w_gu = dm.fuse_gate_up(g["w_gate"], g["w_up"])
    # calibration cases: fresh token sets through the router of this layer
    accum = torch.zeros(E, dtype=torch.float64, device=DEV)
    n_cases = 4
    ref_cases = []
    for c in range(n_cases):
        xc = W.make_x(W.with_(base, T=base.T // 2 + 16 * c), device="cuda", seed=100 + c)
        logits = torch.empty(xc.shape[0], E, dtype=torch.float32, device=DEV)
        dm.decomoe_router_logits(xc, g["w_r"], g["bias"], logits)
        ws = dm.workspace(dm.decomoe_calib_workspace_bytes(xc.shape[0], E), DEV)
        v0, nv = (xc.shape[0] // 4, xc.shape[0] // 2)
        dm.decomoe_calib_case_mass(logits, k, v0, nv, accum, ws)
        torch.cuda.synchronize()
        ref_cases.append(O.text_routed_mass(O.drop_visual_block(logits.cpu().numpy(), v0, nv), k))
    pi = torch.empty(E, dtype=torch.int32, device=DEV)
    mean = torch.empty(E, dtype=torch.float64, device=DEV)
    dm.decomoe_mean_mass_order(accum, n_cases, pi, mean)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    new = {}
    for name, t in (("w_r", g["w_r"]), ("bias", g["bias"]), ("w_gu", w_gu), ("w_down", g["w_down"])):
        new[name] = torch.empty_like(t)
        dm.decomoe_permute_experts(t, new[name], pi, st)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(st) == 0
    mn = mean.cpu().numpy()
    assert (np.diff(mn[pi.cpu().numpy()]) <= 0).all()
    # the order puts the experts the shuffled bias favours first (clear gaps only)
    pi_o, mean_o = O.mean_mass_order(np.stack(ref_cases))
    lead = min(8, E // 2)
    if mean_o[pi_o[lead - 1]] - mean_o[pi_o[lead]] > 1e-6:
        assert set(pi.cpu().numpy()[:lead].tolist()) == set(pi_o[:lead].tolist())
    # identity on the unsliced layer (K = E): same output bits
    T = g["x"].shape[0]
    outs = []
    for w_r, b, gu, wd in ((g["w_r"], g["bias"], w_gu, g["w_down"]),
                           (new["w_r"], new["bias"], new["w_gu"], new["w_down"])):
        out = torch.empty_like(g["x"])
        ws = dm.workspace(dm.decomoe_moe_layer_workspace_bytes(T, d, E, k, m, dm.DECOMOE_BF16 if dt ==
                                                               torch.bfloat16 else dm.DECOMOE_F32), DEV)
        dm.decomoe_moe_layer(g["x"], w_r, b, gu, wd, k, out, ws, K_fixed=E, p=0.0, status=st)
        outs.append(out)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(st) == 0
    assert torch.equal(outs[0].view(torch.uint8) if dt == torch.bfloat16 else outs[0],
                       outs[1].view(torch.uint8) if dt == torch.bfloat16 else outs[1])


# ----------------------------------------------------------------- SAVB gate

def _gate_params(d, H, seed, b2=(0.0, 0.0)):
    r = np.random.default_rng(seed)
    w1 = (r.standard_normal((H, 2 * d)) / np.sqrt(2 * d)).astype(np.float32)
    b1 = (r.standard_normal(H) * 0.1).astype(np.float32)
    w2 = (r.standard_normal((2, H)) / np.sqrt(H)).astype(np.float32)
    b2 = np.asarray(b2, np.float32)
    return w1, b1, w2, b2


GATE_CASES = [
    # T, v0, nv, d, H, dtype
    (64, 8, 48, 256, 64, "f32"),           # tiny workload's sequence
    (1552, 16, 1280, 2048, 512, "bf16"),   # stack workload: 272 text rows
    (16384, 0, 14336, 2048, 512, "bf16"),  # large prefill: 2048 text rows
    (300, 0, 0, 128, 100, "bf16"),         # no visual block, H not a multiple of 8
    (10, 2, 8, 64, 8, "f32"),              # two text rows: pooled half = first row
    (10, 0, 9, 64, 8, "bf16"),             # one text row: pooled half = 0
]


@pytest.mark.parametrize("T,v0,nv,d,H,dt", GATE_CASES)
def test_savb_gate_parity(T, v0, nv, d, H, dt):
    dtype = torch.bfloat16 if dt == "bf16" else torch.float32
    h = torch.randn(T, d, generator=torch.Generator().manual_seed(T + d)).to(dtype)
    w1, b1, w2, b2 = _gate_params(d, H, seed=T)
    dev = [torch.from_numpy(v).to(DEV) for v in (w1, b1, w2, b2)]
    hd = h.to(DEV)
    p = torch.empty(1, dtype=torch.float32, device=DEV)
    ex = torch.empty(1, dtype=torch.int32, device=DEV)
    ws = dm.workspace(dm.decomoe_savb_gate_workspace_bytes(d, H), DEV)
    ws.fill_(0x77)
    for theta in (0.3, 0.5, 0.7):
        dm.decomoe_savb_gate(hd, v0, nv, *dev, theta, p, ex, ws)
        torch.cuda.synchronize()
        x = O.gate_feature(f64(h), v0, nv)
        z = O.gate_logits(x, w1, b1, w2, b2)
        p_ref = O.gate_exit_prob(z)
        got = float(p.item())
        # fp32 feature sums and dot products over 2d and H terms: the logits
        # carry a relative error of a few 1e-6 of their magnitude sums
        tol = 2e-5
        assert abs(got - p_ref) <= tol, (got, p_ref)
        if abs(p_ref - theta) > tol:
            assert int(ex.item()) == int(O.gate_decision(p_ref, theta))


def test_savb_gate_fires_on_a_biased_head_and_graph_replays():
    T, v0, nv, d, H = 1552, 16, 1280, 2048, 512
    h = torch.randn(T, d, generator=torch.Generator().manual_seed(4)).to(torch.bfloat16).to(DEV)
    p = torch.empty(1, dtype=torch.float32, device=DEV)
    ex = torch.empty(1, dtype=torch.int32, device=DEV)
    ws = dm.workspace(dm.decomoe_savb_gate_workspace_bytes(d, H), DEV)
    for b2, want in (((4.0, -4.0), 0), ((-4.0, 4.0), 1)):
        prm = [torch.from_numpy(v).to(DEV) for v in _gate_params(d, H, seed=1, b2=b2)]
        g = dm.capture_graph(lambda prm=prm: dm.decomoe_savb_gate(h, v0, nv, *prm, 0.5, p, ex, ws))
        for _ in range(2):
            ex.fill_(-1)
            g.replay()
            torch.cuda.synchronize()
            assert int(ex.item()) == want
