"""GPU parity of every C-ABI call against the CPU oracle, on seeded inputs.

Index, count and byte outputs must match bit for bit; floating outputs must
meet the stated tolerances. Sizes span several tiles with ragged tails; the
full workload sizes appear where the oracle can follow them (whole arrays for
routing, dispatch and compaction; sampled tokens for the expert FFN).
"""
import numpy as np
import pytest
import torch

import paper_2609_38823_gb300 as dm
import workloads as W
from oracle import decomoe_oracle as O
from tests.helpers import (BF16_MAX_ABS, BF16_REL_L2, F32_MAX_ABS, F32_REL_L2, MARGIN_SAME_LOGITS, MASS_P_BAND,
                           MASS_REL, W_ABS,
                           assert_close_out, bf16_round, f64, logit_error_bound)

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__

    __graft_entry__.build()
    torch.cuda.set_device(0)
    dm.lib()


def _zipf_bias(E, s=1.1):
    return torch.tensor(-s * np.log(np.arange(E) + 1.0), dtype=torch.float32)


# ----------------------------------------------------------------- bounded waits

def test_bounded_wait_times_out_and_context_survives():
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    dm.decomoe_selftest_wait(status, 2_000_000)
    assert dm.decomoe_read_status(status) == dm.DECOMOE_ERR_TIMEOUT
    assert dm.decomoe_read_status(status) == 0  # read clears it
    x = torch.ones(1 << 20, device=DEV)
    assert float((x * 2).sum()) == 2.0 * (1 << 20)


# ----------------------------------------------------------------- routing

ROUTE_CASES = [
    (1, 16, 10, 2), (63, 16, 2, 2), (64, 16, 16, 2), (65, 128, 64, 8), (2048, 128, 128, 8),
    (2048, 128, 96, 8), (2048, 128, 40, 8), (2048, 128, 8, 8), (777, 256, 200, 32), (300, 128, 9, 8),
    (16384, 128, 39, 8), (128, 128, 64, 8), (5, 33, 33, 1),
]


def _route_gpu(a, K, k, E=None, mass=False):
    T = a.shape[0]
    E = a.shape[1] if E is None else E
    ad = a.to(DEV)
    idx = torch.empty((T, k), dtype=torch.int32, device=DEV)
    w = torch.empty((T, k), dtype=torch.float32, device=DEV)
    ms = torch.empty(E, dtype=torch.float64, device=DEV) if mass else None
    ws = dm.workspace(dm.decomoe_route_workspace_bytes(T, E), DEV) if mass else None
    dm.decomoe_route_prefix(ad, K, k, idx, w, ms, ws, E=E)
    torch.cuda.synchronize()
    return idx.cpu().numpy(), w.cpu().numpy().astype(np.float64), (ms.cpu().numpy() if mass else None)


@pytest.mark.parametrize("T,E,K,k", ROUTE_CASES)
def test_route_prefix_parity(T, E, K, k):
    a = W.make_logits(T, E, std=0.9, bias=_zipf_bias(E), seed=0, wid=10 + E)
    idx, w, _ = _route_gpu(a, K, k)
    an = a.numpy()
    ri, rw = O.route_prefix(an, K, k)
    keep = O.prefix_margin(an, K, k) >= MARGIN_SAME_LOGITS
    assert keep.mean() > 0.95, f"too many near-ties: {(~keep).sum()}"
    assert np.array_equal(idx[keep], ri[keep]), "routing indices differ"
    assert np.abs(w[keep] - rw[keep]).max() <= W_ABS
    # properties on every token, including the excluded ones
    assert ((idx >= 0) & (idx < K)).all()
    assert np.abs(w.sum(-1) - 1.0).max() <= W_ABS
    picked = np.take_along_axis(an[:, :K], idx.astype(np.int64), axis=1)
    assert (np.diff(picked, axis=1) <= 0).all()
    for t in range(T):
        assert len(set(idx[t].tolist())) == k


def test_route_exact_ties_take_lower_index():
    a = torch.round(W.make_logits(512, 64, std=1.0, seed=3) * 2) / 2  # many exact ties
    for K, k in ((64, 8), (20, 4), (8, 8)):
        idx, w, _ = _route_gpu(a, K, k)
        ri, rw = O.route_prefix(a.numpy(), K, k)
        assert np.array_equal(idx, ri)
        assert np.abs(w - rw).max() <= W_ABS


def test_route_full_pool_topk_not_intersected():
    a = torch.tensor([[0.1, 0.4, 0.2, 0.3, -1.0, -2.0, 5.0, 6.0]], dtype=torch.float32)
    idx, w, _ = _route_gpu(a, 4, 2)
    assert idx[0].tolist() == [1, 3]


@pytest.mark.parametrize("T,K", [(1, 128), (64, 128), (100, 40), (2048, 64), (16384, 128), (777, 8)])
def test_activated_mass_parity_and_reproducible(T, K):
    # the mass is Eq. 11 over the full pool whatever prefix K the same launch routes
    E, k = 128, 8
    a = W.make_logits(T, E, std=0.9, bias=_zipf_bias(E), seed=1, wid=20)
    idx, w, m1 = _route_gpu(a, K, k, mass=True)
    _, _, m2 = _route_gpu(a, K, k, mass=True)
    ri, rw = O.route_prefix(a.numpy(), K, k)
    keep = O.prefix_margin(a.numpy(), K, k) >= MARGIN_SAME_LOGITS
    assert np.array_equal(idx[keep], ri[keep]) and np.abs(w[keep] - rw[keep]).max() <= W_ABS
    assert np.array_equal(m1.view(np.uint64), m2.view(np.uint64)), "mass not bit-reproducible"
    ref = O.activated_mass(a.numpy(), k)
    # fp32 per-token weights (expf, one division, sums of <= 8 terms per
    # block): a few fp32 ulps relative to each expert's mass
    assert (np.abs(m1 - ref) <= MASS_REL * ref + 1e-30).all()
    assert abs(m1.sum() - T) <= MASS_REL * T
    cum = np.cumsum(ref) / ref.sum()
    for p in (0.3, 0.5, 0.7, 0.9, 1.0):
        if p < 1.0 and np.abs(cum - p).min() < MASS_P_BAND:
            continue  # ratio within rounding of p: K is reported, not compared
        assert dm.decomoe_select_prefix(m1, k, p) == O.select_prefix(ref, p, k)


# ----------------------------------------------------------------- dispatch

def _idx_pattern(T, k, K, pattern, seed):
    r = np.random.default_rng(seed)
    if pattern == "route":
        E = max(K, 16)
        a = W.make_logits(T, E, std=0.9, bias=_zipf_bias(E), seed=seed, wid=30)
        return O.route_prefix(a.numpy(), K, k)[0]
    if pattern == "one_expert":
        return np.full((T, k), K - 1, np.int64)
    if pattern == "uniform":
        return r.integers(0, K, size=(T, k))
    if pattern == "sizes":  # k = 1, expert e routed SIZES[e] tokens, in random token order
        assert k == 1 and K == len(SIZES) and T == sum(SIZES)
        return r.permutation(np.repeat(np.arange(K), SIZES))[:, None].astype(np.int64)
    raise ValueError(pattern)


# expert row counts around the swapped-tile boundaries: 16-row MMA widths, the
# 32-token epilogue chunks, the 128-row threshold and empty experts
SIZES = [1, 15, 16, 17, 31, 32, 33, 63, 64, 65, 96, 127, 128, 129, 200, 0, 5]


DISPATCH_CASES = [
    (1, 8, 64, 2048, "bf16", "route"), (7, 2, 10, 256, "f32", "route"), (2048, 8, 128, 2048, "bf16", "route"),
    (2048, 8, 40, 2048, "bf16", "route"), (16384, 8, 39, 2048, "bf16", "route"), (100, 4, 8, 256, "bf16", "one_expert"),
    (1000, 3, 256, 64, "bf16", "uniform"), (129, 8, 16, 2048, "bf16", "uniform"), (1552, 8, 128, 2048, "bf16", "route"),
    (272, 8, 37, 2048, "bf16", "route"),
    # row sizes around the bulk-copy gather's ring limits: 6 KiB (32 buffers),
    # 8 KiB (16 buffers), 16 KiB (warp-per-row kernel)
    (300, 4, 16, 3072, "bf16", "route"), (300, 4, 16, 4096, "bf16", "uniform"), (64, 2, 8, 4096, "f32", "uniform"),
]


@pytest.mark.parametrize("T,k,K,d,dt,pattern", DISPATCH_CASES)
def test_dispatch_parity(T, k, K, d, dt, pattern):
    idx = _idx_pattern(T, k, K, pattern, seed=T + K)
    dtype = torch.bfloat16 if dt == "bf16" else torch.float32
    x = torch.randn(T, d, generator=torch.Generator().manual_seed(T), dtype=torch.float32).to(dtype).to(DEV)
    idx_d = torch.from_numpy(idx.astype(np.int32)).to(DEV)
    counts = torch.empty(K, dtype=torch.int32, device=DEV)
    offsets = torch.empty(K + 1, dtype=torch.int32, device=DEV)
    perm = torch.empty(T * k, dtype=torch.int32, device=DEV)
    inv = torch.empty(T * k, dtype=torch.int32, device=DEV)
    xp = torch.empty((T * k, d), dtype=dtype, device=DEV)
    ws = dm.workspace(dm.decomoe_dispatch_workspace_bytes(T, k, K), DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    dm.decomoe_dispatch(idx_d, K, x, counts, offsets, perm, inv, xp, ws, status)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(status) == 0
    c, o, p, i = O.dispatch(idx, K)
    assert np.array_equal(counts.cpu().numpy(), c)
    assert np.array_equal(offsets.cpu().numpy(), o)
    assert np.array_equal(perm.cpu().numpy(), p)
    assert np.array_equal(inv.cpu().numpy(), i)
    assert torch.equal(xp, x[perm.long()])
    # the row gather alone, after the index passes: the same rows
    xp2 = torch.zeros_like(xp)
    dm.decomoe_gather_rows(x, perm, offsets, K, xp2)
    torch.cuda.synchronize()
    assert torch.equal(xp2, xp)


def test_dispatch_flags_bad_expert_id():
    T, k, K = 50, 2, 8
    idx = np.random.default_rng(0).integers(0, K, size=(T, k))
    idx[3, 1] = K + 5
    idx_d = torch.from_numpy(idx.astype(np.int32)).to(DEV)
    counts = torch.empty(K, dtype=torch.int32, device=DEV)
    offsets = torch.empty(K + 1, dtype=torch.int32, device=DEV)
    perm = torch.empty(T * k, dtype=torch.int32, device=DEV)
    inv = torch.empty(T * k, dtype=torch.int32, device=DEV)
    ws = dm.workspace(dm.decomoe_dispatch_workspace_bytes(T, k, K), DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    dm.decomoe_dispatch(idx_d, K, None, counts, offsets, perm, inv, None, ws, status)
    assert dm.decomoe_read_status(status) == dm.DECOMOE_ERR_BAD_INPUT
    assert int(offsets[-1]) == T * k - 1 and int(inv[7]) == -1


# ----------------------------------------------------------------- expert FFN

def _expert_case(T, k, K, d, m, pattern, seed, dtype=torch.bfloat16):
    E = K
    wl = W.Workload("t", 40 + seed, T=T, d=d, E=E, k=k, m=m, dtype="bf16" if dtype == torch.bfloat16 else "f32",
                    x_std=1.0, wr_std=0.02, w_std=0.02, bias_kind="zipf", zipf_s=1.1, K_list=(K,), v0=0, nv=0)
    L = W.make_layer(wl, seed=seed, device="cpu")
    idx = _idx_pattern(T, k, K, pattern, seed)
    counts, offsets, perm, inv = O.dispatch(idx, K)
    x_perm = L["x"][torch.from_numpy(perm)]
    L["perm"] = perm
    return L, x_perm, offsets


EXPERT_CASES = [
    # T, k, K, d, m, pattern
    (150, 2, 10, 256, 128, "route"),      # several experts, ragged M tiles
    (64, 2, 16, 256, 128, "route"),
    (300, 1, 3, 256, 256, "one_expert"),  # one expert, 3 M tiles (300 rows)
    (512, 8, 64, 2048, 768, "route"),     # full layer width, 4096 rows
    (1100, 8, 64, 2048, 768, "route"),    # 8800 rows: the layer's launch gathers its own rows
    (129, 8, 16, 2048, 768, "uniform"),
    (1, 8, 64, 2048, 768, "route"),       # decode T=1 (8 rows)
    (8, 8, 64, 2048, 768, "route"),       # decode T=8 (64 rows)
    (9, 8, 64, 2048, 768, "route"),       # 72 rows: smallest tensor-core case
    (40, 2, 4, 2048, 768, "one_expert"),  # decode path, 40 rows on one expert (> 8 per chunk)
    (sum(SIZES), 1, len(SIZES), 2048, 768, "sizes"),  # swapped (<= 128 rows) and tokens-as-M experts
    (sum(SIZES), 1, len(SIZES), 256, 128, "sizes"),   # one N-tile per GEMM
]


@pytest.mark.parametrize("T,k,K,d,m,pattern", EXPERT_CASES)
def test_expert_swiglu_bf16_parity(T, k, K, d, m, pattern):
    L, x_perm, offsets = _expert_case(T, k, K, d, m, pattern, seed=T % 7)
    R = T * k
    g = {n: L[n].to(DEV) for n in ("w_gate", "w_up", "w_down")}
    w_gu = dm.fuse_gate_up(g["w_gate"], g["w_up"])
    xp = x_perm.to(DEV)
    off = torch.from_numpy(offsets.astype(np.int32)).to(DEV)
    h = torch.empty((R, m), dtype=torch.bfloat16, device=DEV)
    y = torch.empty((R, d), dtype=torch.bfloat16, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    dm.decomoe_expert_swiglu(xp, off, K, w_gu, g["w_down"], h, y, status)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(status) == 0
    ref = O.expert_swiglu(f64(x_perm), offsets, f64(L["w_gate"]), f64(L["w_up"]), f64(L["w_down"]))
    assert_close_out(f64(y), ref, BF16_REL_L2, BF16_MAX_ABS, "expert_swiglu vs oracle")
    # the CUDA-core reference computes the same bf16 arithmetic: much tighter agreement
    h2 = torch.empty_like(h)
    y2 = torch.empty_like(y)
    dm.decomoe_expert_swiglu_ref(xp, off, K, w_gu, g["w_down"], h2, y2)
    torch.cuda.synchronize()
    assert_close_out(f64(y), f64(y2), 2e-3, 1e-2, "tensor-core vs CUDA-core reference")
    # dynamic tile scheduling hands the same tiles out in another order: same bits
    sched = torch.zeros(1, dtype=torch.int32, device=DEV)
    h4 = torch.empty_like(h)
    y4 = torch.empty_like(y)
    dm.decomoe_expert_swiglu(xp, off, K, w_gu, g["w_down"], h4, y4, status, sched)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(status) == 0
    assert torch.equal(y4, y) and torch.equal(h4, h)
    # gather form: rows read from the token-ordered x through perm_token give
    # the same shared-memory tiles, so the same bits
    h3 = torch.empty_like(h)
    y3 = torch.empty_like(y)
    perm_d = torch.from_numpy(L["perm"].astype(np.int32)).to(DEV)
    dm.decomoe_expert_swiglu_gather(L["x"].to(DEV), perm_d, off, K, w_gu, g["w_down"], h3, y3, status)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(status) == 0
    assert torch.equal(y3, y) and torch.equal(h3, h)
    # both GEMMs in one launch where the library fuses them: same tiles and
    # k order, so the same bits; counters zero at the call
    ready = torch.zeros(dm.decomoe_expert_swiglu_ready_ints(R, K), dtype=torch.int32, device=DEV)
    h5 = torch.empty_like(h)
    y5 = torch.empty_like(y)
    dm.decomoe_expert_swiglu_fused(xp, off, K, w_gu, g["w_down"], h5, y5, ready, status)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(status) == 0
    assert torch.equal(y5, y) and torch.equal(h5, h)
    # the one launch that also gathers the dispatched rows (as the layer runs
    # it from 8192 routed rows): same tiles, same bits, and the gathered rows
    # are x[perm_token]
    if 8 * K < R <= 32768 and (2 * m) % 256 == 0:
        ready.zero_()
        xg = torch.zeros_like(xp)
        h6 = torch.empty_like(h)
        y6 = torch.empty_like(y)
        dm.decomoe_expert_swiglu_fused_gather(L["x"].to(DEV), perm_d, off, K, w_gu, g["w_down"], xg, h6, y6, ready,
                                              status)
        torch.cuda.synchronize()
        assert dm.decomoe_read_status(status) == 0
        assert torch.equal(y6, y) and torch.equal(h6, h)
        assert torch.equal(xg.view(torch.int16), xp.view(torch.int16))
    else:
        with pytest.raises(dm.DecomoeError) as e:
            dm.decomoe_expert_swiglu_fused_gather(L["x"].to(DEV), perm_d, off, K, w_gu, g["w_down"],
                                                  torch.empty_like(xp), torch.empty_like(h), torch.empty_like(y),
                                                  ready, status)
        assert e.value.code == dm.DECOMOE_ERR_INVALID_ARG


def test_expert_swiglu_f32_parity():
    T, k, K, d, m = 64, 2, 10, 256, 128
    L, x_perm, offsets = _expert_case(T, k, K, d, m, "route", seed=1, dtype=torch.float32)
    g = {n: L[n].to(DEV) for n in ("w_gate", "w_up", "w_down")}
    w_gu = dm.fuse_gate_up(g["w_gate"], g["w_up"])
    off = torch.from_numpy(offsets.astype(np.int32)).to(DEV)
    h = torch.empty((T * k, m), dtype=torch.float32, device=DEV)
    y = torch.empty((T * k, d), dtype=torch.float32, device=DEV)
    dm.decomoe_expert_swiglu(x_perm.to(DEV), off, K, w_gu, g["w_down"], h, y)
    torch.cuda.synchronize()
    ref = O.expert_swiglu(f64(x_perm), offsets, f64(L["w_gate"]), f64(L["w_up"]), f64(L["w_down"]))
    assert_close_out(f64(y), ref, F32_REL_L2, F32_MAX_ABS, "fp32 expert_swiglu")
    y3 = torch.empty_like(y)
    perm_d = torch.from_numpy(L["perm"].astype(np.int32)).to(DEV)
    dm.decomoe_expert_swiglu_gather(L["x"].to(DEV), perm_d, off, K, w_gu, g["w_down"], torch.empty_like(h), y3)
    torch.cuda.synchronize()
    assert torch.equal(y3, y)


def test_weight_layout_interleave():
    E, m, d = 3, 256, 64
    wg = torch.randn(E, m, d).to(torch.bfloat16).to(DEV)
    wu = torch.randn(E, m, d).to(torch.bfloat16).to(DEV)
    out = dm.fuse_gate_up(wg, wu)
    G = dm.GU_BLOCK
    for e in range(E):
        for b in range(m // G):
            assert torch.equal(out[e, 2 * G * b:2 * G * b + G], wg[e, G * b:G * (b + 1)])
            assert torch.equal(out[e, 2 * G * b + G:2 * G * (b + 1)], wu[e, G * b:G * (b + 1)])


# ----------------------------------------------------------------- combine

@pytest.mark.parametrize("T,k,d,dt,resid", [(1, 8, 2048, "bf16", False), (2048, 8, 2048, "bf16", True),
                                             (64, 2, 256, "f32", True), (333, 3, 128, "bf16", False),
                                             (50, 1, 64, "f32", False)])
def test_combine_parity(T, k, d, dt, resid):
    dtype = torch.bfloat16 if dt == "bf16" else torch.float32
    g = torch.Generator().manual_seed(T * 7 + k)
    y = torch.randn(T * k, d, generator=g).to(dtype)
    inv = torch.randperm(T * k, generator=g).to(torch.int32)
    w = torch.softmax(torch.randn(T, k, generator=g), -1).float()
    res = torch.randn(T, d, generator=g).to(dtype) if resid else None
    out = torch.empty(T, d, dtype=dtype, device=DEV)
    dm.decomoe_combine(y.to(DEV), inv.to(DEV), w.to(DEV), out, None if res is None else res.to(DEV))
    torch.cuda.synchronize()
    ref = O.combine(f64(y), inv.numpy(), f64(w), None if res is None else f64(res))
    if dtype == torch.float32:
        assert_close_out(f64(out), ref, 1e-6, 1e-6, "combine f32")
    else:
        # fp32 accumulation of k+1 terms (<= 2e-6 of the summed magnitudes),
        # then one rounding to bf16 (<= 2^-9 relative, taken as 2^-8)
        got = f64(out)
        mag = O.combine(np.abs(f64(y)), inv.numpy(), np.abs(f64(w)), None if res is None else np.abs(f64(res)))
        assert (np.abs(got - ref) <= np.abs(ref) * 2.0 ** -8 + 2e-6 * mag).all()
        assert_close_out(got, ref, BF16_REL_L2, BF16_MAX_ABS, "combine bf16")


@pytest.mark.parametrize("T,k,d,dt,resid,v0,nv", [(2048, 8, 2048, "bf16", True, 0, 1792),
                                                   (333, 3, 128, "bf16", False, 100, 200),
                                                   (64, 2, 256, "f32", True, 10, 0),
                                                   (50, 1, 64, "f32", False, 0, 50),
                                                   (40, 8, 2048, "bf16", False, 39, 1)])
def test_combine_drop_visual_block_equals_two_calls(T, k, d, dt, resid, v0, nv):
    """The fused combine + visual-block removal writes the same out and the
    same compacted text rows as decomoe_combine followed by
    decomoe_drop_visual_block, bit for bit (a block at the start, in the
    middle, empty, the whole sequence, the last row)."""
    dtype = torch.bfloat16 if dt == "bf16" else torch.float32
    g = torch.Generator().manual_seed(T * 5 + k)
    y = torch.randn(T * k, d, generator=g).to(dtype).to(DEV)
    inv = torch.randperm(T * k, generator=g).to(torch.int32).to(DEV)
    w = torch.softmax(torch.randn(T, k, generator=g), -1).float().to(DEV)
    res = torch.randn(T, d, generator=g).to(dtype).to(DEV) if resid else None
    out1, out2 = (torch.empty(T, d, dtype=dtype, device=DEV) for _ in range(2))
    text1 = torch.full((T - nv, d), 7, dtype=dtype, device=DEV)
    text2 = torch.full((T - nv, d), -7, dtype=dtype, device=DEV)
    dm.decomoe_combine_drop_visual_block(y, inv, w, out1, text1, v0, nv, res)
    dm.decomoe_combine(y, inv, w, out2, res)
    dm.decomoe_drop_visual_block(out2, text2, v0, nv)
    torch.cuda.synchronize()
    iv = torch.int16 if dtype == torch.bfloat16 else torch.int32
    assert torch.equal(out1.view(iv), out2.view(iv))
    assert torch.equal(text1.view(iv), text2.view(iv))


def test_combine_drop_visual_block_rejects_bad_block():
    T, k, d = 16, 2, 64
    y = torch.zeros(T * k, d, device=DEV)
    inv = torch.arange(T * k, dtype=torch.int32, device=DEV)
    w = torch.full((T, k), 0.5, device=DEV)
    out = torch.empty(T, d, device=DEV)
    with pytest.raises(dm.DecomoeError) as e:
        dm.decomoe_combine_drop_visual_block(y, inv, w, out, torch.empty(4, d, device=DEV), 10, 12)
    assert e.value.code == dm.DECOMOE_ERR_INVALID_ARG


# ----------------------------------------------------------------- visual-block removal

@pytest.mark.parametrize("shape,v0,nv,dt", [
    ((64, 256), 8, 48, torch.float32),            # tiny hidden, rows 8..55
    ((2048, 2048), 0, 1792, torch.bfloat16),      # prefill hidden -> 256 text rows
    ((16384, 2048), 0, 14336, torch.bfloat16),    # large hidden -> 2048 text rows
    ((48, 1552, 512), 16, 1280, torch.bfloat16),  # KV of the 48-layer stack -> 272 rows
    ((10, 7, 3), 2, 3, torch.bfloat16),           # 6-byte rows: byte path
    ((100, 64), 0, 0, torch.bfloat16),            # nv = 0: plain copy
    ((100, 64), 60, 40, torch.bfloat16),          # block at the end
    ((100, 64), 0, 100, torch.bfloat16),          # everything removed
    ((2, 9, 5, 16), 1, 3, torch.float32),         # [batch, rows, ...] with extra dims
])
def test_drop_visual_block_bit_exact(shape, v0, nv, dt):
    src = torch.randn(*shape, generator=torch.Generator().manual_seed(5)).to(dt)
    if len(shape) == 2:
        out_shape = (shape[0] - nv, shape[1])
        ref = O.drop_visual_block(src.view(torch.int16 if dt == torch.bfloat16 else torch.int32).numpy(), v0, nv)
    else:
        out_shape = (shape[0], shape[1] - nv) + tuple(shape[2:])
        iv = src.view(torch.int16 if dt == torch.bfloat16 else torch.int32).numpy()
        ref = np.stack([O.drop_visual_block(iv[b], v0, nv) for b in range(shape[0])])
    dst = torch.full(out_shape, 7.0, dtype=dt, device=DEV)
    if dst.numel() > 0:
        dm.decomoe_drop_visual_block(src.to(DEV).contiguous(), dst, v0, nv)
    torch.cuda.synchronize()
    got = dst.cpu().view(torch.int16 if dt == torch.bfloat16 else torch.int32).numpy()
    assert got.shape == ref.shape and np.array_equal(got, ref)


@pytest.mark.parametrize("shape,v0,nv,dt", [((300, 2048), 16, 256, torch.bfloat16),
                                             ((4, 100, 512), 10, 80, torch.bfloat16),
                                             ((9, 7, 6), 2, 3, torch.float32)])  # byte path (24-byte rows)
def test_drop_visual_block_if_follows_the_device_flag(shape, v0, nv, dt):
    """The gate-triggered removal compacts exactly when the device flag holds
    1 (then bit-identical to the unconditional call) and leaves dst untouched
    for 0 or any other value."""
    src = torch.randn(*shape, generator=torch.Generator().manual_seed(9)).to(dt).to(DEV)
    out_shape = (shape[0] - nv,) + tuple(shape[1:]) if len(shape) == 2 else \
        (shape[0], shape[1] - nv) + tuple(shape[2:])
    iv = torch.int16 if dt == torch.bfloat16 else torch.int32
    ref = torch.empty(out_shape, dtype=dt, device=DEV)
    dm.decomoe_drop_visual_block(src, ref, v0, nv)
    for fv in (0, 1, 2, -1):
        flag = torch.tensor([fv], dtype=torch.int32, device=DEV)
        dst = torch.full(out_shape, 3.0, dtype=dt, device=DEV)
        dm.decomoe_drop_visual_block_if(flag, src, dst, v0, nv)
        torch.cuda.synchronize()
        if fv == 1:
            assert torch.equal(dst.view(iv), ref.view(iv))
        else:
            assert (dst == 3.0).all()


# ----------------------------------------------------------------- router logits

@pytest.mark.parametrize("T,d,E", [(2048, 2048, 128), (1, 2048, 128), (300, 2048, 256), (1552, 2048, 128),
                                   (129, 256, 128), (7, 2048, 128), (192, 2048, 128), (193, 2048, 256),
                                   (33, 4096, 64), (5, 2056, 16), (8, 2048, 128), (9, 2048, 256), (96, 2048, 128),
                                   (3, 4096, 64), (6, 2048, 256)])
def test_router_logits_bf16_tensor_cores(T, d, E):
    g = torch.Generator().manual_seed(T + E)
    x = torch.randn(T, d, generator=g).to(torch.bfloat16)
    w = (torch.randn(E, d, generator=g) * 0.02).to(torch.bfloat16)
    b = _zipf_bias(E)
    lg = torch.empty(T, E, dtype=torch.float32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    dm.decomoe_router_logits(x.to(DEV), w.to(DEV), b.to(DEV), lg, status)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(status) == 0
    x64, w64, b64 = f64(x), f64(w), b.numpy().astype(np.float64)
    ref = O.router_logits(x64, w64, b64).astype(np.float64)
    err = np.abs(f64(lg) - ref)
    assert (err <= logit_error_bound(x64, w64, b64)).all(), f"max err {err.max():.3e}"


def test_router_logits_f32():
    T, d, E = 64, 256, 16
    g = torch.Generator().manual_seed(1)
    x = torch.randn(T, d, generator=g)
    w = torch.randn(E, d, generator=g) * 0.05
    b = torch.linspace(1, -1, E)
    lg = torch.empty(T, E, device=DEV)
    dm.decomoe_router_logits(x.to(DEV), w.to(DEV), b.to(DEV), lg)
    torch.cuda.synchronize()
    x64, w64, b64 = f64(x), f64(w), f64(b)
    err = np.abs(f64(lg) - O.router_logits(x64, w64, b64))
    assert (err <= logit_error_bound(x64, w64, b64)).all()


def test_rmsnorm():
    for dt, tol in ((torch.float32, 1e-6), (torch.bfloat16, 2.0 ** -8)):
        x = torch.randn(100, 2048, generator=torch.Generator().manual_seed(2)).to(dt)
        y = torch.empty(100, 2048, dtype=dt, device=DEV)
        dm.decomoe_rmsnorm(x.to(DEV), y, 1e-6)
        torch.cuda.synchronize()
        ref = O.rmsnorm(f64(x), 1e-6)
        assert np.abs(f64(y) - ref).max() <= tol * np.abs(ref).max() * 2


# ----------------------------------------------------------------- routing + dispatch in one call

@pytest.mark.parametrize("T,E,K,k,p", [(1, 128, 64, 8, 0.0), (7, 16, 10, 2, 0.0), (100, 128, 40, 8, 0.0),
                                       (256, 128, 128, 8, 0.0), (257, 128, 64, 8, 0.0), (2048, 128, 64, 8, 0.0),
                                       (33, 256, 200, 32, 0.0), (1, 128, -1, 8, 0.7), (64, 128, -1, 8, 0.9),
                                       (256, 128, -1, 8, 0.5), (300, 128, -1, 8, 0.7), (2048, 128, -1, 8, 1.0)])
def test_route_dispatch_equals_separate_calls_and_oracle(T, E, K, k, p):
    """decomoe_route_dispatch (one block at decode sizes, the separate kernels
    above them) equals the separate C-ABI calls bit for bit, and its dispatch
    is the oracle's stable sort of its own picks."""
    a = W.make_logits(T, E, std=0.9, bias=_zipf_bias(E), seed=3, wid=60 + E)
    ad = a.to(DEV)
    d = 256
    x = torch.randn(T, d, generator=torch.Generator().manual_seed(T)).to(torch.bfloat16).to(DEV)
    Kd = E if K == -1 else K
    idx = torch.full((T, k), -9, dtype=torch.int32, device=DEV)
    w = torch.empty(T, k, dtype=torch.float32, device=DEV)
    mass = torch.empty(E, dtype=torch.float64, device=DEV)
    Kdev = torch.zeros(1, dtype=torch.int32, device=DEV)
    counts = torch.empty(Kd, dtype=torch.int32, device=DEV)
    offsets = torch.empty(Kd + 1, dtype=torch.int32, device=DEV)
    perm = torch.empty(T * k, dtype=torch.int32, device=DEV)
    inv = torch.empty(T * k, dtype=torch.int32, device=DEV)
    xp = torch.empty(T * k, d, dtype=torch.bfloat16, device=DEV)
    ws = dm.workspace(dm.decomoe_route_dispatch_workspace_bytes(T, k, E), DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    dm.decomoe_route_dispatch(ad, K, k, idx, w, x, counts, offsets, perm, inv, xp, ws, p=p, mass_out=mass,
                              K_dev=Kdev if K == -1 else None, status=st)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(st) == 0
    # separate calls
    rws = dm.workspace(dm.decomoe_route_workspace_bytes(T, E), DEV)
    idx2 = torch.empty(T, k, dtype=torch.int32, device=DEV)
    w2 = torch.empty(T, k, dtype=torch.float32, device=DEV)
    mass2 = torch.empty(E, dtype=torch.float64, device=DEV)
    if K == -1:
        Kdev2 = torch.empty(1, dtype=torch.int32, device=DEV)
        dm.decomoe_route_prefix(ad, E, k, None, None, mass2, rws)
        dm.decomoe_select_prefix_device(mass2, k, p, Kdev2)
        dm.decomoe_route_prefix_dk(ad, Kdev2, k, idx2, w2)
        Ksel = int(Kdev2)
        assert int(Kdev) == Ksel
    else:
        dm.decomoe_route_prefix(ad, K, k, idx2, w2, mass2, rws)
        Ksel = K
    c2 = torch.empty(Kd, dtype=torch.int32, device=DEV)
    o2 = torch.empty(Kd + 1, dtype=torch.int32, device=DEV)
    p2 = torch.empty(T * k, dtype=torch.int32, device=DEV)
    i2 = torch.empty(T * k, dtype=torch.int32, device=DEV)
    xp2 = torch.empty(T * k, d, dtype=torch.bfloat16, device=DEV)
    dm.decomoe_dispatch(idx2, Kd, x, c2, o2, p2, i2, xp2, dm.workspace(dm.decomoe_dispatch_workspace_bytes(T, k, Kd),
                                                                      DEV))
    torch.cuda.synchronize()
    for got, ref in ((idx, idx2), (counts, c2), (offsets, o2), (perm, p2), (inv, i2)):
        assert torch.equal(got, ref)
    assert torch.equal(w.view(torch.int32), w2.view(torch.int32))
    assert torch.equal(mass.view(torch.int64), mass2.view(torch.int64))
    assert torch.equal(xp.view(torch.int16), xp2.view(torch.int16))
    # oracle: dispatch of the picks, routing away from near-ties, mass
    c, o, pp, ii = O.dispatch(idx.cpu().numpy().astype(np.int64), Kd)
    assert np.array_equal(counts.cpu().numpy(), c) and np.array_equal(perm.cpu().numpy(), pp)
    ri, rw = O.route_prefix(a.numpy(), Ksel, k)
    keep = O.prefix_margin(a.numpy(), Ksel, k) >= MARGIN_SAME_LOGITS
    assert np.array_equal(idx.cpu().numpy()[keep], ri[keep])
    ref_m = O.activated_mass(a.numpy(), k)
    assert (np.abs(mass.cpu().numpy() - ref_m) <= MASS_REL * ref_m + 1e-30).all()


@pytest.mark.parametrize("T,E", [(97, 128), (193, 128), (300, 256), (576, 128), (577, 128), (2048, 128),
                                 (2432, 256), (2433, 128), (16384, 128), (100, 128)])
def test_router_logits_k_split(T, E):
    """The workspace router (k slices on the tensor cores, partial sums added
    in slice order, the bias last) stays within the fp32 summation bound at
    every slice count it picks (16, 4, or none)."""
    d = 2048
    g = torch.Generator().manual_seed(T + 7 * E)
    x = torch.randn(T, d, generator=g).to(torch.bfloat16)
    w = (torch.randn(E, d, generator=g) * 0.02).to(torch.bfloat16)
    b = _zipf_bias(E)
    lg = torch.full((T, E), float("nan"), dtype=torch.float32, device=DEV)
    ws = dm.workspace(dm.decomoe_router_logits_ws_bytes(T, d, E), DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    dm.decomoe_router_logits_ws(x.to(DEV), w.to(DEV), b.to(DEV), lg, ws, status)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(status) == 0
    x64, w64, b64 = f64(x), f64(w), b.numpy().astype(np.float64)
    rows = np.arange(T) if T <= 2433 else np.random.default_rng(T).choice(T, 512, replace=False)
    ref = O.router_logits(x64[rows], w64, b64).astype(np.float64)
    err = np.abs(f64(lg)[rows] - ref)
    assert np.isfinite(f64(lg)).all()
    assert (err <= logit_error_bound(x64[rows], w64, b64)).all(), f"max err {err.max():.3e}"


@pytest.mark.parametrize("T,E,K,p", [(1, 128, 64, 0.7), (6, 128, 64, 0.7), (7, 128, -1, 0.7), (8, 128, 64, 0.7),
                                     (96, 128, 64, 0.7), (97, 128, 64, 0.7), (100, 128, -1, 0.7),
                                     (193, 128, 64, 0.7), (300, 256, -1, 0.7),
                                     (576, 128, 64, 0.0), (577, 128, -1, 0.5), (2048, 128, 64, 0.7),
                                     (2048, 128, -1, 0.7), (2432, 256, 40, 0.7), (2433, 128, 64, 0.7),
                                     (4096, 128, -1, 0.9)])
def test_router_route_dispatch_equals_separate_calls(T, E, K, p):
    """The one-call front half (router logits, routing, dispatch) equals
    decomoe_router_logits_ws + decomoe_route_dispatch bit for bit, whether
    the routing kernel reads the split router's partial sums (97 <= T <=
    2432) or plain logits, with the mass finished by the dispatch launch or by
    its own kernel."""
    d, k = 2048, 8
    g = torch.Generator().manual_seed(T + 3 * E)
    x = torch.randn(T, d, generator=g).to(torch.bfloat16).to(DEV)
    w_r = (torch.randn(E, d, generator=g) * 0.02).to(torch.bfloat16).to(DEV)
    bias = _zipf_bias(E).to(DEV)
    Kd = E if K == -1 else K

    def outs():
        return dict(logits=torch.empty(T, E, device=DEV), idx=torch.full((T, k), -9, dtype=torch.int32, device=DEV),
                    w=torch.empty(T, k, device=DEV), mass=torch.full((E,), -1.0, dtype=torch.float64, device=DEV),
                    Kdev=torch.zeros(1, dtype=torch.int32, device=DEV),
                    counts=torch.empty(Kd, dtype=torch.int32, device=DEV),
                    offsets=torch.empty(Kd + 1, dtype=torch.int32, device=DEV),
                    perm=torch.empty(T * k, dtype=torch.int32, device=DEV),
                    inv=torch.empty(T * k, dtype=torch.int32, device=DEV),
                    xp=torch.empty(T * k, d, dtype=torch.bfloat16, device=DEV))

    a, b = outs(), outs()
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    ws = dm.workspace(dm.decomoe_router_route_dispatch_workspace_bytes(T, d, E, k), DEV)
    dm.decomoe_router_route_dispatch(x, w_r, bias, a["logits"], K, k, a["idx"], a["w"], a["counts"], a["offsets"],
                                     a["perm"], a["inv"], a["xp"], ws, p=p, mass_out=a["mass"] if p > 0 else None,
                                     K_dev=a["Kdev"] if K == -1 else None, status=st)
    rws = dm.workspace(dm.decomoe_router_logits_ws_bytes(T, d, E), DEV)
    dm.decomoe_router_logits_ws(x, w_r, bias, b["logits"], rws, st)
    dws = dm.workspace(dm.decomoe_route_dispatch_workspace_bytes(T, k, E), DEV)
    dm.decomoe_route_dispatch(b["logits"], K, k, b["idx"], b["w"], x, b["counts"], b["offsets"], b["perm"], b["inv"],
                              b["xp"], dws, p=p, mass_out=b["mass"] if p > 0 else None,
                              K_dev=b["Kdev"] if K == -1 else None, status=st)
    torch.cuda.synchronize()
    assert dm.decomoe_read_status(st) == 0
    for key in a:
        u, v = a[key], b[key]
        if u.dtype in (torch.float32, torch.float64, torch.bfloat16):
            u = u.view({torch.float32: torch.int32, torch.float64: torch.int64, torch.bfloat16: torch.int16}[u.dtype])
            v = v.view(u.dtype)
        assert torch.equal(u, v), key
    if p > 0:
        assert (a["mass"] >= 0).all()
