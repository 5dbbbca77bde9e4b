"""Edge cases of every C-ABI call on the GPU: empty invocations (T = 0, no
rows, no batches), a visual block that is the whole sequence, the degenerate
prefixes K = k (every token takes the whole prefix) and k = 1, and the gate
without text rows (rejected before any launch)."""
import numpy as np
import pytest
import torch

import paper_2609_38823_gb300 as dm
import workloads as W
from oracle import decomoe_oracle as O
from tests.helpers import W_ABS

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__

    __graft_entry__.build()
    torch.cuda.set_device(0)
    dm.lib()


def _i32(*shape, fill=-5):
    return torch.full(shape, fill, dtype=torch.int32, device=DEV)


def test_empty_invocation_every_call():
    E, k, d, m = 128, 8, 256, 128
    x = torch.empty(0, d, dtype=torch.bfloat16, device=DEV)
    w_r = torch.randn(E, d, device=DEV).to(torch.bfloat16)
    bias = torch.zeros(E, device=DEV)
    logits = torch.empty(0, E, device=DEV)
    dm.decomoe_router_logits(x, w_r, bias, logits)
    # routing with the mass: an empty invocation has zero mass
    mass = torch.full((E,), 7.0, dtype=torch.float64, device=DEV)
    idx = torch.empty(0, k, dtype=torch.int32, device=DEV)
    w = torch.empty(0, k, device=DEV)
    dm.decomoe_route_prefix(logits, 64, k, idx, w, mass, dm.workspace(dm.decomoe_route_workspace_bytes(0, E), DEV))
    torch.cuda.synchronize()
    assert (mass == 0).all()
    # dispatch: zero counts and offsets
    counts, offsets = _i32(64), _i32(65)
    perm, inv = torch.empty(0, dtype=torch.int32, device=DEV), torch.empty(0, dtype=torch.int32, device=DEV)
    xp = torch.empty(0, d, dtype=torch.bfloat16, device=DEV)
    dm.decomoe_dispatch(idx, 64, x, counts, offsets, perm, inv, xp,
                        dm.workspace(dm.decomoe_dispatch_workspace_bytes(0, k, 64), DEV))
    torch.cuda.synchronize()
    assert (counts == 0).all() and (offsets == 0).all()
    # routing + dispatch with a device-selected prefix: zero mass selects K = k
    counts, offsets, K_dev = _i32(E), _i32(E + 1), _i32(1)
    dm.decomoe_route_dispatch(logits, -1, k, idx, w, x, counts, offsets, perm, inv, xp,
                              dm.workspace(dm.decomoe_route_dispatch_workspace_bytes(0, k, E), DEV), p=0.7,
                              mass_out=mass, K_dev=K_dev)
    torch.cuda.synchronize()
    assert int(K_dev) == k and (counts == 0).all() and (offsets == 0).all()
    # experts with no rows, combine of no tokens
    w_gu = (torch.randn(E, 2 * m, d, device=DEV) * 0.02).to(torch.bfloat16)
    w_dn = (torch.randn(E, d, m, device=DEV) * 0.02).to(torch.bfloat16)
    h = torch.empty(0, m, dtype=torch.bfloat16, device=DEV)
    y = torch.empty(0, d, dtype=torch.bfloat16, device=DEV)
    dm.decomoe_expert_swiglu(xp, offsets[:65], 64, w_gu, w_dn, h, y)
    out = torch.empty(0, d, dtype=torch.bfloat16, device=DEV)
    dm.decomoe_combine(y, inv, w.view(0, k), out)
    # the whole layer
    ws = dm.workspace(dm.decomoe_moe_layer_workspace_bytes(0, d, E, k, m, dm.DECOMOE_BF16), DEV)
    for K in (64, -1, 0):
        dm.decomoe_moe_layer(x, w_r, bias, w_gu, w_dn, k, out, ws, K_fixed=K, p=0.7)
    # compaction of no batches, and of a sequence that is all visual
    src = torch.randn(3, 10, 64, device=DEV).to(torch.bfloat16)
    none = torch.empty(0, 64, dtype=torch.bfloat16, device=DEV)
    dm.decomoe_drop_visual_block(none, torch.empty(0, 64, dtype=torch.bfloat16, device=DEV), 0, 0)
    dm.decomoe_drop_visual_block(src, torch.empty(3, 0, 64, dtype=torch.bfloat16, device=DEV), 0, 10)
    dm.decomoe_rmsnorm(x, x, 1e-6)
    torch.cuda.synchronize()


def test_gate_without_text_rows_is_rejected():
    d, H = 64, 8
    h = torch.randn(10, d, device=DEV)
    prm = [torch.zeros(H, 2 * d, device=DEV), torch.zeros(H, device=DEV), torch.zeros(2, H, device=DEV),
           torch.zeros(2, device=DEV)]
    p = torch.empty(1, device=DEV)
    ex = torch.empty(1, dtype=torch.int32, device=DEV)
    ws = dm.workspace(dm.decomoe_savb_gate_workspace_bytes(d, H), DEV)
    with pytest.raises(dm.DecomoeError) as e:
        dm.decomoe_savb_gate(h, 0, 10, *prm, 0.5, p, ex, ws)
    assert e.value.code == dm.DECOMOE_ERR_INVALID_ARG


@pytest.mark.parametrize("T,E,K,k", [(300, 128, 8, 8), (64, 16, 2, 2), (129, 128, 1, 1), (50, 256, 256, 1)])
def test_degenerate_prefixes(T, E, K, k):
    """K = k: every token routes to every expert of the prefix (weights = the
    softmax over the prefix); k = 1: one expert per token with weight 1."""
    a = W.make_logits(T, E, std=0.9, seed=9, wid=70 + E)
    idx = torch.empty(T, k, dtype=torch.int32, device=DEV)
    w = torch.empty(T, k, device=DEV)
    dm.decomoe_route_prefix(a.to(DEV), K, k, idx, w)
    torch.cuda.synchronize()
    ri, rw = O.route_prefix(a.numpy(), K, k)
    keep = O.prefix_margin(a.numpy(), K, k) >= 1e-6
    assert np.array_equal(idx.cpu().numpy()[keep], ri[keep])
    assert np.abs(w.cpu().numpy().astype(np.float64) - rw).max() <= W_ABS
    if K == k:
        assert (np.sort(idx.cpu().numpy(), axis=1) == np.arange(K)[None, :]).all()
    if k == 1:
        assert (w.cpu().numpy() == 1.0).all()
