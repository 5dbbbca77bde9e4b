"""Host-side checks of the C ABI that need no GPU: the library loads, exports
every function include/decomoe.h declares, rejects bad arguments before
launching anything, and its plain-C prefix selection (Eq. 12) matches the
oracle exactly."""
import ctypes
import os
import re

import numpy as np
import pytest

import paper_2609_38823_gb300 as dm
from oracle import decomoe_oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built_lib():
    import __graft_entry__

    __graft_entry__.build()
    return dm.lib()


def _declared():
    names = []
    for fn in sorted(os.listdir(os.path.join(ROOT, "include"))):
        if fn.endswith(".h"):
            txt = open(os.path.join(ROOT, "include", fn)).read()
            names += re.findall(r"DECOMOE_API\s+[\w\s\*]+?\b(decomoe_\w+)\s*\(", txt)
    return names


def test_every_declared_symbol_is_exported_and_bound():
    names = _declared()
    assert len(names) >= 20
    L = dm.lib()
    for n in names:
        assert hasattr(L, n), n
        assert n in dm.SIGNATURES, f"{n} has no binding"


def test_version():
    assert dm.decomoe_version() == 100


@pytest.mark.parametrize("seed", range(40))
def test_select_prefix_c_matches_oracle(seed):
    r = np.random.default_rng(seed)
    E = int(r.choice([2, 16, 64, 128, 256]))
    k = int(r.integers(1, min(E, 32) + 1))
    s = (1.0 / (np.arange(E) + 1.0) ** r.uniform(0.0, 2.0)) * r.uniform(0.0, 2.0, E) * r.uniform(1, 3000)
    if seed % 5 == 0:
        s[r.integers(0, E, size=E // 3)] = 0.0
    for p in (0.05, 0.1, 0.2, 0.5, 0.7, 0.9, 0.99, 1.0):
        assert dm.decomoe_select_prefix(s, k, p) == O.select_prefix(s, p, k)


def test_select_prefix_c_edge_cases():
    assert dm.decomoe_select_prefix(np.zeros(8), 3, 0.7) == 3
    assert dm.decomoe_select_prefix(np.array([0.0, 0.0, 5.0, 0.0]), 1, 1.0) == 4
    for bad_p in (0.0, -0.1, 1.5, float("nan")):
        with pytest.raises(dm.DecomoeError) as e:
            dm.decomoe_select_prefix(np.ones(4), 1, bad_p)
        assert e.value.code == dm.DECOMOE_ERR_INVALID_ARG
    with pytest.raises(dm.DecomoeError):
        dm.decomoe_select_prefix(np.ones(4), 5, 0.5)  # k > E
    with pytest.raises(dm.DecomoeError):
        dm.decomoe_select_prefix(np.array([1.0, -1.0]), 1, 0.5)


def test_argument_errors_are_caught_before_launch():
    L = dm.lib()
    fake = ctypes.c_void_p(0x1000)  # never dereferenced: the checks fail first
    # k > K
    assert L.decomoe_route_prefix(fake, 4, 16, 16, 2, 3, fake, fake, None, None, 0, None) == 1
    # K > E
    assert L.decomoe_route_prefix(fake, 4, 16, 16, 17, 2, fake, fake, None, None, 0, None) == 1
    # E beyond the kernel's limit
    assert L.decomoe_route_prefix(fake, 4, 300, 300, 8, 2, fake, fake, None, None, 0, None) == 1
    # visual block past the end
    assert L.decomoe_drop_visual_block(fake, fake, 10, 16, 8, 3, 1, 160, 112, None) == 1
    # m not a multiple of the gate/up block
    assert L.decomoe_expert_swiglu(fake, fake, 100, 4, 256, 100, 0, fake, fake, fake, fake, None, None, None) == 1
    # bf16: m a multiple of the block but not of 128 (the tensor-core tiles span
    # 256 interleaved gate/up columns); the fused form and the layer refuse it too
    assert L.decomoe_expert_swiglu(fake, fake, 100, 4, 256, 192, 0, fake, fake, fake, fake, None, None, None) == 1
    assert "m % 128" in L.decomoe_last_error().decode()
    assert L.decomoe_expert_swiglu_fused(fake, fake, 100, 4, 256, 192, 0, fake, fake, fake, fake, fake, None,
                                         None) == 1
    assert L.decomoe_expert_swiglu_fused(fake, fake, 20, 4, 256, 192, 0, fake, fake, fake, fake, fake, None,
                                         None) == 1
    assert L.decomoe_moe_layer(fake, fake, None, fake, fake, 4, 256, 16, 4, 192, 0, 4, 0.0, None, fake,
                               None, None, fake, 1 << 30, None, None) == 1
    assert "m % 128" in L.decomoe_last_error().decode()
    # K_fixed < k
    assert L.decomoe_moe_layer(fake, fake, None, fake, fake, 4, 256, 16, 4, 128, 0, 2, 0.0, None, fake,
                               None, None, fake, 1 << 30, None, None) == 1
    msg = L.decomoe_last_error().decode()
    assert "K_fixed" in msg
    # SAVB gate: d not a multiple of 64; no text rows
    assert L.decomoe_savb_gate(fake, 10, 100, 0, 0, 0, fake, fake, fake, fake, 8, 0.5, fake, fake, fake, 1 << 20,
                               None) == 1
    assert L.decomoe_savb_gate(fake, 10, 64, 0, 0, 10, fake, fake, fake, fake, 8, 0.5, fake, fake, fake, 1 << 20,
                               None) == 1
    # calibration: a case without text tokens; overlapping permutation buffers
    assert L.decomoe_calib_case_mass(fake, 8, 16, 16, 2, 0, 8, fake, fake, 1 << 20, None) == 1
    assert L.decomoe_permute_experts(fake, ctypes.c_void_p(0x1000 + 64), fake, 4, 64, None, None) == 1
    assert L.decomoe_mean_mass_order(fake, 300, 1, fake, None, None, None) == 1
    # too-small workspace
    assert L.decomoe_dispatch(fake, 4, 2, 4, None, 0, 0, fake, fake, fake, fake, None, fake, 1, None,
                              None) == dm.DECOMOE_ERR_WORKSPACE


def test_workspace_queries():
    assert dm.decomoe_route_workspace_bytes(2048, 128) >= 32 * 128 * 8
    assert dm.decomoe_dispatch_workspace_bytes(2048, 8, 128) >= 16 * 128 * 4
    b = dm.decomoe_moe_layer_workspace_bytes(2048, 2048, 128, 8, 768, 0)
    assert b >= 2048 * 8 * (2048 * 2 * 2 + 768 * 2)  # x_perm, y_perm and h
    offs = dm.decomoe_moe_layer_workspace_layout(2048, 2048, 128, 8, 768, 0)
    assert offs == sorted(offs) and all(o % 256 == 0 for o in offs)


def test_expert_ready_counter_count():
    # the one-launch expert FFN needs two counters per possible M-tile
    # (h stored, rows gathered): at most rows/128 + K M-tiles, one spare each
    for rows, K in ((16384, 64), (1, 1), (1000, 128), (0, 8)):
        assert dm.decomoe_expert_swiglu_ready_ints(rows, K) == 2 * (rows // 128 + K + 1)
    assert dm.decomoe_expert_swiglu_ready_ints(-1, 8) == 0
    assert dm.decomoe_expert_swiglu_ready_ints(100, 0) == 0
