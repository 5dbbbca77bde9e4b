"""The allocation-free dispatch entry point (decomoe_dispatch_noalloc).

It is meant for callers that cannot allocate device memory (a runtime that
owns all of HBM from start-up), so its scratch is a fixed array inside the
library. These checks call it through the C ABI and compare it with the
workspace-taking decomoe_dispatch and with the oracle's dispatch on the same
inputs, on calls in a row with different inputs (the shared array keeps the
previous call's contents, which must not leak into the next result): one-tile
decode sizes, many tiles, no rows at all, no row copy, and an expert id
outside [0, K). The file sorts last so that a stop-at-first-failure run has
already run every other test.
"""
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

import paper_2609_38823_gb300 as dm
from oracle import decomoe_oracle as O

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda")
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__

    __graft_entry__.build()
    dm.lib()


def _inputs(T, k, K, d, seed):
    g = torch.Generator().manual_seed(seed)
    # skewed expert ids over [0, K): low ids more frequent, like a mass-ordered pool
    p = 1.0 / torch.arange(1, K + 1, dtype=torch.float64) ** 1.1
    if T > 0:
        idx = torch.multinomial(p.expand(T, K), k, replacement=False, generator=g).to(torch.int32)
    else:
        idx = torch.zeros((0, k), dtype=torch.int32)
    x = torch.randn(max(T, 1), d, generator=g).to(torch.bfloat16)[:T]
    return idx.to(DEV), x.to(DEV)


def _outputs(T, k, K, d):
    return (torch.full((K,), -7, dtype=torch.int32, device=DEV),
            torch.full((K + 1,), -7, dtype=torch.int32, device=DEV),
            torch.full((max(T * k, 1),), -7, dtype=torch.int32, device=DEV)[:T * k],
            torch.full((max(T * k, 1),), -7, dtype=torch.int32, device=DEV)[:T * k],
            torch.zeros((max(T * k, 1), d), dtype=torch.bfloat16, device=DEV)[:T * k])


# (T, k, K, d, seed, copy rows): one tile (T*k <= 1024) and several tiles, in
# an order where each call has a different tile count or K from the one before
CASES = ((300, 8, 64, 2048, 1, True), (1, 8, 64, 2048, 2, True), (2048, 8, 128, 2048, 3, True),
         (100, 8, 64, 2048, 4, True), (0, 8, 64, 2048, 5, True), (1100, 8, 96, 512, 6, False),
         (32, 2, 16, 256, 7, False), (16384, 8, 128, 64, 8, True))


def test_noalloc_dispatch_matches_workspace_dispatch_and_oracle_in_a_row():
    for (T, k, K, d, seed, rows) in CASES:
        idx, x = _inputs(T, k, K, d, seed)
        ref = _outputs(T, k, K, d)
        ws = dm.workspace(dm.decomoe_dispatch_workspace_bytes(T, k, K), DEV)
        dm.decomoe_dispatch(idx, K, x, *ref[:4], ref[4] if rows else None, ws)
        got = _outputs(T, k, K, d)
        status = torch.zeros(1, dtype=torch.int32, device=DEV)
        dm.decomoe_dispatch_noalloc(idx, K, x, *got[:4], got[4] if rows else None, status)
        torch.cuda.synchronize()
        assert dm.decomoe_read_status(status) == 0
        for a, b in zip(got, ref):
            assert torch.equal(a, b), (T, k, K)  # integer and copied bytes: bit-exact
        # the oracle's dispatch (a stable sort by expert id), element by element
        counts, offsets, perm, inv = O.dispatch(idx.cpu().numpy(), K)
        assert np.array_equal(got[0].cpu().numpy(), counts)
        assert np.array_equal(got[1].cpu().numpy(), offsets)
        assert np.array_equal(got[2].cpu().numpy(), perm)
        assert np.array_equal(got[3].cpu().numpy(), inv)
        assert int(got[1][-1]) == T * k
        if rows and T > 0:
            assert torch.equal(got[4].view(torch.int16), x[got[2].long()].view(torch.int16))
        elif not rows:
            assert not got[4].view(torch.int16).any()  # no rows copied when x_perm is null


@pytest.mark.parametrize("T,k,K", [(50, 2, 8), (400, 8, 64)])
def test_noalloc_dispatch_flags_expert_id_outside_prefix(T, k, K):
    # one tile and several tiles: the bad pair is reported and left out
    idx = np.random.default_rng(T).integers(0, K, size=(T, k))
    idx[3, 1] = K + 5
    idx_d = torch.from_numpy(idx.astype(np.int32)).to(DEV)
    counts = torch.empty(K, dtype=torch.int32, device=DEV)
    offsets = torch.empty(K + 1, dtype=torch.int32, device=DEV)
    perm = torch.empty(T * k, dtype=torch.int32, device=DEV)
    inv = torch.empty(T * k, dtype=torch.int32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    dm.decomoe_dispatch_noalloc(idx_d, K, None, counts, offsets, perm, inv, None, status)
    assert dm.decomoe_read_status(status) == dm.DECOMOE_ERR_BAD_INPUT
    assert int(offsets[-1]) == T * k - 1 and int(inv[3 * k + 1]) == -1


def test_noalloc_dispatch_rejects_oversized_input():
    # ceil(T*k/1024) * K beyond the fixed 65536-entry scratch
    T, k, K = 70000, 8, 128
    idx = torch.zeros((T, k), dtype=torch.int32, device=DEV)
    outs = _outputs(1, 1, K, 8)
    with pytest.raises(dm.DecomoeError) as e:
        dm.decomoe_dispatch_noalloc(idx, K, None, outs[0], outs[1], torch.empty(T * k, dtype=torch.int32, device=DEV),
                                    torch.empty(T * k, dtype=torch.int32, device=DEV), None)
    assert e.value.code == dm.DECOMOE_ERR_INVALID_ARG
    assert "fixed scratch" in str(e.value)


_FIRST_CALL_IN_CAPTURE = r"""
import torch
import paper_2609_38823_gb300 as dm
idx = torch.zeros((4, 2), dtype=torch.int32, device="cuda")
c = torch.empty(8, dtype=torch.int32, device="cuda")
o = torch.empty(9, dtype=torch.int32, device="cuda")
p = torch.empty(8, dtype=torch.int32, device="cuda")
v = torch.empty(8, dtype=torch.int32, device="cuda")
torch.cuda.synchronize()
g = torch.cuda.CUDAGraph()
s = torch.cuda.Stream()
code = None
with torch.cuda.stream(s):
    g.capture_begin()
    try:
        dm.decomoe_dispatch_noalloc(idx, 8, None, c, o, p, v, None)
    except dm.DecomoeError as e:
        code = e.code
    finally:
        g.capture_end()
assert code == dm.DECOMOE_ERR_INVALID_ARG, code
dm.decomoe_dispatch_noalloc(idx, 8, None, c, o, p, v, None)  # outside the capture: looks the array up
torch.cuda.synchronize()
assert c.tolist() == [8, 0, 0, 0, 0, 0, 0, 0] and o.tolist()[-1] == 8
print("ok")
"""


def test_noalloc_dispatch_first_call_inside_capture_is_rejected():
    # a fresh process, so that this is the first call on the device
    r = subprocess.run([sys.executable, "-c", _FIRST_CALL_IN_CAPTURE], cwd=ROOT, capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0 and r.stdout.strip().endswith("ok"), r.stdout + r.stderr
