"""The allocation-free dispatch entry point (decomoe_dispatch_noalloc).

It is meant for callers that cannot allocate device memory (a runtime that
owns all of HBM from start-up), so its scratch is a fixed array inside the
library. These checks call it through the C ABI and compare it with the
workspace-taking decomoe_dispatch on the same inputs, on two calls in a row
with different inputs (the shared array keeps the previous call's contents,
which must not leak into the next result). The file sorts last so that a
stop-at-first-failure run has already run every other test.
"""
import numpy as np
import pytest
import torch

import paper_2609_38823_gb300 as dm

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__

    __graft_entry__.build()
    dm.lib()


def _inputs(T, k, K, d, seed):
    g = torch.Generator().manual_seed(seed)
    # skewed expert ids over [0, K): low ids more frequent, like a mass-ordered pool
    p = 1.0 / torch.arange(1, K + 1, dtype=torch.float64) ** 1.1
    idx = torch.multinomial(p.expand(T, K), k, replacement=False, generator=g).to(torch.int32)
    x = torch.randn(T, d, generator=g).to(torch.bfloat16)
    return idx.to(DEV), x.to(DEV)


def _outputs(T, k, K, d):
    return (torch.full((K,), -7, dtype=torch.int32, device=DEV),
            torch.full((K + 1,), -7, dtype=torch.int32, device=DEV),
            torch.full((T * k,), -7, dtype=torch.int32, device=DEV),
            torch.full((T * k,), -7, dtype=torch.int32, device=DEV),
            torch.zeros((T * k, d), dtype=torch.bfloat16, device=DEV))


def test_noalloc_dispatch_matches_workspace_dispatch_twice():
    # second call: more tiles and a different K than the first, so stale
    # histogram entries from call 1 would show up if they were ever read
    for (T, k, K, d, seed) in ((300, 8, 64, 2048, 1), (2048, 8, 128, 2048, 2)):
        idx, x = _inputs(T, k, K, d, seed)
        ref = _outputs(T, k, K, d)
        ws = dm.workspace(dm.decomoe_dispatch_workspace_bytes(T, k, K), DEV)
        dm.decomoe_dispatch(idx, K, x, *ref[:4], ref[4], ws)
        got = _outputs(T, k, K, d)
        status = torch.zeros(1, dtype=torch.int32, device=DEV)
        dm.decomoe_dispatch_noalloc(idx, K, x, *got[:4], got[4], status)
        torch.cuda.synchronize()
        assert dm.decomoe_read_status(status) == 0
        for a, b in zip(got, ref):
            assert torch.equal(a, b)  # integer and copied bytes: bit-exact
        assert int(got[1][-1]) == T * k


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
