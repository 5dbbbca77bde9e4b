"""Attention on the compacted sequence and over the text-only KV cache
(decomoe_attention) against the oracle's causal grouped-head attention:
decode steps (up to 64 queries per KV head: split keys in one thread-block
cluster per KV head, warp-level tensor-core products) and prefill (more: the
tcgen05 kernel), with ragged tiles, chunked prefill (n < C), sampled rows at
the full 16384-token sequence.

The layer shape is the 30B-A3B decoder's: 32 query heads and 4 KV heads of
128 (q = 4096, k_v = 512); the caches are one layer slice of the KV buffers
that the visual-block removal compacts ([T, 4, 128] bf16). Outputs are
compared at the bf16 output tolerance (fp32 scores, softmax and sums).
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
HQ, HKV, D = 32, 4, 128


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__

    __graft_entry__.build()
    dm.lib()


def _qkv(n, C, seed, Hq=HQ, Hkv=HKV):
    g = torch.Generator().manual_seed(seed)
    q = torch.randn(n, Hq, D, generator=g).to(torch.bfloat16)
    k = torch.randn(C, Hkv, D, generator=g).to(torch.bfloat16)
    v = torch.randn(C, Hkv, D, generator=g).to(torch.bfloat16)
    return q, k, v


def _run(q, k, v, scale=0.0):
    n, Hq, _ = q.shape
    C, Hkv, _ = k.shape
    out = torch.full((n, Hq, D), 9.0, dtype=torch.bfloat16, device=DEV)
    ws = dm.workspace(dm.decomoe_attention_workspace_bytes(n, C, Hq, Hkv, D), DEV)
    dm.decomoe_attention(q.to(DEV), k.to(DEV), v.to(DEV), out, ws, scale=scale)
    torch.cuda.synchronize()
    return out


@pytest.mark.parametrize("n,C", [(1, 1), (1, 63), (1, 64), (1, 65), (1, 127), (1, 128), (1, 272), (1, 2049),
                                 (2, 300), (8, 1552), (1, 8192), (1, 8193), (1, 16384), (1, 16385), (3, 129),
                                 (5, 40000), (8, 20000), (4, 1900), (4, 2049), (7, 1000), (2, 2), (3, 3),
                                 (8, 8)])
def test_attention_decode_parity(n, C):
    # (4, 1900): 32 query rows on a cluster of 15, the most receive slots
    # (ceil(32 / 15) * 15 = 45); (7, 1000): a second query tile of 24 rows;
    # (2, 2), (3, 3), (8, 8): every query's causal limit inside the one chunk
    q, k, v = _qkv(n, C, seed=C + n)
    out = _run(q, k, v)
    ref = O.attention(f64(q), f64(k), f64(v))
    assert_close_out(f64(out), ref, BF16_REL_L2, BF16_MAX_ABS, f"attention n={n} C={C}")


@pytest.mark.parametrize("n,C", [(9, 9), (9, 300), (128, 128), (129, 200), (300, 300), (640, 1000), (1024, 1024)])
def test_attention_prefill_parity(n, C):
    q, k, v = _qkv(n, C, seed=7 * C + n)
    out = _run(q, k, v)
    ref = O.attention(f64(q), f64(k), f64(v))
    assert_close_out(f64(out), ref, BF16_REL_L2, BF16_MAX_ABS, f"prefill attention n={n} C={C}")


def _sampled_rows(out, q, k, v, rows, label):
    """Query row i of a launch over (n, C) is attention at position C - n + i
    over keys 0..C - n + i: the oracle on that one row and prefix."""
    n, C = q.shape[0], k.shape[0]
    got = f64(out[rows].cpu())
    ref = np.concatenate([O.attention(f64(q[i:i + 1]), f64(k[:C - n + i + 1]), f64(v[:C - n + i + 1]))
                          for i in rows])
    assert_close_out(got, ref, BF16_REL_L2, BF16_MAX_ABS, label)


@pytest.mark.parametrize("n,C", [(2048, 2048), (16384, 16384), (2048, 16384)])
def test_attention_prefill_full_sizes_sampled(n, C):
    """The two prefill sizes of the 16384-token workload: the full sequence
    (layers before the exit) and its 2048 text rows (after it), plus a
    2048-query chunk at the end of the full cache."""
    q, k, v = _qkv(n, C, seed=n + C)
    out = _run(q, k, v)
    rng = np.random.default_rng(n)
    rows = sorted(set([0, 1, 127, 128, n - 129, n - 1] + rng.integers(0, n, 10).tolist()))
    _sampled_rows(out, q, k, v, rows, f"prefill attention n={n} C={C} (sampled rows)")


def test_attention_prefill_grouping_and_scale():
    # 8 query heads on 2 KV heads: 40 queries make 160 per KV head
    q, k, v = _qkv(40, 333, seed=6, Hq=8, Hkv=2)
    out = _run(q, k, v, scale=0.05)
    ref = O.attention(f64(q), f64(k), f64(v), scale=0.05)
    assert_close_out(f64(out), ref, BF16_REL_L2, BF16_MAX_ABS, "prefill grouping and scale")


def test_attention_prefill_is_deterministic():
    q, k, v = _qkv(300, 700, seed=9)
    a = _run(q, k, v)
    b = _run(q, k, v)
    assert torch.equal(a, b)


def test_attention_decode_workspace_and_repeats_bitwise():
    """Decode sizes take no workspace while one cluster per KV head streams
    at most four chunks per block (a null pointer is accepted there); a
    longer cache is split over several clusters per head where the SMs allow
    and takes a small workspace for their merged rows (a missing one is
    rejected). Every call gives the same bits, in any order of sizes."""
    sizes = [(1, 16384), (1, 300), (8, 2049), (2, 64), (1, 1), (4, 5000), (1, 40000)]
    for n, C in sizes:
        if C <= 16 * 128 * 4:
            assert dm.decomoe_attention_workspace_bytes(n, C, HQ, HKV, D) == 0
    lib = dm.lib()
    first = {}
    for rep in range(2):
        for n, C in sizes:
            # device copies held in variables: a temporary's memory could be
            # handed to the next copy before the launch reads it
            q, k, v = (t.to(DEV) for t in _qkv(n, C, seed=31 * C + n))
            out = torch.empty(n, HQ, D, dtype=torch.bfloat16, device=DEV)
            nbytes = dm.decomoe_attention_workspace_bytes(n, C, HQ, HKV, D)
            ws = dm.workspace(nbytes, DEV)
            args = (q.data_ptr(), n, k.data_ptr(), v.data_ptr(), C, HQ, HKV, D, 0.0, out.data_ptr())
            stream = torch.cuda.current_stream().cuda_stream
            if nbytes > 0 and rep == 0:
                assert lib.decomoe_attention(*args, None, 0, None, stream) == dm.DECOMOE_ERR_WORKSPACE
            rc = lib.decomoe_attention(*args, None if ws is None else ws.data_ptr(), nbytes, None, stream)
            torch.cuda.synchronize()
            assert rc == 0
            if rep == 0:
                first[(n, C)] = out.cpu()
            else:
                assert torch.equal(out.cpu(), first[(n, C)]), (n, C)


def test_attention_grouping_and_scale():
    # 8 query heads on 2 KV heads and an explicit scale
    q, k, v = _qkv(2, 200, seed=5, Hq=8, Hkv=2)
    out = _run(q, k, v, scale=0.05)
    ref = O.attention(f64(q), f64(k), f64(v), scale=0.05)
    assert_close_out(f64(out), ref, BF16_REL_L2, BF16_MAX_ABS, "grouping and scale")


def test_attention_on_compacted_cache_equals_masked_full_cache():
    """The stack workload's sequence (16 system rows, 1280 visual, 256 text):
    a text token's decode step over the compacted cache (the visual block
    removed by decomoe_drop_visual_block) matches the oracle run on the full
    cache with the visual rows removed, and equals what the oracle gives on
    the full sequence with those keys hidden (oracle pin)."""
    wl = W.STACK
    C_full = wl.T
    q, k, v = _qkv(1, C_full, seed=11)
    kc = torch.empty(C_full - wl.nv, HKV, D, dtype=torch.bfloat16, device=DEV)
    vc = torch.empty_like(kc)
    dm.decomoe_drop_visual_block(k.to(DEV).view(C_full, HKV * D), kc.view(-1, HKV * D), wl.v0, wl.nv)
    dm.decomoe_drop_visual_block(v.to(DEV).view(C_full, HKV * D), vc.view(-1, HKV * D), wl.v0, wl.nv)
    out = _run(q, kc.cpu(), vc.cpu())
    ref = O.attention(f64(q), O.drop_visual_block(f64(k), wl.v0, wl.nv), O.drop_visual_block(f64(v), wl.v0, wl.nv))
    assert_close_out(f64(out), ref, BF16_REL_L2, BF16_MAX_ABS, "decode over the compacted cache")


def test_attention_prefill_on_compacted_sequence():
    """Prefill after the visual block has left: the compacted hidden rows'
    queries over the compacted K and V (1552 - 1280 = 272 rows) equal the
    oracle's attention on the full sequence's caches with the visual rows
    removed."""
    wl = W.STACK
    C_full = wl.T
    q, k, v = _qkv(C_full, C_full, seed=12)
    dev = [t.to(DEV).view(C_full, -1) for t in (q, k, v)]
    comp = [torch.empty(C_full - wl.nv, t.shape[1], dtype=torch.bfloat16, device=DEV) for t in dev]
    for src, dst in zip(dev, comp):
        dm.decomoe_drop_visual_block(src, dst, wl.v0, wl.nv)
    qc, kc, vc = (comp[0].view(-1, HQ, D).cpu(), comp[1].view(-1, HKV, D).cpu(), comp[2].view(-1, HKV, D).cpu())
    out = _run(qc, kc, vc)
    drop = lambda t: O.drop_visual_block(f64(t), wl.v0, wl.nv)  # noqa: E731
    ref = O.attention(drop(q), drop(k), drop(v))
    assert_close_out(f64(out), ref, BF16_REL_L2, BF16_MAX_ABS, "prefill over the compacted sequence")


def test_attention_rejects_unsupported_shapes():
    q, k, v = _qkv(1, 10, seed=1)
    ws = dm.workspace(1 << 20, DEV)
    out = torch.empty(1, HQ, D, dtype=torch.bfloat16, device=DEV)
    with pytest.raises(dm.DecomoeError) as e:  # more queries than keys
        dm.decomoe_attention(q.to(DEV).repeat(11, 1, 1), k.to(DEV), v.to(DEV), out.repeat(11, 1, 1), ws)
    assert e.value.code == dm.DECOMOE_ERR_INVALID_ARG
    with pytest.raises(dm.DecomoeError) as e:  # 31 query heads on 4 KV heads
        dm.decomoe_attention(q.to(DEV)[:, :31].contiguous(), k.to(DEV), v.to(DEV), out[:, :31].contiguous(), ws)
    assert e.value.code == dm.DECOMOE_ERR_INVALID_ARG
    q3, k3, v3 = _qkv(40, 100, seed=2, Hq=12, Hkv=4)  # prefill sizes with an odd group (3 heads per KV head)
    with pytest.raises(dm.DecomoeError) as e:
        dm.decomoe_attention(q3.to(DEV), k3.to(DEV), v3.to(DEV), torch.empty(40, 12, D, dtype=torch.bfloat16,
                                                                               device=DEV), ws)
    assert e.value.code == dm.DECOMOE_ERR_INVALID_ARG


@pytest.mark.parametrize("n,C,Hq,Hkv", [(1, 20000, 16, 8), (2, 12000, 32, 2), (1, 9000, 8, 8), (4, 30000, 8, 1)])
def test_attention_decode_long_caches_other_groupings(n, C, Hq, Hkv):
    """Long caches split over several clusters per KV head (the cluster size
    and count follow the number of (head, query tile) sets) for other head
    groupings, against the oracle, and bit-identical on a second call."""
    q, k, v = _qkv(n, C, seed=C + Hkv, Hq=Hq, Hkv=Hkv)
    out = _run(q, k, v)
    ref = O.attention(f64(q), f64(k), f64(v))
    assert_close_out(f64(out), ref, BF16_REL_L2, BF16_MAX_ABS, f"attention n={n} C={C} Hq={Hq} Hkv={Hkv}")
    assert torch.equal(_run(q, k, v), out)


def test_attention_decode_chained_calls_in_a_graph():
    """Three decode steps in a row, each step's query the previous step's
    output, over a long cache (several clusters per head and the merge
    launch), the text-only one and the long one again, all sharing one
    workspace: the launches are programmatic, so each must wait for the one
    before it both to read its output and to reuse the workspace. Captured
    in a CUDA graph and replayed, the outputs equal the eager calls'
    bits."""
    sizes = [16385, 2049, 16385]
    g = torch.Generator().manual_seed(77)
    q0 = torch.randn(1, HQ, D, generator=g).to(torch.bfloat16).to(DEV)
    kv = [(torch.randn(C, HKV, D, generator=g).to(torch.bfloat16).to(DEV),
           torch.randn(C, HKV, D, generator=g).to(torch.bfloat16).to(DEV)) for C in sizes]
    nbytes = max(dm.decomoe_attention_workspace_bytes(1, C, HQ, HKV, D) for C in sizes)
    assert nbytes > 0
    ws = dm.workspace(nbytes, DEV)

    def chain(outs):
        q = q0
        for (k, v), o in zip(kv, outs):
            dm.decomoe_attention(q, k, v, o, ws)
            q = o

    eager = [torch.empty(1, HQ, D, dtype=torch.bfloat16, device=DEV) for _ in sizes]
    chain(eager)
    torch.cuda.synchronize()
    graphed = [torch.full((1, HQ, D), 7.0, dtype=torch.bfloat16, device=DEV) for _ in sizes]
    gr = dm.capture_graph(lambda: chain(graphed))
    for _ in range(3):
        for o in graphed:
            o.fill_(7.0)
        gr.replay()
        torch.cuda.synchronize()
        for i, (a, b) in enumerate(zip(eager, graphed)):
            assert torch.equal(a, b), i
    ref = O.attention(f64(q0.cpu()), f64(kv[0][0].cpu()), f64(kv[0][1].cpu()))
    assert_close_out(f64(eager[0].cpu()), ref, BF16_REL_L2, BF16_MAX_ABS, "chained step 1")
