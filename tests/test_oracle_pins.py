"""Pins of the CPU oracle against what the paper and the mathematics fix.

Every check here computes its expectation by a route other than the oracle's
own code: brute force on tiny inputs, a textbook top-k MoE written with torch
CPU ops, closed forms, or invariants the paper states. No test here needs a GPU.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import decomoe_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
rng = np.random.default_rng(1234)


def _logits(T, E, seed, bias=None, std=1.0):
    r = np.random.default_rng(seed)
    a = r.standard_normal((T, E)) * std
    if bias is not None:
        a = a + bias[None, :]
    return a.astype(np.float32)


# ---------------------------------------------------------------- router (Eq. 1)

def test_router_logits_bruteforce_fsum():
    r = np.random.default_rng(0)
    x = r.standard_normal((5, 7)).astype(np.float32)
    w = r.standard_normal((4, 7)).astype(np.float32)
    b = r.standard_normal(4).astype(np.float32)
    a = O.router_logits(x, w, b)
    assert a.dtype == np.float32
    for t in range(5):
        for e in range(4):
            exact = math.fsum([float(x[t, j]) * float(w[e, j]) for j in range(7)] + [float(b[e])])
            # both round a float64-accurate value once to float32: at most 1 ulp apart
            assert abs(float(a[t, e]) - exact) <= np.spacing(np.float32(abs(exact)))


def test_router_logits_onehot_closed_form():
    d, E = 6, 5
    w = np.arange(E * d, dtype=np.float32).reshape(E, d) / 7.0
    b = np.linspace(1, -1, E).astype(np.float32)
    x = np.eye(d, dtype=np.float32)
    a = O.router_logits(x, w, b)
    np.testing.assert_array_equal(a, (w.T + b[None, :]).astype(np.float32))


def test_softmax_closed_forms():
    a, c = 0.3, -1.7
    s = O.softmax(np.array([[a, c]]))
    assert s[0, 0] == pytest.approx(1.0 / (1.0 + math.exp(c - a)), rel=1e-15)
    v = rng.standard_normal((3, 9))
    np.testing.assert_allclose(O.softmax(v).sum(-1), 1.0, rtol=0, atol=1e-15)
    np.testing.assert_allclose(O.softmax(v + 11.0), O.softmax(v), rtol=1e-13)


# ---------------------------------------------------------------- top-k (Eqs. 7, 10)

def test_topk_bruteforce_subsets():
    for seed in range(20):
        E, k = 7, 3
        v = np.random.default_rng(seed).standard_normal(E).astype(np.float32)
        got = O.topk(v[None, :], k)[0]
        best = max(itertools.combinations(range(E), k), key=lambda S: sum(float(v[e]) for e in S))
        assert set(got.tolist()) == set(best)
        assert all(v[got[i]] >= v[got[i + 1]] for i in range(k - 1))


def test_topk_ties_lower_index_first():
    v = np.array([[0.5, 2.0, 0.5, 2.0, 0.5]], np.float32)
    assert O.topk(v, 3)[0].tolist() == [1, 3, 0]


def test_full_pool_route_matches_textbook_torch():
    a = _logits(40, 16, 3)
    R, w = O.full_pool_route(a, 4)
    t = torch.from_numpy(a.astype(np.float64))
    p = torch.softmax(t, dim=-1)
    tv, ti = torch.topk(p, 4, dim=-1, sorted=True)
    tw = tv / tv.sum(-1, keepdim=True)
    assert np.array_equal(R, ti.numpy())
    np.testing.assert_allclose(w, tw.numpy(), rtol=1e-13, atol=1e-15)


def test_ranking_by_probability_equals_ranking_by_logit():
    a = _logits(200, 32, 9, std=3.0)
    by_q = np.argsort(-O.softmax(a), axis=-1, kind="stable")[:, :8]
    assert np.array_equal(O.topk(a, 8), by_q)


# ---------------------------------------------------------------- activated mass (Eq. 11)

def test_activated_mass_bruteforce_per_expert():
    T, E, k = 12, 9, 3
    a = _logits(T, E, 5)
    s = O.activated_mass(a, k)
    s_bf = np.zeros(E)
    for e in range(E):
        for i in range(T):
            row = [float(v) for v in a[i]]
            q = [math.exp(v - max(row)) for v in row]
            top = sorted(range(E), key=lambda j: (-row[j], j))[:k]
            if e in top:
                s_bf[e] += q[e] / sum(q[j] for j in top)
    np.testing.assert_allclose(s, s_bf, rtol=1e-13, atol=1e-15)


def test_activated_mass_total_is_token_count():
    a = _logits(300, 64, 7)
    s = O.activated_mass(a, 8)
    assert s.sum() == pytest.approx(300.0, rel=1e-13)
    assert (s >= 0).all()


def test_activated_mass_equal_top_logits_split_evenly():
    # two tokens whose two largest logits are equal: each gets weight 1/2
    a = np.array([[3.0, 3.0, -1.0, -2.0], [-5.0, 0.0, 7.0, 7.0]], np.float32)
    s = O.activated_mass(a, 2)
    np.testing.assert_allclose(s, [0.5, 0.5, 0.5, 0.5], rtol=0, atol=1e-15)


# ---------------------------------------------------------------- prefix length (Eq. 12)

def _select_bruteforce(s, p, k):
    E = len(s)
    tot = math.fsum(s)
    ok = [K for K in range(1, E + 1) if math.fsum(s[:K]) >= p * tot * (1 - 1e-12)]
    return max(k, min(ok))


def test_select_prefix_bruteforce():
    for seed in range(50):
        r = np.random.default_rng(seed)
        E = int(r.integers(2, 40))
        k = int(r.integers(1, E + 1))
        s = r.random(E) ** 3 * 10
        for p in (0.05, 0.3, 0.5, 0.7, 0.9, 0.999):
            K = O.select_prefix(s, p, k)
            # tolerance-free brute force can differ only when a partial ratio
            # is within rounding of p; such draws are skipped
            ratios = np.cumsum(s) / s.sum()
            if np.min(np.abs(ratios - p)) < 1e-9:
                continue
            assert K == _select_bruteforce(list(s), p, k)


def test_select_prefix_invariants_from_paper():
    # K >= k always; K monotone non-decreasing in p; p = 1 keeps the full pool
    # (Appendix sweep: average prefix 128.0 of 128 at p = 1.0)
    with open(os.path.join(GOLDEN, "rcep_prefix_vs_p.json")) as f:
        g = json.load(f)
    E, k = g["E"], g["k_moe"]
    for seed in range(30):
        r = np.random.default_rng(100 + seed)
        # Zipf-like skew over the reordered index, like a calibrated order
        s = (1.0 / (np.arange(E) + 1.0) ** r.uniform(0.5, 2.0)) * r.uniform(0.5, 1.5, E)
        Ks = [O.select_prefix(s, p, k) for p in g["p"]]
        assert all(K >= k for K in Ks)
        assert all(Ks[i] <= Ks[i + 1] for i in range(len(Ks) - 1))
        assert Ks[-1] == E
        # mass concentrated so that the first k experts cover >= 20%: the
        # clamp gives exactly k at p = 0.1 and 0.2 (sweep: 8.0 = k_moe there)
        if np.cumsum(s)[k - 1] / s.sum() >= 0.2:
            assert Ks[0] == k and Ks[1] == k
    # the published sweep itself is monotone, starts at k_moe and ends at E
    avg = g["avg_prefix"]
    assert avg[0] == k and avg[1] == k and avg[-1] == E
    assert all(avg[i] <= avg[i + 1] for i in range(len(avg) - 1))


def test_select_prefix_edge_cases():
    s = np.array([0.0, 0.0, 5.0, 0.0])
    assert O.select_prefix(s, 0.5, 1) == 3
    assert O.select_prefix(s, 1.0, 1) == 4          # p = 1 -> E
    assert O.select_prefix(np.zeros(4), 0.7, 2) == 2  # empty invocation -> k
    with pytest.raises(ValueError):
        O.select_prefix(s, 0.0, 1)
    with pytest.raises(ValueError):
        O.select_prefix(s, 1.5, 1)


# ---------------------------------------------------------------- prefix routing

def test_route_prefix_full_span_is_ordinary_topk_moe():
    a = _logits(50, 16, 11)
    i1, w1 = O.route_prefix(a, 16, 2)
    i2, w2 = O.full_pool_route(a, 2)
    assert np.array_equal(i1, i2)
    np.testing.assert_allclose(w1, w2, rtol=1e-13)


def test_route_prefix_bruteforce_and_softmax_over_picks():
    for seed in range(10):
        a = _logits(6, 10, 20 + seed)
        for K in (3, 5, 10):
            idx, w = O.route_prefix(a, K, 3)
            assert (idx < K).all()
            np.testing.assert_allclose(w.sum(-1), 1.0, atol=1e-14)
            for t in range(6):
                best = max(itertools.combinations(range(K), 3),
                           key=lambda S: sum(float(a[t, e]) for e in S))
                assert set(idx[t].tolist()) == set(best)
                picks = [float(a[t, e]) for e in idx[t]]
                z = [math.exp(v - max(picks)) for v in picks]
                np.testing.assert_allclose(w[t], np.array(z) / sum(z), rtol=1e-13)


def test_route_prefix_does_not_intersect_full_pool_topk():
    # full-pool top-2 of this token is {7, 6}, both outside the prefix K=4.
    # Intersecting would leave no expert; the paper's rule reruns top-k
    # inside the prefix and still returns exactly k experts.
    a = np.array([[0.1, 0.4, 0.2, 0.3, -1.0, -2.0, 5.0, 6.0]], np.float32)
    idx, w = O.route_prefix(a, 4, 2)
    assert idx[0].tolist() == [1, 3]
    v = a[0, [1, 3]].astype(np.float64)
    e = np.exp(v - v[0])
    np.testing.assert_allclose(w[0], e / e.sum(), rtol=1e-14)


def test_route_prefix_weights_invariant_to_K_when_set_unchanged():
    a = _logits(30, 20, 4, bias=-np.log(np.arange(20) + 1.0))
    i1, w1 = O.route_prefix(a, 20, 4)
    i2, w2 = O.route_prefix(a, 12, 4)
    same = (i1 == i2).all(-1)
    assert same.any()
    np.testing.assert_allclose(w1[same], w2[same], rtol=1e-13)


def test_route_prefix_K_equals_k_takes_whole_prefix():
    a = _logits(8, 12, 8)
    idx, _ = O.route_prefix(a, 3, 3)
    assert all(sorted(r) == [0, 1, 2] for r in idx.tolist())


# ---------------------------------------------------------------- prefix margin (near-tie rule)

def test_prefix_margin_closed_forms():
    # prefix [0, 5) sorted is 5, 4, 3, 2, 1: the gap between the 2nd and 3rd is
    # 4 - 3; the 100 at index 5 lies outside the prefix and must be ignored
    a = np.array([[5.0, 1.0, 3.0, 2.0, 4.0, 100.0, -7.0]])
    assert O.prefix_margin(a, 5, 2)[0] == 1.0
    assert O.prefix_margin(a, 5, 1)[0] == 1.0   # 5 - 4
    assert O.prefix_margin(a, 5, 4)[0] == 1.0   # 2 - 1
    assert O.prefix_margin(a, 7, 1)[0] == 95.0  # full span: 100 - 5
    assert O.prefix_margin(a, 6, 2)[0] == 1.0   # 100, 5 | 4: 5 - 4
    # an exact tie at the boundary gives 0; ties above it do not matter
    t = np.array([[2.0, 1.0, 1.0, 0.0], [3.0, 3.0, 1.0, 0.0]])
    np.testing.assert_array_equal(O.prefix_margin(t, 4, 2), [0.0, 2.0])
    # K == k: the whole prefix is selected, nothing can swap in
    assert np.isinf(O.prefix_margin(a, 3, 3)).all()
    # one value per row is returned, in row order
    assert O.prefix_margin(np.zeros((0, 6)), 4, 2).shape == (0,)


def test_prefix_margin_bruteforce_best_subset():
    # the margin is min over the best k-subset minus max over the rest of the
    # prefix; the best subset comes from enumerating all k-subsets
    for seed in range(40):
        r = np.random.default_rng(500 + seed)
        E = int(r.integers(3, 9))
        K = int(r.integers(1, E + 1))
        k = int(r.integers(1, K + 1))
        row = r.standard_normal(E)
        if seed % 5 == 0:
            row = np.round(row * 2) / 2  # coarse grid: frequent exact ties
        got = O.prefix_margin(row[None, :], K, k)[0]
        if K == k:
            assert np.isinf(got)
            continue
        pre = [float(v) for v in row[:K]]
        best = max(itertools.combinations(range(K), k), key=lambda S: sum(pre[e] for e in S))
        rest = [pre[e] for e in range(K) if e not in best]
        assert got == min(pre[e] for e in best) - max(rest)
        srt = sorted(pre)
        assert got == srt[-k] - srt[-k - 1]


def test_prefix_margin_decides_stability_of_the_routed_set():
    # perturbing every prefix logit by less than half the margin leaves the
    # prefix top-k set unchanged; moving the k-th down and the (k+1)-th up by
    # a little more than half swaps them
    for seed in range(30):
        a = _logits(1, 16, 900 + seed).astype(np.float64)
        K, k = 12, 4
        m = O.prefix_margin(a, K, k)[0]
        S = set(O.route_prefix(a, K, k)[0][0].tolist())
        r = np.random.default_rng(seed)
        noise = r.uniform(-0.49, 0.49, a.shape) * m
        assert set(O.route_prefix(a + noise, K, k)[0][0].tolist()) == S
        order = np.argsort(-a[0, :K], kind="stable")
        b = a.copy()
        b[0, order[k - 1]] -= 0.51 * m
        b[0, order[k]] += 0.51 * m
        S2 = set(O.route_prefix(b, K, k)[0][0].tolist())
        assert S2 != S and int(order[k]) in S2 and int(order[k - 1]) not in S2


# ---------------------------------------------------------------- dispatch

def test_dispatch_is_stable_sort_by_expert():
    for seed in range(10):
        r = np.random.default_rng(seed)
        T, k, K = int(r.integers(1, 60)), int(r.integers(1, 5)), int(r.integers(1, 9))
        idx = r.integers(0, K, size=(T, k))
        counts, offsets, perm_token, inv_slot = O.dispatch(idx, K)
        order = np.argsort(idx.reshape(-1), kind="stable")
        assert np.array_equal(perm_token, order // k)
        assert counts.sum() == T * k and offsets[-1] == T * k and offsets[0] == 0
        assert np.array_equal(np.bincount(idx.reshape(-1), minlength=K), counts)
        assert np.array_equal(inv_slot[order], np.arange(T * k))
        assert sorted(inv_slot.tolist()) == list(range(T * k))
        # within one expert, rows follow increasing flat index
        for e in range(K):
            fl = order[offsets[e]:offsets[e + 1]]
            assert (np.diff(fl) > 0).all() and (idx.reshape(-1)[fl] == e).all()


def test_dispatch_empty_and_single_expert():
    counts, offsets, perm, inv = O.dispatch(np.zeros((0, 2), np.int64), 4)
    assert counts.tolist() == [0, 0, 0, 0] and offsets.tolist() == [0] * 5 and len(perm) == 0
    counts, offsets, perm, inv = O.dispatch(np.full((5, 1), 2), 3)
    assert counts.tolist() == [0, 0, 5] and perm.tolist() == [0, 1, 2, 3, 4]


# ---------------------------------------------------------------- expert FFN + combine

def _tiny_layer(seed, T=9, d=6, m=5, E=6):
    r = np.random.default_rng(seed)
    x = r.standard_normal((T, d))
    wg = r.standard_normal((E, m, d)) * 0.5
    wu = r.standard_normal((E, m, d)) * 0.5
    wd = r.standard_normal((E, d, m)) * 0.5
    return x, wg, wu, wd


def test_silu_closed_forms():
    assert O.silu(0.0) == 0.0
    assert O.silu(1.0) == pytest.approx(1.0 / (1.0 + math.exp(-1.0)), rel=1e-15)
    assert O.silu(-40.0) == pytest.approx(-40.0 * math.exp(-40.0), rel=1e-9)
    np.testing.assert_allclose(O.silu(np.array([3.0])), torch.nn.functional.silu(
        torch.tensor([3.0], dtype=torch.float64)).numpy(), rtol=1e-15)


def test_layer_matches_dense_equivalent_formulation():
    # Appendix "Dense-equivalent expert convention": run every retained expert
    # on every token, then apply the sparse routing weights. It must equal the
    # sparse grouped computation.
    for seed in range(4):
        x, wg, wu, wd = _tiny_layer(seed)
        T, E, k, K = x.shape[0], wg.shape[0], 2, 4
        a = _logits(T, E, 50 + seed)
        idx, w = O.route_prefix(a, K, k)
        counts, offsets, perm, inv = O.dispatch(idx, K)
        y = O.expert_swiglu(x[perm], offsets, wg, wu, wd)
        out = O.combine(y, inv, w)
        xt = torch.from_numpy(x)
        dense = torch.stack([
            torch.nn.functional.linear(
                torch.nn.functional.silu(torch.nn.functional.linear(xt, torch.from_numpy(wg[e])))
                * torch.nn.functional.linear(xt, torch.from_numpy(wu[e])),
                torch.from_numpy(wd[e]))
            for e in range(K)])                                    # [K, T, d]
        Wsp = torch.zeros(T, K, dtype=torch.float64)
        Wsp.scatter_(1, torch.from_numpy(idx), torch.from_numpy(w))
        ref = torch.einsum("tk,ktd->td", Wsp, dense).numpy()
        np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-12)


def test_expert_swiglu_diagonal_closed_form():
    d = m = 4
    al, be, ga = 0.7, -1.3, 2.0
    wg = np.stack([al * np.eye(d)] * 2)
    wu = np.stack([be * np.eye(d)] * 2)
    wd = np.stack([ga * np.eye(d)] * 2)
    x = np.array([[1.0, -2.0, 0.5, 0.0], [3.0, 0.25, -1.0, 2.0]])
    y = O.expert_swiglu(x, np.array([0, 1, 2]), wg, wu, wd)
    z = al * x
    np.testing.assert_allclose(y, ga * (z / (1 + np.exp(-z))) * (be * x), rtol=1e-14)


def test_combine_single_slot_and_residual():
    y = np.arange(12.0).reshape(4, 3)
    inv = np.array([2, 0, 3, 1])
    w = np.ones((4, 1))
    res = np.full((4, 3), 0.5)
    out = O.combine(y, inv, w, res)
    np.testing.assert_array_equal(out, y[[2, 0, 3, 1]] + 0.5)


def test_full_span_layer_matches_textbook_moe_torch():
    # K = E reduces to the ordinary top-k MoE (reordering only permutes storage)
    x, wg, wu, wd = _tiny_layer(7, T=11, E=5)
    r = np.random.default_rng(3)
    w_r = r.standard_normal((5, x.shape[1])).astype(np.float32)
    b = np.linspace(0.5, -0.5, 5).astype(np.float32)
    x32 = x.astype(np.float32)
    res = O.moe_layer(x32, w_r, b, wg, wu, wd, k=2, K=5)
    xt = torch.from_numpy(x32.astype(np.float64))
    logits = (xt @ torch.from_numpy(w_r.astype(np.float64)).T + torch.from_numpy(b.astype(np.float64))).float()
    prob = torch.softmax(logits.double(), -1)
    tv, ti = torch.topk(prob, 2, -1)
    tw = tv / tv.sum(-1, keepdim=True)
    ref = torch.zeros_like(xt)
    for t in range(xt.shape[0]):
        for j in range(2):
            e = int(ti[t, j])
            h = torch.nn.functional.silu(torch.from_numpy(wg[e]) @ xt[t]) * (torch.from_numpy(wu[e]) @ xt[t])
            ref[t] += tw[t, j] * (torch.from_numpy(wd[e]) @ h)
    np.testing.assert_allclose(res["out"], ref.numpy(), rtol=1e-12, atol=1e-12)


def test_moe_token_equals_layer_rows():
    x, wg, wu, wd = _tiny_layer(9, T=7, E=6)
    a = _logits(7, 6, 77)
    idx, w = O.route_prefix(a, 4, 2)
    counts, offsets, perm, inv = O.dispatch(idx, 4)
    out = O.combine(O.expert_swiglu(x[perm], offsets, wg, wu, wd), inv, w)
    for t in range(7):
        o, _, _ = O.moe_token(x[t], a[t], wg, wu, wd, 4, 2)
        np.testing.assert_allclose(o, out[t], rtol=1e-12, atol=1e-13)


def test_adaptive_K_path_uses_select_prefix():
    x, wg, wu, wd = _tiny_layer(2, T=20, E=6)
    r = np.random.default_rng(1)
    w_r = r.standard_normal((6, x.shape[1])).astype(np.float32)
    b = (-1.1 * np.log(np.arange(6) + 1.0)).astype(np.float32)
    res = O.moe_layer(x.astype(np.float32), w_r, b, wg, wu, wd, k=2, p=0.7)
    a = O.router_logits(x.astype(np.float32), w_r, b)
    assert res["K"] == _select_bruteforce(list(O.activated_mass(a, 2)), 0.7, 2)


# ---------------------------------------------------------------- SAVB removal

def test_drop_visual_block_keeps_text_rows_in_order():
    rows = np.arange(40).reshape(10, 4)
    out = O.drop_visual_block(rows, 3, 4)
    np.testing.assert_array_equal(out, np.delete(rows, np.s_[3:7], axis=0))
    assert out.shape[0] == 6
    np.testing.assert_array_equal(O.drop_visual_block(rows, 5, 0), rows)
    np.testing.assert_array_equal(O.drop_visual_block(rows, 0, 10), rows[:0])
    np.testing.assert_array_equal(O.drop_visual_block(rows, 0, 3), rows[3:])
    np.testing.assert_array_equal(O.drop_visual_block(rows, 7, 3), rows[:7])


# ---------------------------------------------------------------- stack

def test_rmsnorm_closed_form():
    x = np.full((1, 8), -3.0)
    np.testing.assert_allclose(O.rmsnorm(x, eps=0.0), -np.ones((1, 8)), rtol=1e-15)
    y = O.rmsnorm(np.array([[3.0, 4.0]]), eps=0.0)
    np.testing.assert_allclose(y, [[3.0 / math.sqrt(12.5), 4.0 / math.sqrt(12.5)]], rtol=1e-15)


def test_stack_one_layer_is_residual_moe():
    x, wg, wu, wd = _tiny_layer(5, T=4, E=6)
    r = np.random.default_rng(2)
    w_r = r.standard_normal((6, x.shape[1])).astype(np.float32)
    b = np.zeros(6, np.float32)
    layer = dict(w_r=w_r, bias=b, w_gate=wg, w_up=wu, w_down=wd)
    for t in range(4):
        h, _ = O.stack_token(x[t], [layer], [4], 2)
        xn = O.rmsnorm(x[t:t + 1])
        ref = O.moe_layer(xn, w_r, b, wg, wu, wd, k=2, K=4)["out"][0] + x[t]
        np.testing.assert_allclose(h, ref, rtol=1e-13, atol=1e-13)


# ---------------------------------------------------------------- calibration (Eqs. 8-9)

def test_text_routed_mass_closed_form_and_sum():
    # token 0 ties its top 2 at 3.0 (weights 1/2, 1/2); token 1 picks experts
    # 3 and 1 with logits differing by ln 3 (weights 3/4, 1/4)
    a = np.array([[3.0, -9.0, 3.0, -9.0, -9.0],
                  [-9.0, 1.0, -9.0, 1.0 + math.log(3.0), -9.0]], dtype=np.float32)
    M = O.text_routed_mass(a, 2)
    w1 = math.exp(float(np.float32(1.0))) / (math.exp(float(np.float32(1.0))) + math.exp(float(a[1, 3])))
    expect = np.array([0.25, w1 / 2, 0.25, (1 - w1) / 2, 0.0])
    assert np.allclose(M, expect, rtol=0, atol=1e-15)
    r = np.random.default_rng(3)
    for n, E, k in ((1, 16, 2), (37, 128, 8), (200, 64, 4)):
        M = O.text_routed_mass(r.standard_normal((n, E)).astype(np.float32), k)
        assert abs(M.sum() - 1.0) < 1e-12 and (M >= 0).all()
        assert (M > 0).sum() <= min(E, n * k)


def test_mean_mass_order_ties_and_case_weighting():
    # case means: e0 (0.1+0.3)/2 = 0.2, e1 0.4, e2 0.2, e3 0.2 -> ties keep index order
    M = np.array([[0.1, 0.5, 0.2, 0.2], [0.3, 0.3, 0.2, 0.2]])
    pi, mean = O.mean_mass_order(M)
    assert pi.tolist() == [1, 0, 2, 3]
    assert np.allclose(mean, [0.2, 0.4, 0.2, 0.2])
    # every case counts once, however many tokens it had: duplicating the
    # cases leaves the order unchanged
    pi2, _ = O.mean_mass_order(np.concatenate([M, M]))
    assert pi2.tolist() == pi.tolist()


def test_mean_mass_order_maximises_every_prefix_bruteforce():
    # the sorted order puts the largest total mean mass into every prefix
    r = np.random.default_rng(11)
    M = r.dirichlet(np.ones(6), size=5)
    pi, mean = O.mean_mass_order(M)
    for K in range(1, 7):
        best = max(sum(mean[list(c)]) for c in itertools.combinations(range(6), K))
        assert abs(sum(mean[pi[:K]]) - best) < 1e-15
    assert sorted(pi.tolist()) == list(range(6))


def _calib_layer(seed, E=6, d=8, m=4):
    r = np.random.default_rng(seed)
    return dict(w_r=r.standard_normal((E, d)) * 0.5, bias=r.standard_normal(E) * 0.3,
                w_gate=r.standard_normal((E, m, d)) * 0.3, w_up=r.standard_normal((E, m, d)) * 0.3,
                w_down=r.standard_normal((E, d, m)) * 0.3)


def test_reorder_is_identity_on_unsliced_layer():
    # Section 3.3 / Appendix: the permutation of router rows and expert tensors
    # changes only the storage order; with every expert kept (K = E) the layer
    # output is unchanged
    L = _calib_layer(5)
    x = np.random.default_rng(6).standard_normal((9, 8))
    pi = np.array([4, 0, 5, 2, 1, 3])
    w_r, b, wg, wu, wd = O.apply_expert_order(pi, L["w_r"], L["bias"], L["w_gate"], L["w_up"], L["w_down"])
    ref = O.moe_layer(x, L["w_r"], L["bias"], L["w_gate"], L["w_up"], L["w_down"], k=2, K=6)["out"]
    got = O.moe_layer(x, w_r, b, wg, wu, wd, k=2, K=6)["out"]
    assert np.allclose(got, ref, rtol=0, atol=1e-12)
    # a mistake in one tensor (gate/up permuted, down not) breaks it
    bad = O.moe_layer(x, w_r, b, wg, wu, L["w_down"], k=2, K=6)["out"]
    assert np.abs(bad - ref).max() > 1e-3


def test_reorder_by_calibrated_order_sorts_the_calibration_mass():
    # after applying pi, recomputing the cases' routed mass gives experts in
    # non-increasing mean mass: the leading positions form the mass prefix
    L = _calib_layer(8, E=6)
    r = np.random.default_rng(9)
    cases = [r.standard_normal((int(n), 8)) for n in (3, 11, 6)]
    Ms = [O.text_routed_mass(O.router_logits(c, L["w_r"], L["bias"]), 2) for c in cases]
    pi, mean = O.mean_mass_order(np.stack(Ms))
    w_r, b, _, _, _ = O.apply_expert_order(pi, L["w_r"], L["bias"], L["w_gate"], L["w_up"], L["w_down"])
    Ms2 = [O.text_routed_mass(O.router_logits(c, w_r, b), 2) for c in cases]
    _, mean2 = O.mean_mass_order(np.stack(Ms2))
    assert np.allclose(mean2, mean[pi], rtol=0, atol=1e-12)
    assert (np.diff(mean2) <= 1e-15).all()


# ---------------------------------------------------------------- SAVB gate (Eqs. 2-3)

def test_candidate_layers_every_fourth_from_three():
    assert O.candidate_layers(48) == [3 + 4 * i for i in range(12)]
    assert O.candidate_layers(48)[-1] == 47 and 19 in O.candidate_layers(48)


def test_gate_feature_pooling_closed_forms():
    h = np.arange(7 * 3, dtype=np.float64).reshape(7, 3)
    # visual rows 1..3 removed: text rows 0, 4, 5, 6; pooled over 0, 4, 5; last = 6
    x = O.gate_feature(h, 1, 3)
    assert np.allclose(x[:3], (h[0] + h[4] + h[5]) / 3) and np.array_equal(x[3:], h[6])
    # n = 2: the pooled half is the first text row itself
    x2 = O.gate_feature(h[:2], 0, 0)
    assert np.array_equal(x2, np.concatenate([h[0], h[1]]))
    # one text row: pooled half zero
    assert np.array_equal(O.gate_feature(h[:3], 0, 2), np.concatenate([np.zeros(3), h[2]]))
    # the pooled half does not depend on the order of the preceding text rows
    perm = h[[5, 0, 4, 6]]
    assert np.allclose(O.gate_feature(perm, 0, 0)[:3], x[:3])


def test_gate_mlp_closed_form_sigmoid():
    # W1 picks x0 and -x0 through the ReLU, W2 subtracts them: z = [0, x0],
    # so p_exit = softmax(z)_1 = 1 / (1 + exp(-x0))
    w1 = np.zeros((2, 4)); w1[0, 0] = 1.0; w1[1, 0] = -1.0
    w2 = np.array([[0.0, 0.0], [1.0, -1.0]])
    for x0 in (-3.0, -0.5, 0.0, 0.7, 4.0):
        x = np.array([x0, 9.0, -2.0, 1.0])
        z = O.gate_logits(x, w1, np.zeros(2), w2, np.zeros(2))
        assert np.allclose(z, [0.0, x0])
        assert abs(O.gate_exit_prob(z) - 1.0 / (1.0 + math.exp(-x0))) < 1e-15
    assert O.gate_decision(0.5, 0.5) and not O.gate_decision(0.4999, 0.5)
    # the hidden layer really is rectified: a negative pre-activation is dropped
    z = O.gate_logits(np.array([-1.0, 0, 0, 0]), np.array([[1.0, 0, 0, 0]]), np.zeros(1),
                      np.array([[0.0], [5.0]]), np.array([0.25, 0.0]))
    assert np.allclose(z, [0.25, 0.0])


# ---------------------------------------------------------------- attention on the compacted sequence

def test_attention_single_key_returns_its_value():
    r = np.random.default_rng(3)
    q = r.standard_normal((1, 4, 8))
    k = r.standard_normal((1, 2, 8))
    v = r.standard_normal((1, 2, 8))
    out = O.attention(q, k, v)
    for h in range(4):
        np.testing.assert_allclose(out[0, h], v[0, h // 2], rtol=0, atol=1e-15)


def test_attention_two_keys_closed_form_and_equal_keys_mean():
    r = np.random.default_rng(4)
    D = 16
    q = r.standard_normal((1, 1, D))
    k = r.standard_normal((2, 1, D))
    v = r.standard_normal((2, 1, D))
    s0, s1 = (float(k[j, 0] @ q[0, 0]) / np.sqrt(D) for j in range(2))
    w1 = 1.0 / (1.0 + math.exp(s0 - s1))
    np.testing.assert_allclose(O.attention(q, k, v)[0, 0], (1 - w1) * v[0, 0] + w1 * v[1, 0], rtol=1e-13)
    # identical keys: every visible key weighs the same (the mean of the values)
    k_same = np.repeat(k[:1], 5, axis=0)
    v5 = r.standard_normal((5, 1, D))
    np.testing.assert_allclose(O.attention(q, k_same, v5)[0, 0], v5[:, 0].mean(0), rtol=1e-13)


def test_attention_matches_torch_sdpa_with_grouped_heads():
    # prefill (n = C, causal) and a decode step (n < C) against torch's
    # scaled_dot_product_attention with the KV heads repeated per group and
    # the visibility written as a mask
    r = np.random.default_rng(5)
    for (n, C, Hq, Hkv, D) in ((7, 7, 8, 2, 16), (1, 9, 4, 1, 8), (3, 11, 6, 3, 32)):
        q = r.standard_normal((n, Hq, D))
        k = r.standard_normal((C, Hkv, D))
        v = r.standard_normal((C, Hkv, D))
        got = O.attention(q, k, v)
        g = Hq // Hkv
        qt = torch.from_numpy(q).permute(1, 0, 2)                      # [Hq, n, D]
        kt = torch.from_numpy(k).permute(1, 0, 2).repeat_interleave(g, 0)
        vt = torch.from_numpy(v).permute(1, 0, 2).repeat_interleave(g, 0)
        mask = torch.tensor([[j <= C - n + i for j in range(C)] for i in range(n)])
        ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, attn_mask=mask)
        np.testing.assert_allclose(got, ref.permute(1, 0, 2).numpy(), rtol=1e-12, atol=1e-12)


def test_attention_on_compacted_sequence_equals_masking_the_visual_keys():
    # removing the visual block [v0, v0 + nv) from the keys and values (the
    # SAVB exit) gives each text query the same output as attending over the
    # full sequence with the visual keys hidden: the removal changes the work,
    # not what text tokens see
    r = np.random.default_rng(6)
    S, v0, nv, Hq, Hkv, D = 20, 3, 11, 4, 2, 16
    x_q = r.standard_normal((S, Hq, D))
    k = r.standard_normal((S, Hkv, D))
    v = r.standard_normal((S, Hkv, D))
    text = [i for i in range(S) if not (v0 <= i < v0 + nv)]
    comp = O.attention(x_q[text], O.drop_visual_block(k, v0, nv), O.drop_visual_block(v, v0, nv))
    # brute force on the full sequence: causal, visual keys excluded
    for a, i in enumerate(text):
        for h in range(Hq):
            vis = [j for j in text if j <= i]
            s = np.array([k[j, h // 2] @ x_q[i, h] for j in vis]) / np.sqrt(D)
            w = np.exp(s - s.max())
            w /= w.sum()
            np.testing.assert_allclose(comp[a, h], w @ v[vis, h // 2], rtol=1e-12, atol=1e-12)


def test_attention_decode_step_equals_last_row_of_prefill():
    # the decode step over the cache gives what the prefill gives its last rows
    r = np.random.default_rng(8)
    C, Hq, Hkv, D = 13, 4, 2, 8
    q = r.standard_normal((C, Hq, D))
    k = r.standard_normal((C, Hkv, D))
    v = r.standard_normal((C, Hkv, D))
    full = O.attention(q, k, v)
    np.testing.assert_allclose(O.attention(q[-2:], k, v), full[-2:], rtol=1e-13, atol=1e-14)
