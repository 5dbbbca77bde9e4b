"""CPU oracle of the DecoMoE prefix-restricted MoE layer, its offline Mean-Mass
expert calibration, the SAVB exit gate and visual-block removal.

TEST INFRASTRUCTURE ONLY. This module is the plain, slow, obviously-correct
statement of what the DecoMoE paper's method computes, in float64 with numpy.
Only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline and
reference legs of ``bench.py`` may import it. The library (the CUDA path under
``paper_2609_38823_gb300``) never imports, calls or links anything here, and
nothing here imports the library.

Each function cites the paper passage it follows (section / equation /
algorithm). Where the paper is silent the reading taken is stated in the
docstring. Library primitives used as steps: numpy matmul (fp64), exp, argsort.

Pins (tests/test_oracle_pins.py) tie every function to something other than
itself: brute force on tiny inputs, the textbook top-k MoE routine (torch CPU)
for the full-span special case, closed forms, invariants the paper states.
The absolute values of a layer output have no worked example in the paper;
they are pinned through the dense-equivalent formulation (Appendix, "Dense-
equivalent expert convention") and brute-force per-row loops, not by printed
numbers.
"""
from __future__ import annotations

import numpy as np

F64 = np.float64


# ---------------------------------------------------------------------------
# Router (Section 3.1, Eq. 1)
# ---------------------------------------------------------------------------

def router_logits(x, w_r, bias=None):
    """Router logits a_{i,e} over the whole (reordered) expert pool.

    Section 3.1 defines rho = softmax(a) from router logits a; the logits are the
    token's hidden state times each router row. The per-expert ``bias`` is part
    of the synthetic workload recipe (it sets the routed-mass skew over the
    reordered index). Accumulated in float64, then rounded once to float32:
    routing decisions on both sides of the parity tests are taken on float32
    logits.
    """
    a = np.asarray(x, F64) @ np.asarray(w_r, F64).T
    if bias is not None:
        a = a + np.asarray(bias, F64)[None, :]
    return a.astype(np.float32)


def softmax(v):
    """Row softmax (Eq. 1) in float64: exp(v - max) / sum exp(v - max)."""
    v = np.asarray(v, F64)
    z = v - v.max(axis=-1, keepdims=True)
    e = np.exp(z)
    return e / e.sum(axis=-1, keepdims=True)


def topk(values, k):
    """TopK of Eqs. 7 and 10: indices of the k largest entries of each row.

    Order inside the result is by value, largest first. The paper does not say
    how equal values are ordered; equal values are taken lower index first.
    """
    v = np.asarray(values)
    order = np.argsort(-v, axis=-1, kind="stable")
    return order[..., :k].astype(np.int64)


# ---------------------------------------------------------------------------
# RCEP runtime: full-pool top-k, activated mass, prefix length (Section 3.3)
# ---------------------------------------------------------------------------

def full_pool_route(a, k):
    """Eq. 10 and the renormalised weight inside Eq. 11.

    q = softmax over all E reordered experts, R_i = TopK(q_i, k), and each
    selected expert's weight is q_e / sum_{e' in R_i} q_e'. Ranking by q equals
    ranking by the logits, because softmax is strictly increasing in each logit
    for a fixed row; the ranking is taken on the float32 logits so both sides
    of a parity test decide in the same precision.
    Returns (R [T,k] int64, w [T,k] float64).
    """
    a = np.asarray(a)
    q = softmax(a)
    R = topk(a, k)
    qs = np.take_along_axis(q, R, axis=-1)
    w = qs / qs.sum(axis=-1, keepdims=True)
    return R, w


def activated_mass(a, k):
    """Eq. 11: s_e = sum over tokens of the invocation of the renormalised
    full-pool top-k weight of expert e (zero where e is not in R_i).

    Summed in token order, in float64. Returns s [E] float64.
    """
    a = np.asarray(a)
    T, E = a.shape
    R, w = full_pool_route(a, k)
    s = np.zeros(E, F64)
    for i in range(T):
        for j in range(k):
            s[R[i, j]] += w[i, j]
    return s


def select_prefix(s, p, k):
    """Eq. 12: K_hat = min{K in 1..E : sum_{e<K} s_e / sum_e s_e >= p};
    K = max(k, K_hat).

    Readings where the paper is silent:
      * sums run in expert order e = 0..E-1, sequentially, in float64; the
        total is the last partial sum;
      * p >= 1 gives K_hat = E (the paper's sweep reports a prefix of 128.0 of
        128 at p = 1.0);
      * if the ratio never reaches p (rounding) K_hat = E;
      * an empty invocation (total mass 0) gives K = k.
    """
    s = np.asarray(s, F64)
    E = s.shape[0]
    if not (0.0 < p <= 1.0):
        raise ValueError("p must lie in (0, 1]")
    if k > E:
        raise ValueError("k > E")
    cum = []
    acc = 0.0
    for e in range(E):
        acc = acc + float(s[e])
        cum.append(acc)
    tot = cum[-1]
    if tot <= 0.0:
        return int(k)
    if p >= 1.0:
        K_hat = E
    else:
        K_hat = E
        for K in range(1, E + 1):
            if cum[K - 1] / tot >= p:
                K_hat = K
                break
    return int(max(k, K_hat))


def route_prefix(a, K, k):
    """Prefix-restricted routing (Section 3.3, last paragraph; Algorithm 2).

    Slice the logits to the first K reordered experts, take a new softmax over
    that prefix, rerun TopK(k) inside the prefix and renormalise the selected
    weights. The full-pool top-k set is never intersected with the prefix.
    Slot j of a token holds its j-th largest prefix logit.
    Returns (idx [T,k] int64 in [0,K), w [T,k] float64).
    """
    a = np.asarray(a)
    E = a.shape[-1]
    if not (k <= K <= E):
        raise ValueError("need k <= K <= E")
    ap = a[:, :K]
    q_tilde = softmax(ap)
    idx = topk(ap, k)
    qs = np.take_along_axis(q_tilde, idx, axis=-1)
    w = qs / qs.sum(axis=-1, keepdims=True)
    return idx, w


def prefix_margin(a, K, k):
    """Gap between the k-th and (k+1)-th largest logit inside [0,K) per token
    (+inf when K == k). Tokens with a gap below a tolerance are reported and
    left out of index-exact comparisons."""
    ap = np.asarray(a, F64)[:, :K]
    if K <= k:
        return np.full(ap.shape[0], np.inf)
    srt = -np.sort(-ap, axis=-1)
    return srt[:, k - 1] - srt[:, k]


# ---------------------------------------------------------------------------
# Dispatch, expert FFN, combine (Algorithm 2: "evaluate and combine only the
# first K physically contiguous expert MLPs")
# ---------------------------------------------------------------------------

def dispatch(idx, K):
    """Group the T*k (token, slot) pairs by expert.

    counts[e] = number of pairs routed to expert e (e < K); offsets is its
    exclusive prefix sum (length K+1). Pairs are ordered by expert id, and
    within one expert by the flat index f = t*k + j (a stable sort).
    perm_token[r] = token of row r of the grouped order; inv_slot[f] = row r
    holding pair f.
    """
    idx = np.asarray(idx, np.int64)
    T, k = idx.shape
    flat = idx.reshape(-1)
    counts = np.zeros(K, np.int64)
    for e in flat:
        counts[e] += 1
    offsets = np.zeros(K + 1, np.int64)
    for e in range(K):
        offsets[e + 1] = offsets[e] + counts[e]
    order = sorted(range(T * k), key=lambda f: (flat[f], f))
    perm_token = np.array([f // k for f in order], np.int64)
    inv_slot = np.empty(T * k, np.int64)
    for r, f in enumerate(order):
        inv_slot[f] = r
    return counts, offsets, perm_token, inv_slot


def silu(z):
    """SiLU z * sigmoid(z) = z / (1 + exp(-z)) (float64)."""
    z = np.asarray(z, F64)
    return z / (1.0 + np.exp(-z))


def expert_swiglu(x_rows, offsets, w_gate, w_up, w_down):
    """Expert MLP on grouped rows: for every row r of expert e,
    h = silu(W_gate[e] x_r) * (W_up[e] x_r), y_r = W_down[e] h.

    The paper names gate, up and down projections (Algorithm 1) and counts
    three matmuls per expert (Appendix, C_expert = 6Kdm); the activation is
    SwiGLU. Everything in float64; h is not rounded.
    """
    x_rows = np.asarray(x_rows, F64)
    R, d = x_rows.shape
    K = len(offsets) - 1
    y = np.zeros((R, d), F64)  # the down projection maps back to width d
    for e in range(K):
        r0, r1 = int(offsets[e]), int(offsets[e + 1])
        if r1 == r0:
            continue
        xe = x_rows[r0:r1]
        g = xe @ np.asarray(w_gate[e], F64).T
        u = xe @ np.asarray(w_up[e], F64).T
        h = silu(g) * u
        y[r0:r1] = h @ np.asarray(w_down[e], F64).T
    return y


def combine(y_rows, inv_slot, w, residual=None):
    """out_t = sum_j w[t,j] * y[inv_slot[t*k+j]] (+ residual_t), slot order
    j = 0..k-1, float64."""
    y_rows = np.asarray(y_rows, F64)
    w = np.asarray(w, F64)
    T, k = w.shape
    out = np.zeros((T, y_rows.shape[1]), F64)
    for j in range(k):
        out += w[:, j:j + 1] * y_rows[np.asarray(inv_slot)[np.arange(T) * k + j]]
    if residual is not None:
        out += np.asarray(residual, F64)
    return out


def moe_layer(x, w_r, bias, w_gate, w_up, w_down, k, K=None, p=None, residual=None):
    """One RCEP MoE invocation (Algorithm 2, exited branch; Eqs. 10-12).

    Either a fixed prefix K is given, or a mass target p from which K is
    selected (full-pool route -> activated mass -> shortest covering prefix).
    Returns a dict with every intermediate.
    """
    a = router_logits(x, w_r, bias)
    E = a.shape[1]
    res = {"logits": a}
    if K is None:
        s = activated_mass(a, k)
        K = select_prefix(s, p, k)
        res["mass"] = s
    res["K"] = int(K)
    idx, w = route_prefix(a, K, k)
    counts, offsets, perm_token, inv_slot = dispatch(idx, K)
    x_rows = np.asarray(x, F64)[perm_token]
    y = expert_swiglu(x_rows, offsets, w_gate, w_up, w_down)
    out = combine(y, inv_slot, w, residual)
    res.update(idx=idx, w=w, counts=counts, offsets=offsets, perm_token=perm_token,
               inv_slot=inv_slot, y=y, out=out, E=E)
    return res


def moe_token(x_t, a_t, w_gate, w_up, w_down, K, k):
    """Layer output of ONE token given its logits and the prefix K (tokens are
    independent once K is fixed). Used for sampled checks at full size."""
    idx, w = route_prefix(np.asarray(a_t)[None, :], K, k)
    x_t = np.asarray(x_t, F64)
    out = np.zeros(x_t.shape[0], F64)
    for j in range(k):
        e = int(idx[0, j])
        g = np.asarray(w_gate[e], F64) @ x_t
        u = np.asarray(w_up[e], F64) @ x_t
        out += w[0, j] * (np.asarray(w_down[e], F64) @ (silu(g) * u))
    return out, idx[0], w[0]


# ---------------------------------------------------------------------------
# RCEP offline calibration: text-token routed mass and the Mean-Mass expert
# order (Section 3.3, Eqs. 8-9; Algorithm 1, last two loops; Appendix, "RCEP
# Calibration and Text-Routing Alignment")
# ---------------------------------------------------------------------------

def text_routed_mass(a_text, k):
    """Eq. 9: M_{c,l,e} = (1/|T|) * sum over the case's text tokens i of the
    renormalised full-pool top-k weight of expert e (rho_e / sum of rho over
    the k selected experts; zero where e is not selected).

    ``a_text``: float32 router logits [n, E] of the case's text tokens at one
    layer (n >= 1). The top-k sets and weights are those of Eq. 10 / Eq. 11
    (full_pool_route), summed in token order in float64, then divided by n.
    Returns M [E] float64 (it sums to 1 up to rounding).
    """
    a_text = np.asarray(a_text)
    n = a_text.shape[0]
    if n < 1:
        raise ValueError("a case needs at least one text token")
    return activated_mass(a_text, k) / F64(n)


def mean_mass_order(case_masses):
    """Eq. 8: pi_l = argsort over experts of the case-mean routed mass,
    descending. The Appendix averages within a case first (Eq. 9) and then
    across cases, so every case has equal weight.

    Reading where the paper is silent: equal means keep ascending expert index
    (a stable sort), so pi is unique. The mean is the float64 sum over cases in
    their given order divided by the case count.
    ``case_masses``: [C, E]. Returns (pi [E] int64, mean [E] float64): new
    expert position i holds original expert pi[i].
    """
    M = np.asarray(case_masses, F64)
    C, E = M.shape
    if C < 1:
        raise ValueError("need at least one calibration case")
    tot = np.zeros(E, F64)
    for c in range(C):
        tot = tot + M[c]
    mean = tot / F64(C)
    pi = np.argsort(-mean, kind="stable")
    return pi.astype(np.int64), mean


def apply_expert_order(pi, w_r, bias, w_gate, w_up, w_down):
    """Algorithm 1, last loop; Section 3.3 after Eq. 8: the same permutation
    applied to the router output rows (and the per-expert router bias of the
    synthetic workload) and to the gate/up and down tensors of the experts.
    Only the storage order changes. Returns the reordered copies."""
    pi = np.asarray(pi, np.int64)
    return (np.asarray(w_r)[pi], None if bias is None else np.asarray(bias)[pi], np.asarray(w_gate)[pi],
            np.asarray(w_up)[pi], np.asarray(w_down)[pi])


# ---------------------------------------------------------------------------
# SAVB gate (Section 3.2, Eqs. 2-3; Appendix, "SAVB Supervision")
# ---------------------------------------------------------------------------

def candidate_layers(n_layers, first=3, step=4):
    """The sparse candidate set G = {3, 7, 11, ...} (zero-based layer indices,
    Appendix "Offline Calibration"), every fourth decoder layer."""
    return list(range(first, n_layers, step))


def gate_feature(h, v0, nv):
    """Eq. 2: x = [mean of text states 1..n-1 ; text state n] in R^{2d}.

    Reading: the text tokens are the rows outside the contiguous visual block
    [v0, v0+nv), in sequence order (system-prompt rows before the block and the
    text after it). With a single text row the pooled half is zero. Float64.
    """
    T = drop_visual_block(np.asarray(h, F64), v0, nv)
    n, d = T.shape
    if n < 1:
        raise ValueError("no text rows")
    pooled = np.zeros(d, F64)
    for j in range(n - 1):
        pooled = pooled + T[j]
    if n > 1:
        pooled = pooled / F64(n - 1)
    return np.concatenate([pooled, T[n - 1]])


def gate_logits(x, w1, b1, w2, b2):
    """The two-class MLP g_phi of Eq. 3 with one hidden layer (512 wide in the
    Appendix): z = W2 relu(W1 x + b1) + b2, z in R^2.

    Reading: the paper does not name the hidden activation; ReLU is taken.
    w1: [H, 2d], b1: [H], w2: [2, H], b2: [2]. Float64.
    """
    hdn = np.asarray(w1, F64) @ np.asarray(x, F64) + np.asarray(b1, F64)
    hdn = np.maximum(hdn, 0.0)
    return np.asarray(w2, F64) @ hdn + np.asarray(b2, F64)


def gate_exit_prob(z):
    """Eq. 3: p_exit = softmax(z)_1 (class 1 is "exit")."""
    return float(softmax(np.asarray(z, F64)[None, :])[0, 1])


def gate_decision(p_exit, theta):
    """Eq. 3: Exit = [p_exit >= theta]."""
    return bool(p_exit >= theta)


# ---------------------------------------------------------------------------
# SAVB visual-block removal (Section 3.2; Algorithm 2; Appendix layer-index
# convention)
# ---------------------------------------------------------------------------

def drop_visual_block(rows, v0, nv):
    """Remove the contiguous visual block rows [v0, v0+nv) and keep every other
    row in its original order (hidden state or one layer's KV rows)."""
    rows = np.asarray(rows)
    keep = [i for i in range(rows.shape[0]) if not (v0 <= i < v0 + nv)]
    return rows[keep]


# ---------------------------------------------------------------------------
# Attention-free stack used by the 48-layer workload
# ---------------------------------------------------------------------------

def rmsnorm(x, eps=1e-6, gamma=None):
    """x / sqrt(mean(x^2) + eps) * gamma, per row (workload choice: eps=1e-6,
    gamma=1; the paper leaves norms out of the method)."""
    x = np.asarray(x, F64)
    y = x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)
    if gamma is not None:
        y = y * np.asarray(gamma, F64)
    return y


def stack_token(h_t, layers, K_sched, k, eps=1e-6, round_bf16=None):
    """Trajectory of one token through the attention-free stack
    h <- h + MoE(RMSNorm(h)) with per-layer prefix K_l. Without attention and
    with K_l given, tokens are independent, so a token can be followed alone.
    ``layers`` is a sequence of dicts with w_r, bias, w_gate, w_up, w_down.
    ``round_bf16`` optionally rounds the layer input and the stored hidden
    state to the storage precision between layers (a callable).
    Returns the final hidden state and the per-layer minimum prefix margin.
    """
    h = np.asarray(h_t, F64)
    margins = []
    for l, Lw in enumerate(layers):
        xn = rmsnorm(h[None, :], eps)
        if round_bf16 is not None:
            xn = round_bf16(xn)
        a = router_logits(xn, Lw["w_r"], Lw["bias"])
        margins.append(float(prefix_margin(a, K_sched[l], k)[0]))
        out, _, _ = moe_token(xn[0], a[0], Lw["w_gate"], Lw["w_up"], Lw["w_down"], K_sched[l], k)
        h = h + out
        if round_bf16 is not None:
            h = round_bf16(h[None, :])[0]
    return h, margins


# ---------------------------------------------------------------------------
# Self-attention on the compacted sequence and over the text-only KV cache
# (Section 3.2: once the visual block exits, attention in that layer and every
# later one runs on the shortened text-only sequence; Algorithm 2, last step:
# decoding reuses the shortened text-only cache; Appendix FLOPs: 2qS(S+1) per
# prefill layer, 4qC per decode forward with cache length C)
# ---------------------------------------------------------------------------

def attention(q, k_cache, v_cache, scale=None):
    """Causal scaled-dot-product attention with grouped KV heads.

    q: [n, Hq, D] queries of the last n positions of a sequence whose keys and
    values are k_cache, v_cache: [C, Hkv, D] (C >= n; the queries' own keys are
    the last n rows). Query i sits at position C - n + i and attends to keys
    j <= C - n + i: n = C is a prefill over the sequence, n < C a decode step
    over a cache. Query head h reads KV head h // (Hq // Hkv). The score is
    q . k * scale (scale = 1 / sqrt(D) unless given); weights are the softmax
    over the visible keys; the output is the weighted sum of their values.
    The paper does not restate attention; this is the standard causal form of
    the decoder it accelerates. Float64. Returns [n, Hq, D].
    """
    q = np.asarray(q, F64)
    k_cache = np.asarray(k_cache, F64)
    v_cache = np.asarray(v_cache, F64)
    n, Hq, D = q.shape
    C, Hkv, _ = k_cache.shape
    if not (1 <= n <= C) or Hq % Hkv != 0:
        raise ValueError("need 1 <= n <= C and Hq a multiple of Hkv")
    if scale is None:
        scale = 1.0 / np.sqrt(D)
    group = Hq // Hkv
    out = np.zeros((n, Hq, D), F64)
    for i in range(n):
        last = C - n + i  # position of query i: keys 0..last are visible
        for h in range(Hq):
            g = h // group
            s = (k_cache[:last + 1, g, :] @ q[i, h, :]) * scale
            w = softmax(s)
            out[i, h, :] = w @ v_cache[:last + 1, g, :]
    return out
