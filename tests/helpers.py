"""Shared helpers of the GPU parity tests (comparison rules and tolerances)."""
import numpy as np
import torch

from oracle import decomoe_oracle as O

# Output tolerance for bf16 storage with fp32 accumulation (stated with the
# method's parity requirements): relative L2 and max-abs relative to max|ref|.
BF16_REL_L2 = 5e-3
BF16_MAX_ABS = 2e-2
# fp32 storage (CUDA-core path): derived in the design notes from fp32
# accumulation over d=256 and m=128 terms (~sqrt(n) * 2^-24 relative).
F32_REL_L2 = 1e-5
F32_MAX_ABS = 1e-5
# Routing weights: |delta| bound on the renormalised top-k weights.
W_ABS = 1e-6
# Activated mass (Eq. 11) from fp32 per-token weights: relative error bound
# (expf <= 2 ulp, one division, renormalising sum over k <= 32 terms and the
# in-block sum of <= 8 token weights, each ~2^-24 relative), and the band
# around p inside which the prefix length is reported but not compared.
MASS_REL = 4e-6
MASS_P_BAND = 2e-5
# Tokens whose k-th/(k+1)-th logit gap inside the prefix is below this are
# reported and left out of index-exact comparisons when both sides use the same
# fp32 logits.
MARGIN_SAME_LOGITS = 1e-6


def f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


def assert_close_out(got, ref, rel_l2, max_abs, what=""):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    den = np.linalg.norm(ref)
    rel = np.linalg.norm(got - ref) / (den if den > 0 else 1.0)
    mref = np.abs(ref).max() if ref.size else 0.0
    mx = np.abs(got - ref).max() / (mref if mref > 0 else 1.0) if ref.size else 0.0
    assert rel <= rel_l2 and mx <= max_abs, f"{what}: rel-L2 {rel:.3e} (<= {rel_l2}), max-abs/max {mx:.3e} (<= {max_abs})"
    return rel, mx


def logit_error_bound(x64, w64, b64):
    """Per-element bound on |fl32-accumulated logit - exact logit| for any
    summation order (Higham: gamma_n * sum|terms|, n = d + 1), plus half an
    fp32 ulp for the oracle's own rounding of its float64 value to fp32."""
    d = x64.shape[1]
    u = 2.0 ** -24
    n = d + 1
    gamma = n * u / (1 - n * u)
    s = np.abs(x64) @ np.abs(w64).T + (np.abs(b64)[None, :] if b64 is not None else 0.0)
    exact = x64 @ w64.T + (b64[None, :] if b64 is not None else 0.0)
    return gamma * s + np.spacing(np.abs(exact).astype(np.float32)).astype(np.float64)


def bf16_round(a: np.ndarray) -> np.ndarray:
    return torch.from_numpy(np.asarray(a, np.float32)).to(torch.bfloat16).float().numpy().astype(np.float64)


class Experts:
    """Per-expert float64 host view of a (device or host) weight tensor
    [E, rows, cols], each expert copied once on first use."""

    def __init__(self, t):
        self.t = t
        self.cache = {}

    def __getitem__(self, e):
        e = int(e)
        if e not in self.cache:
            self.cache[e] = self.t[e].cpu().double().numpy()
        return self.cache[e]


def check_layer_tokens(x64, wr64, b64, wg, wu, wd, gpu_logits, gpu_idx, gpu_w, gpu_out, K, k, residual64=None,
                       tol=(BF16_REL_L2, BF16_MAX_ABS), label="layer"):
    """Compare one MoE layer's routing and output on some tokens with the
    oracle, given the layer's input rows x64 [n, d] and its GPU results for
    the same rows (fp32 logits [n, E], picks and weights [n, k], output
    [n, d]).

    Every GPU logit must lie within the rigorous fp32 summation bound of the
    oracle's. A token whose oracle prefix margin exceeds twice its own largest
    bound must get exactly the oracle's expert set (and, where the order inside
    the set is clear of the bounds too, the same slot order). For a near-tie
    token several expert sets are correct: the GPU's set must be one that
    logits within the bounds rank first, and the token's weights and output
    are compared with the oracle evaluated on that set. Returns the number of
    near-tie tokens (printed; at most 10 % of the tokens, or 4)."""
    ref_logits = O.router_logits(x64, wr64, b64).astype(np.float64)
    bound = logit_error_bound(x64, wr64, b64)
    err = np.abs(np.asarray(gpu_logits, np.float64) - ref_logits)
    assert (err <= bound).all(), f"{label}: logit error {err.max():.3e} above bound"
    tb = 2.0 * bound[:, :K].max(axis=1)
    keep = O.prefix_margin(ref_logits, K, k) > tb
    n = x64.shape[0]
    n_tie = int((~keep).sum())
    print(f"[{label}] K={K}: {n_tie} of {n} tokens near a tie (compared on the GPU's valid set)")
    assert n_tie <= max(0.1 * n, 4), f"{label}: {n_tie} of {n} tokens near a tie: the logit bound is too loose"
    ref = O.moe_layer(x64, wr64, b64, wg, wu, wd, k=k, K=K, residual=residual64)
    gi = np.asarray(gpu_idx)
    ref_w = np.array(ref["w"])
    ref_out = np.array(ref["out"])
    srt = -np.sort(-ref_logits[:, :K], axis=-1)[:, :min(k + 1, K)]
    ordered = keep & (np.diff(-srt, axis=-1).min(axis=-1, initial=np.inf) > tb)
    assert np.array_equal(gi[ordered], ref["idx"][ordered]), f"{label}: expert order"
    assert np.array_equal(np.sort(gi[keep], -1), np.sort(ref["idx"][keep], -1)), f"{label}: expert sets"
    for i in range(n):
        S = [int(e) for e in gi[i]]
        assert len(set(S)) == k and all(0 <= e < K for e in S)
        a, b = ref_logits[i, :K], bound[i, :K]
        assert all(a[S[j]] + b[S[j]] >= a[S[j + 1]] - b[S[j + 1]] for j in range(k - 1)), f"{label} token {i}: slot order"
        if keep[i]:
            pos = {int(e): j for j, e in enumerate(ref["idx"][i])}
            ref_w[i] = [ref["w"][i][pos[e]] for e in S]
            continue
        rest = [e for e in range(K) if e not in S]
        assert min(a[S] + b[S]) >= max(a[rest] - b[rest]), f"{label} token {i}: experts {S} are not a valid top-{k}"
        a_S = ref_logits[i].copy()
        a_S[rest] = -1e30  # the oracle evaluated on the GPU's set
        o_i, idx_i, w_i = O.moe_token(x64[i], a_S, wg, wu, wd, K, k)
        assert sorted(idx_i.tolist()) == sorted(S)
        pos = {int(e): j for j, e in enumerate(idx_i)}
        ref_w[i] = [w_i[pos[e]] for e in S]
        ref_out[i] = o_i + (0.0 if residual64 is None else residual64[i])
    assert np.abs(np.asarray(gpu_w, np.float64) - ref_w).max() <= 2e-5, f"{label}: routing weights"
    assert_close_out(np.asarray(gpu_out, np.float64), ref_out, tol[0], tol[1], f"{label} output")
    return n_tie
