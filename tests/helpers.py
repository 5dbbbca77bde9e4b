"""Shared helpers of the GPU parity tests (comparison rules and tolerances)."""
import numpy as np
import torch

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
