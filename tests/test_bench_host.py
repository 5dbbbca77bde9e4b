"""bench.py's roofline arithmetic, on the host.

The expert FFN's algorithmic bytes and FLOPs per launch are what the
headline roofline divides by the measured duration; pin them to the sizes
worked out by hand for the T=2048, K=64 prefill workload (64 active experts),
and the bound they select against the measured peaks.
"""
import importlib.util
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    sys.path.insert(0, ROOT)
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    b = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(b)
    return b


def test_ffn_algorithmic_bytes_prefill_k64():
    b = _bench()
    wl = b.W.PREFILL
    R, D = wl.T * wl.k, 64
    assert (wl.T, wl.d, wl.k, wl.m) == (2048, 2048, 8, 768)
    # weights: 64 experts x (gate, up, down) x 2048 x 768 bf16; rows: x_perm
    # read, h written, y written, 16384 rows each
    weights = 64 * 3 * 2048 * 768 * 2
    assert weights == 603979776
    assert b.algo_bytes_ffn(wl, R, D) == weights + 16384 * 2048 * 2 + 16384 * 768 * 2 + 16384 * 2048 * 2
    assert b.algo_bytes_ffn(wl, R, D) == 763363328


def test_ffn_bound_is_hbm_at_the_measured_peaks():
    b = _bench()
    wl = b.W.PREFILL
    R = wl.T * wl.k
    flops = 6.0 * R * wl.d * wl.m
    assert flops == 154618822656.0
    pk = {"hbm_gbs": 6652.7, "bf16_tflops": 1927.5}
    t_mem = b.algo_bytes_ffn(wl, R, 64) / (pk["hbm_gbs"] * 1e9)
    t_compute = flops / (pk["bf16_tflops"] * 1e12)
    assert t_mem > t_compute  # 114.7 us of HBM against 80.2 us of tensor work
    assert abs(t_mem * 1e6 - 114.7) < 0.1 and abs(t_compute * 1e6 - 80.2) < 0.1


def test_ffn_algorithmic_bytes_with_the_row_gather():
    """The layer's own launch from 8192 routed rows reads x once instead of
    the gathered rows: 704.6 MB per launch at T=2048, K=64 (105.9 us at the
    measured HBM peak against 80.2 us of tensor work: still HBM-bound)."""
    b = _bench()
    wl = b.W.PREFILL
    R, D = wl.T * wl.k, 64
    with_gather = b.algo_bytes_ffn(wl, R, D, wl.T)
    assert with_gather == 64 * 3 * 2048 * 768 * 2 + 2048 * 2048 * 2 + 16384 * 768 * 2 + 16384 * 2048 * 2
    assert with_gather == 704643072
    assert abs(with_gather / 6652.7e9 * 1e6 - 105.9) < 0.1


def test_layer_gather_range_matches_the_layer():
    """bench.py times the gathering launch exactly where the layer uses it:
    from 8192 routed rows up to the one-launch limit of 32768."""
    b = _bench()
    assert not b.layer_gathers(8191)
    assert b.layer_gathers(8192) and b.layer_gathers(16384) and b.layer_gathers(32768)
    assert not b.layer_gathers(32769) and not b.layer_gathers(131072)
