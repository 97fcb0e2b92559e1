"""Host-side arithmetic of bench.py, on CPU: the oracle's stratified token sample and the roofline
figures of a line."""
import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def test_stratified_sample_covers_every_batch_element():
    import bench
    import synth
    cfg = synth.CONFIGS["llava_next_7b"]
    toks = bench.stratified_tokens(cfg, 512, seed=0)
    assert len(toks) == 512 and len(np.unique(toks)) == 512
    assert toks.min() >= 0 and toks.max() < cfg.tokens
    b = toks // cfg.n_vis
    i = toks % cfg.n_vis
    counts = np.bincount(b, minlength=cfg.batch)
    assert counts.min() == counts.max() == 64            # 512 over 8 elements, evenly
    for e in range(cfg.batch):                            # each element's share spans its positions
        ie = np.sort(i[b == e])
        assert ie[0] < cfg.n_vis / 64 and ie[-1] >= cfg.n_vis - cfg.n_vis / 64
    small = synth.config("tiny", batch=3, n_vis=5)
    assert sorted(bench.stratified_tokens(small, 100)) == list(range(15))   # capped at T


def test_roofline_figures():
    import bench
    import synth
    cfg = synth.CONFIGS["llava_next_7b"]
    peaks = {"bf16_tflops": 1888.7, "bf16_tflops_sustained": 1708.1, "hbm_gbs": 6764.0}

    class FakeDv:
        @staticmethod
        def kv_kernel(plan, tokens):
            return "kv"

    kv_ms = 26.0
    stage = [0.4 * 10, 0.05 * 10, 0.4 * 10, kv_ms * 10]
    roof, step = bench.roofline_of(FakeDv, None, cfg, stage, 10, ms_total=600.0, ms_step=28.0,
                                   peaks=peaks, peak_src="measured", tokens=cfg.tokens)
    flops = 4.0 * cfg.d * cfg.kv * cfg.tokens * cfg.n_layers
    assert roof["flops_per_launch"] == pytest.approx(flops)
    assert roof["achieved"] == pytest.approx(flops / (kv_ms * 1e-3) / 1e12)
    assert roof["peak"] == 1888.7                          # a 0.6 s region takes the burst figure
    assert roof["frac"] == pytest.approx(roof["achieved"] / 1888.7)
    roof2, _ = bench.roofline_of(FakeDv, None, cfg, stage, 10, ms_total=2500.0, ms_step=28.0,
                                 peaks=peaks, peak_src="measured", tokens=cfg.tokens)
    assert roof2["peak"] == 1708.1                         # 2 s or more: the sustained figure
    t_roof = max(cfg.flops() / 1888.7e12, cfg.min_bytes() / 6764e9) * 1e3
    assert step["t_roof_ms"] == pytest.approx(t_roof) and step["frac"] == pytest.approx(t_roof / 28.0)
    assert 27.0 < t_roof < 27.1                             # 51.02 TFLOP at the burst peak
    # beside them, NVIDIA's dense bf16 figure of 2.25 PFLOP/s: 22.7 ms for the same work
    assert roof["frac_nominal"] == pytest.approx(roof["achieved"] / 2250.0)
    assert step["frac_nominal"] == pytest.approx(cfg.flops() / 2250e12 * 1e3 / 28.0)


def test_scaling_values():
    import bench
    assert bench.strong_scaling_value(23040, 20, 600.0) == pytest.approx(23040 * 20 / 0.6)
    assert bench.weak_scaling_value(4, 23040, 20, 600.0) == pytest.approx(4 * 23040 * 20 / 0.6)
