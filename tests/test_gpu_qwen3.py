"""GPU parity of the Qwen3-VL backbone variant: per-head RMSNorm of K (after the bias, before
RoPE, with a learned gain per head channel) and the interleaved M-RoPE frequency layout, on both
K/V engines (weights as M with the head split over warps, tokens as M with a two-pass head
norm), both head widths, with the embedding and the recurrent adapter, and at the full size of
the Qwen3-VL-4B-shaped image workload (the paper's default backbone) on sampled tokens.
"""
import numpy as np
import pytest

import oracle
import synth
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_34972_gb300.build import build_library
    build_library()


def _full_check(inp, label):
    cfg = inp.cfg
    k, v, plan = gu.run_build(inp)
    toks = np.arange(cfg.tokens)
    ref = oracle.build_tokens(inp, toks)
    gk, gv = gu.gather(k, cfg, toks), gu.gather(v, cfg, toks)
    gu.assert_parity(gk, gv, ref["k"], ref["v"], cfg.head_dim, label)
    return k, v


def _qwen3_small(name, **kw):
    base = dict(d=1024, n_layers=3, n_kv_heads=2, n_heads=8, head_dim=128, rank=64,
                rope="mrope_interleaved", rope_theta=5e6, mrope_section=(24, 20, 20),
                x0_sigma=0.5, k_norm=True, pos_start=15)
    base.update(kw)
    return gu.small_config(name, **base)


def test_k_norm_weights_as_m_head128_bias():
    # T = 2 x 300 = 600 tokens: weights-as-M K/V kernel with 128-token tiles (600 -> 640);
    # each 128-channel head spans the 4 epilogue warps.
    cfg = _qwen3_small("q3_wm", n_vis=300, batch=2, grid=(1, 15, 20), bias_sigma=0.02, seed=71)
    _full_check(synth.make_inputs(cfg), "k-norm weights-as-M head 128")


def test_k_norm_weights_as_m_head64():
    # 8 heads of 64: two heads per 128-channel group, each over two warps.
    cfg = synth.config("tiny", n_vis=100, k_norm=True, seed=72)
    _full_check(synth.make_inputs(cfg), "k-norm weights-as-M head 64")


def test_k_norm_tokens_as_m_head128():
    cfg = _qwen3_small("q3_tm", n_vis=256, batch=2, grid=(1, 16, 16), seed=73)
    _full_check(synth.make_inputs(cfg), "k-norm tokens-as-M head 128")


def test_k_norm_tokens_as_m_head64_interleaved():
    # 64-wide heads: interleaved sections (12, 10, 10) over 32 pairs.
    cfg = synth.config("tiny", n_vis=512, k_norm=True, rope="mrope_interleaved", rope_theta=1e6,
                       mrope_section=(12, 10, 10), grid=(2, 16, 16), seed=74)
    _full_check(synth.make_inputs(cfg), "k-norm tokens-as-M head 64 interleaved")


def test_interleaved_mrope_without_k_norm():
    cfg = _qwen3_small("q3_rope", n_vis=200, batch=1, grid=(1, 10, 20), k_norm=False, seed=75)
    _full_check(synth.make_inputs(cfg), "interleaved M-RoPE")


def test_k_norm_recurrent_adapter():
    cfg = synth.config("tiny", n_vis=100, k_norm=True, adapter="recurrent", w_sigma=0.05, seed=76)
    _full_check(synth.make_inputs(cfg), "k-norm recurrent")


def test_k_norm_with_dropped_layers():
    # The K-norm gain follows the plan's layer compaction.
    import torch
    cfg = _qwen3_small("q3_drop", n_vis=200, batch=1, grid=(1, 10, 20), n_layers=4, seed=77)
    inp = synth.make_inputs(cfg)
    modes = [2, 0, 2, 0]
    k, v, plan = gu.run_build(inp, fill=-3.0, layer_modes=modes)
    toks = np.arange(cfg.tokens)
    ref = oracle.build_tokens(inp, toks, layers=[1, 3])
    gk, gv = gu.gather(k, cfg, toks)[:, [1, 3]], gu.gather(v, cfg, toks)[:, [1, 3]]
    gu.assert_parity(gk, gv, ref["k"], ref["v"], cfg.head_dim, "k-norm dropped layers")
    assert bool((k[0] == -3.0).all()) and bool((k[2] == -3.0).all())


def test_qwen3vl_4b_full_size_sampled():
    import torch
    cfg = synth.CONFIGS["qwen3vl_4b_image"]
    inp = synth.make_inputs(cfg)
    k, v, plan = gu.run_build(inp)
    toks = gu.sample_tokens(cfg.tokens, n=40, seed=3)
    ref = oracle.build_tokens(inp, toks)
    gk, gv = gu.gather(k, cfg, toks), gu.gather(v, cfg, toks)
    gu.assert_parity(gk, gv, ref["k"], ref["v"], cfg.head_dim, "qwen3vl_4b_image")
    assert bool(torch.isfinite(k).all()) and bool(torch.isfinite(v).all())
    del k, v, plan
    torch.cuda.empty_cache()
