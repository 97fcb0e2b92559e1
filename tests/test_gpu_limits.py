"""GPU parity at the limits the ABI accepts (include/dv.h): the widest hidden size (d = 16384,
256 K slabs) with the largest rank (r = 256), the widest K/V (64 heads of 128 = 8192 channels),
the most layers (256), and the largest build (2^24 tokens), each against the fp64 oracle on
sampled tokens (every tile, both ends) plus finiteness everywhere.
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


def _sampled_check(cfg, label, n=32, layers=None):
    import torch
    inp = synth.make_inputs(cfg)
    k, v, plan = gu.run_build(inp)
    toks = gu.sample_tokens(cfg.tokens, n=n, seed=7)
    ref = oracle.build_tokens(inp, toks, layers=layers)
    gk, gv = gu.gather(k, cfg, toks), gu.gather(v, cfg, toks)
    if layers is not None:
        gk, gv = gk[:, layers], gv[:, layers]
    gu.assert_parity(gk, gv, ref["k"], ref["v"], cfg.head_dim, label)
    assert bool(torch.isfinite(k).all()) and bool(torch.isfinite(v).all())
    del k, v, plan
    torch.cuda.empty_cache()


def test_widest_hidden_size_and_rank():
    # d = 16384 (the largest accepted), r = 256; 300 tokens (ragged 128-blocks).
    cfg = gu.small_config("max_d", d=16384, n_layers=2, n_kv_heads=2, n_heads=8, head_dim=128,
                          rank=256, n_vis=300, batch=1, x0_sigma=0.5, w_sigma=0.01, seed=91,
                          pos_start=35)
    _sampled_check(cfg, "d 16384 r 256")


def test_widest_kv():
    # n_kv_heads * head_dim = 8192 (the largest accepted): 64 groups of 128 channels per layer.
    cfg = gu.small_config("max_kv", d=1024, n_layers=2, n_kv_heads=64, n_heads=64, head_dim=128,
                          rank=64, n_vis=256, batch=1, x0_sigma=0.5, seed=92, pos_start=35)
    _sampled_check(cfg, "kv 8192")


def test_most_layers():
    # 256 layers (the largest accepted), checked at every 17th layer and the last.
    cfg = gu.small_config("max_L", d=512, n_layers=256, n_kv_heads=1, n_heads=4, head_dim=128,
                          rank=16, n_vis=200, batch=1, x0_sigma=1.0, seed=93, pos_start=5)
    _sampled_check(cfg, "256 layers", layers=list(range(0, 256, 17)) + [255])


def test_largest_build():
    # 2^24 tokens (64 x 262144, the largest build accepted), d = 64, 1 layer: every index of the
    # kernels runs at its widest; RoPE positions up to 262148.
    cfg = gu.small_config("max_T", d=64, n_layers=1, n_kv_heads=1, n_heads=1, head_dim=128,
                          rank=16, n_vis=262144, batch=64, x0_sigma=1.0, seed=94, pos_start=5)
    assert cfg.tokens == 1 << 24
    _sampled_check(cfg, "2^24 tokens", n=64)
