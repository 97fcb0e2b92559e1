"""GPU parity of the recurrent adapter (Sec. 3.1 Eq. 6): M_0 = E, M_l = M_{l-1} +
SiLU(M_{l-1} D_l) U_l, then the same norm, projections, rotation and cache store as the
embedding adapter. Both ways the library evaluates the chain are compared with the fp64 oracle's
recurrent variant on the same inputs: the chain in the paper's order (on chip, or per-layer
launches where no cluster fits) and the rearranged chain (E D^T, the r-wide recurrence through
the products D_l U_j, the running sum of M_l), element by element on small cases (every r_pad,
both K/V engines, ragged tails, M-RoPE and bias, layer modes, the no-alloc entry) and, with the
automatic choice, on sampled tokens at full size. The intermediates (SiLU(M_{l-1} D_l), bf16 M_l,
the RMS statistic) are checked stage by stage.
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


def _rec(cfg, **kw):
    from dataclasses import replace
    return replace(cfg, adapter="recurrent", **kw)


def _full_check(inp, label, **kw):
    cfg = inp.cfg
    k, v, plan = gu.run_build(inp, **kw)
    toks = np.arange(cfg.tokens)
    ref = oracle.build_tokens(inp, toks)
    gk, gv = gu.gather(k, cfg, toks), gu.gather(v, cfg, toks)
    return gu.assert_parity(gk, gv, ref["k"], ref["v"], cfg.head_dim, label), (k, v, plan)


PATHS = ["chain", "rearranged"]


@pytest.mark.parametrize("path", PATHS)
def test_recurrent_tiny(path):
    _full_check(synth.make_inputs(_rec(synth.CONFIGS["tiny"], recurrent_path=path)),
                f"recurrent tiny, {path}")


def test_recurrent_zero_up_equals_embedding_build():
    # U = 0: every A_l is the identity, so the recurrent and embedding builds both give
    # K/V of RMSNorm(E) at every layer.
    import torch
    emb = synth.make_inputs(synth.config("tiny", zero_up=True, n_vis=96))
    rec = synth.make_inputs(_rec(emb.cfg))
    ke, ve, _ = gu.run_build(emb)
    kr, vr, _ = gu.run_build(rec)
    _full_check(rec, "recurrent zero-U")
    # same math, different rounding paths (the recurrent K/V GEMM reads bf16 M_l = bf16(E)
    # exactly; the embedding one reads E and zero rank columns): agree to bf16 rounding
    assert float((kr.float() - ke.float()).abs().max()) <= 2e-2 * float(ke.float().abs().max())
    assert float((vr.float() - ve.float()).abs().max()) <= 2e-2 * float(ve.float().abs().max())


@pytest.mark.parametrize("path", PATHS)
@pytest.mark.parametrize("rank,d,splits_hint", [(16, 512, "r_pad 64"), (80, 1024, "r_pad 128"),
                                                (150, 768, "r_pad 192"), (256, 512, "r_pad 256")])
def test_recurrent_every_rank_padding(rank, d, splits_hint, path):
    # 300 tokens in 2 batch elements: 3 token blocks (ragged), K split over the cluster.
    cfg = gu.small_config(f"rec_r{rank}", d=d, n_layers=3, n_kv_heads=2, n_heads=4, head_dim=128,
                          rank=rank, n_vis=150, batch=2, x0_sigma=0.5, w_sigma=0.05, seed=50 + rank,
                          pos_start=35, adapter="recurrent")
    _full_check(synth.make_inputs(_rec(cfg, recurrent_path=path)), f"recurrent {splits_hint}, {path}")


@pytest.mark.parametrize("path", PATHS)
@pytest.mark.parametrize("n_layers,n_vis,batch", [(1, 1, 1), (2, 129, 1), (3, 257, 1), (4, 193, 2)])
def test_recurrent_edge_shapes(n_layers, n_vis, batch, path):
    # One layer (no recurrence), two layers (nothing loaded two layers ahead), a single token,
    # and odd token-block counts (the running sum takes two blocks per CTA; the last pair has
    # one block past the build) with ragged tails.
    cfg = synth.config("tiny", n_layers=n_layers, n_vis=n_vis, batch=batch, w_sigma=0.05,
                       seed=70 + n_layers, adapter="recurrent", recurrent_path=path)
    _full_check(synth.make_inputs(cfg), f"recurrent L{n_layers} T{n_vis * batch}, {path}")


@pytest.mark.parametrize("path", PATHS)
@pytest.mark.parametrize("d,rank", [(384, 80), (640, 200)])
def test_recurrent_narrow_slices(d, rank, path):
    # d not a multiple of 256: the running sum takes 128-column slices (its second kernel
    # shape: four stages, two epilogue warps per lane quarter), at r_pad 128 and 256, with a
    # ragged tail and an odd number of token blocks.
    cfg = gu.small_config(f"rec_d{d}", d=d, n_layers=3, n_kv_heads=2, n_heads=4, head_dim=128,
                          rank=rank, n_vis=330, batch=1, x0_sigma=0.5, w_sigma=0.05,
                          seed=90 + rank, pos_start=7, adapter="recurrent")
    _full_check(synth.make_inputs(_rec(cfg, recurrent_path=path)), f"recurrent d {d} r {rank}, {path}")


@pytest.mark.parametrize("path", PATHS)
def test_recurrent_tokens_as_m_mrope_bias(path):
    # T = 2 x 256: the K/V launch takes the tokens-as-M engine over the stacked M_l.
    cfg = gu.small_config("rec_tm", d=512, n_layers=3, n_kv_heads=2, n_heads=8, head_dim=128,
                          rank=64, n_vis=256, batch=2, rope="mrope", rope_theta=1e6,
                          mrope_section=(16, 24, 24), grid=(1, 16, 16), x0_sigma=0.5,
                          bias_sigma=0.02, w_sigma=0.05, seed=61, pos_start=15,
                          adapter="recurrent")
    _full_check(synth.make_inputs(_rec(cfg, recurrent_path=path)), f"recurrent tokens-as-M, {path}")


@pytest.mark.parametrize("path", PATHS)
def test_recurrent_long_chain_head64(path):
    # 12 layers of 8 x 64 heads: the state passes through many steps.
    cfg = synth.config("tiny", n_layers=12, n_vis=200, w_sigma=0.05, seed=62, adapter="recurrent",
                       recurrent_path=path)
    _full_check(synth.make_inputs(cfg), f"recurrent 12 layers, {path}")


@pytest.mark.parametrize("path", PATHS)
def test_recurrent_rebuild_is_deterministic(path):
    # Every sum runs in a fixed order: two builds agree bit for bit.
    import torch
    cfg = gu.small_config("rec_det", d=1024, n_layers=2, n_kv_heads=2, n_heads=4, head_dim=128,
                          rank=64, n_vis=200, batch=1, x0_sigma=0.5, seed=63, adapter="recurrent")
    cfg = _rec(cfg, recurrent_path=path)
    inp = synth.make_inputs(cfg)
    k1, v1, plan = gu.run_build(inp)
    k2, v2, _ = gu.run_build(inp, plan=plan)
    assert torch.equal(k1, k2) and torch.equal(v1, v2)


@pytest.mark.parametrize("path", PATHS)
def test_recurrent_stages(path):
    # H_l = bf16(SiLU(M_{l-1} D_l)), bf16 M_l and rstd_l = 1 / sqrt(mean(M_l^2) + eps) of the
    # chain against the oracle's fp64 chain.
    import torch
    import paper_2609_34972_gb300 as dv
    cfg = gu.small_config("rec_stage", d=1024, n_layers=3, n_kv_heads=2, n_heads=4, head_dim=128,
                          rank=80, n_vis=300, batch=1, x0_sigma=0.5, w_sigma=0.05, seed=64,
                          adapter="recurrent")
    cfg = _rec(cfg, recurrent_path=path)
    inp = synth.make_inputs(cfg)
    k, v, plan = gu.run_build(inp)
    H, rstd, _, r_pad = dv.debug_workspace(plan, cfg.tokens)
    mem = dv.debug_memory(plan, cfg.tokens)
    torch.cuda.synchronize()
    ref = oracle.build_tokens(inp, np.arange(cfg.tokens), want=("h", "m"))
    Hn = H.double().cpu().numpy().reshape(cfg.tokens, cfg.n_layers, r_pad)
    h = ref["h"]
    assert np.all(Hn[:, :, cfg.rank:] == 0.0)
    scale = np.sqrt(np.mean(h * h))
    err = np.abs(Hn[:, :, :cfg.rank] - h) / np.maximum(np.abs(h), scale)
    assert err.max() <= 2e-2, f"H max scaled err {err.max():.3e}"
    m = ref["m"]                                              # [T, L, d]
    mg = mem.double().cpu().numpy().transpose(1, 0, 2)       # [T, L, d]
    ms = np.sqrt(np.mean(m * m, axis=2, keepdims=True))
    merr = np.abs(mg - m) / np.maximum(np.abs(m), ms)
    assert merr.max() <= 1e-2, f"M max scaled err {merr.max():.3e}"
    rs_ref = 1.0 / np.sqrt(np.mean(m * m, axis=2) + cfg.rms_eps)
    np.testing.assert_allclose(rstd.double().cpu().numpy().T, rs_ref, rtol=2e-3)
    dv.free(plan)


@pytest.mark.parametrize("path", PATHS)
def test_recurrent_layer_modes(path):
    # IDENTITY and DROP both pass the state on unchanged (M_l = M_{l-1}); DROP writes no K/V.
    # The oracle sees zero D_l, U_l at those layers and is compared on the kept ones.
    import torch
    cfg = _rec(synth.config("tiny", n_vis=100, w_sigma=0.05, seed=65), recurrent_path=path)
    inp = synth.make_inputs(cfg)
    modes = [1, 0, 2, 0]
    k, v, plan = gu.run_build(inp, fill=-5.0, layer_modes=modes)
    ref_inp = synth.Inputs(cfg=cfg, x0=inp.x0, D=inp.D.copy(), U=inp.U.copy(), gamma=inp.gamma,
                           Wk=inp.Wk, Wv=inp.Wv, bk=inp.bk, bv=inp.bv, pos=inp.pos)
    for l, mo in enumerate(modes):
        if mo != 0:
            ref_inp.D[l] = 0
            ref_inp.U[l] = 0
    kept = [l for l, mo in enumerate(modes) if mo != 2]
    toks = np.arange(cfg.tokens)
    ref = oracle.build_tokens(ref_inp, toks, layers=kept)
    gk = gu.gather(k, cfg, toks)[:, kept]
    gv = gu.gather(v, cfg, toks)[:, kept]
    gu.assert_parity(gk, gv, ref["k"], ref["v"], cfg.head_dim, "recurrent layer modes")
    assert bool((k[2] == -5.0).all()) and bool((v[2] == -5.0).all())


@pytest.mark.parametrize("path", PATHS)
def test_recurrent_noalloc_entry(path):
    import torch
    inp = synth.make_inputs(_rec(synth.config("tiny", n_vis=64, seed=66), recurrent_path=path))
    k1, v1, plan = gu.run_build(inp)
    k2, v2, _ = gu.run_build(inp, plan=plan, noalloc=True)
    assert torch.equal(k1, k2) and torch.equal(v1, v2)


@pytest.mark.parametrize("path", ["auto", "chain"])
@pytest.mark.parametrize("name", ["llava15_7b", "qwen25vl_7b_image", "llava_next_7b",
                                  "qwen25vl_7b_video"])
def test_recurrent_full_size_sampled(name, path):
    # "auto" takes the rearranged chain for all but the LLaVA-1.5 shape; "chain" the paper's order
    import torch
    cfg = _rec(synth.CONFIGS[name], recurrent_path=path)
    inp = synth.make_inputs(cfg)
    k, v, plan = gu.run_build(inp)
    toks = gu.sample_tokens(cfg.tokens, n=24, seed=2)
    ref = oracle.build_tokens(inp, toks)
    gk, gv = gu.gather(k, cfg, toks), gu.gather(v, cfg, toks)
    gu.assert_parity(gk, gv, ref["k"], ref["v"], cfg.head_dim, f"{name} recurrent, {path}")
    assert bool(torch.isfinite(k).all()) and bool(torch.isfinite(v).all())
    del k, v, plan
    torch.cuda.empty_cache()


def test_recurrent_down_projection_on_pairs():
    # r_pad 256 and 10000 tokens (79 blocks of 128, the last ragged): enough token blocks that the
    # down-projection needs no K split, so it runs on CTA pairs with per-layer maps of the
    # previous state and of layer l's rows of D. Sampled tokens against the oracle.
    import torch
    cfg = gu.small_config("rec_pairs", d=512, n_layers=3, n_kv_heads=2, n_heads=4, head_dim=128,
                          rank=200, n_vis=5000, batch=2, x0_sigma=0.5, w_sigma=0.05, seed=171,
                          pos_start=35, adapter="recurrent")
    inp = synth.make_inputs(cfg)
    k, v, plan = gu.run_build(inp)
    toks = gu.sample_tokens(cfg.tokens, n=48, seed=3)
    ref = oracle.build_tokens(inp, toks)
    gk, gv = gu.gather(k, cfg, toks), gu.gather(v, cfg, toks)
    gu.assert_parity(gk, gv, ref["k"], ref["v"], cfg.head_dim, "recurrent down on pairs")
    assert bool(torch.isfinite(k).all()) and bool(torch.isfinite(v).all())
