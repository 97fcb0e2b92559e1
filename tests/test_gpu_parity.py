"""GPU parity: the CUDA build (through the C ABI) against the fp64 oracle on the same inputs.

Small cases are compared element by element over every token; they span several 128-row
tiles with a ragged tail, several K slabs, padded ranks and both head widths. The five
workload configurations run at full size, in the launch configuration the benchmark times,
and are compared on sampled tokens (every tile, both ends, all batch elements).
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


def _full_check(inp, label, **kw):
    cfg = inp.cfg
    k, v, plan = gu.run_build(inp, **kw)
    toks = np.arange(cfg.tokens)
    ref = oracle.build_tokens(inp, toks)
    gk = gu.gather(k, cfg, toks, kw.get("slot"), kw.get("slot0", 0))
    gv = gu.gather(v, cfg, toks, kw.get("slot"), kw.get("slot0", 0))
    return gu.assert_parity(gk, gv, ref["k"], ref["v"], cfg.head_dim, label), (k, v, plan)


def test_tiny_config_full():
    inp = synth.make_inputs(synth.CONFIGS["tiny"])
    _full_check(inp, "tiny")


def test_tiny_zero_up_projection():
    # U = 0: the adapter is the identity (Sec. 3.1), K/V = RoPE(W RMSNorm(E)).
    inp = synth.make_inputs(synth.config("tiny", zero_up=True))
    _full_check(inp, "tiny zero-U")


@pytest.mark.parametrize("n_vis,batch,rank", [(64, 1, 16), (256, 2, 64), (300, 1, 128), (576, 1, 64)])
def test_zero_up_projection_is_bit_identical_to_identity_layers(n_vis, batch, rank):
    # U = 0 is the paper's initialisation, so A_l starts as the identity (Sec. 3.1). The fold
    # then multiplies h_l by exact zeros (the rank slab of the K/V weights, 2U and G of the
    # statistic), so the build must equal, value for value, a build whose layers are all
    # DV_LAYER_IDENTITY (D = U = 0 packed, M_l = E): the adapter path adds nothing, not even
    # rounding. Cases: both K/V engines, the small-token statistic and the statistic GEMM.
    import torch
    import paper_2609_34972_gb300 as dv
    cfg = gu.small_config(f"zu_{n_vis}_{batch}_{rank}", d=512, n_layers=3, n_kv_heads=2, n_heads=4,
                          head_dim=128, rank=rank, n_vis=n_vis, batch=batch, zero_up=True,
                          x0_sigma=0.5, seed=71, pos_start=35)
    inp = synth.make_inputs(cfg)
    k_a, v_a, plan_a = gu.run_build(inp)
    k_i, v_i, plan_i = gu.run_build(inp, layer_modes=[dv.DV_LAYER_IDENTITY] * cfg.n_layers)
    assert torch.equal(k_a, k_i) and torch.equal(v_a, v_i)
    # and it is not vacuous: the adapter's down-projection was live (h_l != 0)
    H, _, _, _ = dv.debug_workspace(plan_a, cfg.tokens)
    assert bool((H != 0).any())
    dv.free(plan_a)
    dv.free(plan_i)


def test_tiny_with_bias():
    inp = synth.make_inputs(synth.config("tiny", bias_sigma=0.02))
    _full_check(inp, "tiny bias")


def test_ragged_multi_tile_1d():
    # T = 3 * 200 = 600 = 4 full 128-row tiles + 88; d = 1024 (16 slabs); r = 64;
    # 4 heads of 128; gamma != 1.
    cfg = gu.small_config("ragged1d", d=1024, n_layers=2, n_kv_heads=4, n_heads=8, head_dim=128,
                          rank=64, n_vis=200, batch=3, x0_sigma=0.5, seed=11, pos_start=35)
    _full_check(synth.make_inputs(cfg), "ragged 1-D")


def test_ragged_mrope_padded_rank_bias():
    # T = 2 * 300 = 600, r = 80 (padded to 128 inside), M-RoPE [16, 24, 24] over a 1x20x15
    # grid, K/V bias, GQA-like 2 KV heads of 128.
    cfg = gu.small_config("raggedm", d=512, n_layers=3, n_kv_heads=2, n_heads=8, head_dim=128,
                          rank=80, n_vis=300, batch=2, rope="mrope", rope_theta=1e6,
                          mrope_section=(16, 24, 24), grid=(1, 20, 15), x0_sigma=0.5,
                          bias_sigma=0.02, seed=12, pos_start=15)
    _full_check(synth.make_inputs(cfg), "ragged M-RoPE")


def test_rank_256_two_frames_mrope():
    cfg = gu.small_config("r256", d=768, n_layers=2, n_kv_heads=2, n_heads=4, head_dim=128,
                          rank=256, n_vis=160, batch=1, rope="mrope", rope_theta=1e6,
                          mrope_section=(16, 24, 24), grid=(2, 8, 10), x0_sigma=0.5,
                          ar1_rho=0.9, seed=13, pos_start=15)
    _full_check(synth.make_inputs(cfg), "rank 256")


def test_slot_mapping_and_untouched_cache():
    # Explicit slots (a permutation with an offset) into a larger cache: the written rows match
    # the oracle and every other row keeps its fill value.
    import torch
    cfg = synth.config("tiny", n_vis=40, batch=2)
    inp = synth.make_inputs(cfg)
    rng = np.random.default_rng(5)
    slot = np.stack([rng.permutation(40) + 7, rng.permutation(40) + 3]).astype(np.int32)
    _, (k, v, _) = _full_check(inp, "slots", seq_len=64, batch_cache=3, slot=slot, fill=-7.0)
    written = torch.zeros(k.shape[1], k.shape[2], dtype=torch.bool)
    for b in range(2):
        written[b, torch.as_tensor(slot[b].astype(np.int64))] = True
    untouched = k[:, ~written]
    assert torch.all(untouched == -7.0) and torch.all(v[:, ~written] == -7.0)


def test_slot0_offset():
    cfg = synth.config("tiny", n_vis=50)
    inp = synth.make_inputs(cfg)
    _full_check(inp, "slot0", seq_len=80, slot0=21)


def test_rebuild_same_plan_is_deterministic():
    import torch
    inp = synth.make_inputs(synth.CONFIGS["tiny"])
    k1, v1, plan = gu.run_build(inp)
    k2, v2, _ = gu.run_build(inp, plan=plan)
    assert torch.equal(k1, k2) and torch.equal(v1, v2)


FULL = ["llava15_7b", "llava_next_7b", "qwen25vl_7b_image", "qwen25vl_7b_video"]


@pytest.mark.parametrize("name", FULL)
def test_full_size_sampled(name):
    import torch
    cfg = synth.CONFIGS[name]
    inp = synth.make_inputs(cfg)
    k, v, plan = gu.run_build(inp)
    toks = gu.sample_tokens(cfg.tokens, n=40, seed=1)
    ref = oracle.build_tokens(inp, toks)
    gk, gv = gu.gather(k, cfg, toks), gu.gather(v, cfg, toks)
    gu.assert_parity(gk, gv, ref["k"], ref["v"], cfg.head_dim, name)
    # Every written value is finite, at every token (property that holds at any size).
    assert bool(torch.isfinite(k).all()) and bool(torch.isfinite(v).all())
    del k, v, plan
    torch.cuda.empty_cache()


# Token counts at (or just under) multiples of 256 take the 2-SM kernels with 256-token M
# blocks for all three GEMMs (the others take 128-token 1-SM blocks and the weights-as-M K/V
# kernel); these cases pin that path, including a ragged 256-block and both head widths.

def test_tokens_as_m_path_ragged_mrope_bias():
    # T = 2 x 250 = 500 = 256 + 244; r = 80 (r_pad 128); M-RoPE; K/V bias; 2 heads of 128.
    cfg = gu.small_config("tm_ragged", d=512, n_layers=3, n_kv_heads=2, n_heads=8, head_dim=128,
                          rank=80, n_vis=250, batch=2, rope="mrope", rope_theta=1e6,
                          mrope_section=(16, 24, 24), grid=(1, 10, 25), x0_sigma=0.5,
                          bias_sigma=0.02, seed=31, pos_start=15)
    _full_check(synth.make_inputs(cfg), "tokens-as-M ragged")


def test_tokens_as_m_path_head64():
    # T = 512, 8 heads of 64 (two heads per 128-channel group), r = 16 (r_pad 64).
    cfg = synth.config("tiny", n_vis=512, seed=32)
    _full_check(synth.make_inputs(cfg), "tokens-as-M head 64")


def test_tokens_as_m_path_rank64_two_batches():
    # T = 2 x 256, r = 64: the RMS statistic tile is 64 wide (32 weight rows per CTA).
    cfg = gu.small_config("tm_r64", d=1024, n_layers=2, n_kv_heads=4, n_heads=8, head_dim=128,
                          rank=64, n_vis=256, batch=2, x0_sigma=0.5, seed=33, pos_start=35)
    _full_check(synth.make_inputs(cfg), "tokens-as-M rank 64")


# The statistic GEMM groups layers into 256-column tiles (4 layers for r_pad = 64, 2 for 128, 1
# for 192 and 256, a 192-wide rank leaving 64 zero rows). These cases pin ranks padded to 192 on
# both rank-r engines and layer counts that leave the last group partly empty.

@pytest.mark.parametrize("n_vis,batch,engine", [(256, 2, "2-SM tokens as M"), (150, 2, "1-SM")])
def test_rank_padded_to_192(n_vis, batch, engine):
    cfg = gu.small_config(f"r150_{n_vis}", d=768, n_layers=3, n_kv_heads=2, n_heads=4, head_dim=128,
                          rank=150, n_vis=n_vis, batch=batch, x0_sigma=0.5, seed=41, pos_start=35)
    _full_check(synth.make_inputs(cfg), f"rank 150 (r_pad 192), {engine}")


@pytest.mark.parametrize("rank,n_layers,n_vis,engine", [(16, 5, 512, "2-SM, groups of 4"),
                                                        (96, 3, 512, "2-SM, groups of 2"),
                                                        (96, 3, 300, "1-SM, groups of 2")])
def test_statistic_layer_groups_partly_empty(rank, n_layers, n_vis, engine):
    cfg = gu.small_config(f"grp_{rank}_{n_layers}_{n_vis}", d=512, n_layers=n_layers, n_kv_heads=2,
                          n_heads=4, head_dim=128, rank=rank, n_vis=n_vis, batch=1, x0_sigma=0.5,
                          seed=42 + n_layers, pos_start=35)
    _full_check(synth.make_inputs(cfg), f"rank {rank}, {n_layers} layers, {engine}")


# Layer-wise adapter skipping (App. J): DV_LAYER_DROP layers get no K/V (their cache rows keep
# the fill value); DV_LAYER_IDENTITY layers build K/V from M_l = E, which the oracle computes with
# that layer's adapter weights set to zero (U_l = 0 gives the identity, Sec. 3.1).

def _check_layer_modes(inp, modes, label, **kw):
    import torch
    cfg = inp.cfg
    k, v, plan = gu.run_build(inp, fill=-5.0, layer_modes=modes, **kw)
    ref_inp = synth.Inputs(cfg=cfg, x0=inp.x0, D=inp.D.copy(), U=inp.U.copy(), gamma=inp.gamma,
                           Wk=inp.Wk, Wv=inp.Wv, bk=inp.bk, bv=inp.bv, pos=inp.pos)
    for l, m in enumerate(modes):
        if m == 1:
            ref_inp.D[l] = 0
            ref_inp.U[l] = 0
    kept = [l for l, m in enumerate(modes) if m != 2]
    toks = np.arange(cfg.tokens)
    ref = oracle.build_tokens(ref_inp, toks, layers=kept)
    gk = gu.gather(k, cfg, toks)[:, kept]
    gv = gu.gather(v, cfg, toks)[:, kept]
    gu.assert_parity(gk, gv, ref["k"], ref["v"], cfg.head_dim, label)
    for l, m in enumerate(modes):
        if m == 2:
            assert bool((k[l] == -5.0).all()) and bool((v[l] == -5.0).all()), f"layer {l} written"


def test_layer_modes_weights_as_m_path():
    inp = synth.make_inputs(synth.config("tiny", n_vis=64))
    _check_layer_modes(inp, [2, 1, 0, 2], "layer modes (weights-as-M K/V)")


def test_layer_modes_tokens_as_m_path():
    cfg = gu.small_config("modes_tm", d=512, n_layers=4, n_kv_heads=2, n_heads=4, head_dim=128,
                          rank=64, n_vis=512, batch=1, x0_sigma=0.5, seed=41, pos_start=35)
    _check_layer_modes(synth.make_inputs(cfg), [1, 0, 2, 0], "layer modes (tokens-as-M)")


def test_layer_modes_noalloc_entry():
    inp = synth.make_inputs(synth.config("tiny", n_vis=64, seed=42))
    _check_layer_modes(inp, [0, 2, 2, 1], "layer modes (no-alloc entry)", noalloc=True)


@pytest.mark.parametrize("adapter", ["embedding", "recurrent"])
def test_single_visual_token_rank_one(adapter):
    # The degenerate build: one visual token (one ragged row of a 128-row tile) and a rank-1
    # adapter (r padded to 64), over three layers, in each adapter variant.
    cfg = gu.small_config(f"one token {adapter}", d=256, n_layers=3, n_kv_heads=2, n_heads=2,
                          head_dim=128, rank=1, n_vis=1, batch=1, x0_sigma=0.5, seed=21,
                          pos_start=7, adapter=adapter)
    _full_check(synth.make_inputs(cfg), f"one token, r = 1, {adapter}")


def test_single_token_mrope_grid_batch_three():
    # A 1x1x1 M-RoPE grid per batch element: every axis sits at the same position.
    cfg = gu.small_config("one-token grid", d=384, n_layers=2, n_kv_heads=2, n_heads=4,
                          head_dim=64, rank=8, n_vis=1, batch=3, rope="mrope",
                          rope_theta=1e6, mrope_section=(8, 12, 12), grid=(1, 1, 1),
                          x0_sigma=0.5, seed=22, pos_start=40)
    _full_check(synth.make_inputs(cfg), "one-token M-RoPE grid, batch 3")
