"""One workload split over ranks, on one GPU: each rank's share is built as that rank would build
it (paper_2609_34972_gb300.shard), one share after the other, and the shares are reassembled.

- Token split: the rank's flat tokens as one batch element at their own positions, into a cache of
  its own.
- Layer split: the rank plans the other layers as DV_LAYER_DROP and builds every token into the
  shared cache layout; its rows of the other layers stay untouched.
Every (token, layer) must be written by exactly one share, and the reassembled K/V must equal the
unsplit build's (bit for bit where both run the same kernels) and meet the parity bar against the
oracle (Sec. 3.1: the tokens, and the layers given E, are independent).
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


def _cfg():
    return gu.small_config("shard", d=512, n_layers=6, n_kv_heads=2, n_heads=4, head_dim=128,
                           rank=64, n_vis=300, batch=3, x0_sigma=0.5, seed=97, pos_start=35,
                           rope="mrope", rope_theta=1e6, mrope_section=(16, 24, 24),
                           grid=(1, 15, 20), bias_sigma=0.02)


@pytest.mark.parametrize("world", [2, 3])
def test_token_split_reassembles_the_build(world):
    import torch
    import paper_2609_34972_gb300 as dv
    from paper_2609_34972_gb300 import shard as sh
    cfg = _cfg()
    inp = synth.make_inputs(cfg)
    k_full, v_full, plan_full = gu.run_build(inp)
    weights = gu.device_weights(inp)
    x0_flat = gu.torch_bf16(inp.x0, "cuda").reshape(cfg.tokens, cfg.d)
    k = torch.full((cfg.n_layers, cfg.tokens, cfg.n_kv_heads, cfg.head_dim), float("nan"),
                   dtype=torch.bfloat16, device="cuda")
    v = torch.full_like(k, float("nan"))
    owned = []
    for r in range(world):
        part = sh.token_shard(cfg.batch, cfg.n_vis, world, r)
        n = part.tokens
        plan = dv.memory_plan(gu.dv_config(cfg, max_batch=1, max_n_vis=n), weights)
        x0 = x0_flat[part.start:part.stop].reshape(1, n, cfg.d).contiguous()
        pos = torch.from_numpy(sh.shard_positions(inp.pos, part)).cuda()
        kr = torch.zeros((cfg.n_layers, 1, n, cfg.n_kv_heads, cfg.head_dim), dtype=torch.bfloat16,
                         device="cuda")
        vr = torch.zeros_like(kr)
        dv.build_visual_memory(plan, x0, pos, kr, vr)
        torch.cuda.synchronize()
        assert dv.plan_status(plan) == dv.DV_OK
        k[:, part.start:part.stop] = kr[:, 0]
        v[:, part.start:part.stop] = vr[:, 0]
        owned.append((np.arange(part.start, part.stop), np.arange(cfg.n_layers)))
        dv.free(plan)
    sh.check_cover(owned, cfg.tokens, cfg.n_layers)
    toks = np.arange(cfg.tokens)
    ref = oracle.build_tokens(inp, toks)
    gk = k.permute(1, 0, 2, 3).reshape(cfg.tokens, cfg.n_layers, -1).double().cpu().numpy()
    gv = v.permute(1, 0, 2, 3).reshape(cfg.tokens, cfg.n_layers, -1).double().cpu().numpy()
    gu.assert_parity(gk, gv, ref["k"], ref["v"], cfg.head_dim, f"token split over {world}")
    # against the unsplit build: equal up to the bf16 rounding of the output
    fk = gu.gather(k_full, cfg, toks)
    fv = gu.gather(v_full, cfg, toks)
    assert gu.parity(gk, fk, cfg.head_dim)[0] <= 1e-2 and gu.parity(gv, fv, cfg.head_dim)[0] <= 1e-2
    dv.free(plan_full)


@pytest.mark.parametrize("world", [2, 4])
def test_layer_split_reassembles_the_build_bit_for_bit(world):
    # Every rank builds every token with the same kernels as the unsplit build (same token count,
    # so the same engines and tiles); dropped layers only leave their rows alone. So the shares
    # reassemble to the unsplit build exactly.
    import torch
    import paper_2609_34972_gb300 as dv
    from paper_2609_34972_gb300 import shard as sh
    cfg = _cfg()
    inp = synth.make_inputs(cfg)
    k_full, v_full, plan_full = gu.run_build(inp)
    k = torch.full_like(k_full, float("nan"))
    v = torch.full_like(v_full, float("nan"))
    owned = []
    for r in range(world):
        modes = sh.layer_modes(cfg.n_layers, world, r)
        kr, vr, plan = gu.run_build(inp, layer_modes=modes, fill=float("nan"))
        first, stop = sh.layer_shard(cfg.n_layers, world, r)
        assert bool(torch.isnan(kr[:first].float()).all()) and bool(torch.isnan(kr[stop:].float()).all())
        k[first:stop] = kr[first:stop]
        v[first:stop] = vr[first:stop]
        owned.append((np.arange(cfg.tokens), np.arange(first, stop)))
        dv.free(plan)
    sh.check_cover(owned, cfg.tokens, cfg.n_layers)
    assert torch.equal(k, k_full) and torch.equal(v, v_full)
    dv.free(plan_full)
