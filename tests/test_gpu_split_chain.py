"""GPU parity of the recurrent adapter with the split chain (Sec. 3.1 Eq. 6, dv_config.split_chain).

The chain M_l = M_{l-1} + SiLU(M_{l-1} D_l) U_l feeds each layer's down-projection from the
previous state, so a bf16 operand there (and for h_l in the up-projection) adds one rounding per
layer, and the error grows with depth. With split_chain the two GEMMs read each operand as a high
and a low bf16 part, and the state keeps about fp32 accuracy; only the K/V GEMM reads the bf16
rounding of M_l. Evaluated in the paper's order, the chain runs on chip at r_pad 64 (the low
parts beside the state in shared memory) and as per-layer launches at larger r_pad; rearranged
(z_l = E D_l^T + sum_{j<l} h_j (D_l U_j)^T), h_j and the products D_l U_j each come in two parts.
The small cases run on both evaluations. These cases check the build against the fp64 oracle,
the chain's state layer by layer, and that the split chain stays at the bar where the one-part
chain drifts toward it.
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


def _errors(inp, toks, **kw):
    cfg = inp.cfg
    k, v, plan = gu.run_build(inp, **kw)
    ref = oracle.build_tokens(inp, toks)
    gk, gv = gu.gather(k, cfg, toks), gu.gather(v, cfg, toks)
    return gk, gv, ref, plan


PATHS = ["chain", "rearranged"]


@pytest.mark.parametrize("path", PATHS)
@pytest.mark.parametrize("rank,d", [(16, 512), (80, 1024), (150, 768), (256, 512), (80, 384),
                                    (200, 640)])
def test_split_chain_every_rank_padding(rank, d, path):
    from dataclasses import replace
    cfg = gu.small_config(f"split_r{rank}", d=d, n_layers=3, n_kv_heads=2, n_heads=4, head_dim=128,
                          rank=rank, n_vis=150, batch=2, x0_sigma=0.5, w_sigma=0.05, seed=80 + rank,
                          pos_start=35, adapter="recurrent", split_chain=True)
    inp = synth.make_inputs(replace(cfg, recurrent_path=path))
    toks = np.arange(cfg.tokens)
    gk, gv, ref, plan = _errors(inp, toks)
    gu.assert_parity(gk, gv, ref["k"], ref["v"], cfg.head_dim, f"split chain r{rank}, {path}")


@pytest.mark.parametrize("path", PATHS)
def test_split_chain_keeps_the_state_accurate_through_depth(path):
    # 8 layers with adapters 2.5x the workloads' scale (sigma 0.05; M_l roughly doubles per
    # layer). The split chain's bf16 M_l is the rounding of an accurate state at every depth
    # (at most 2^-8 of the element), and its K/V meet the bar; the one-part chain on the same
    # inputs carries each layer's operand roundings forward.
    import torch
    import paper_2609_34972_gb300 as dv
    base = gu.small_config("split_deep", d=1024, n_layers=8, n_kv_heads=2, n_heads=4, head_dim=128,
                           rank=64, n_vis=200, batch=1, x0_sigma=0.5, w_sigma=0.05, seed=91,
                           pos_start=35, adapter="recurrent")
    from dataclasses import replace
    base = replace(base, recurrent_path=path)
    toks = np.arange(base.tokens)
    ref = oracle.build_tokens(synth.make_inputs(base), toks, want=("k", "v", "m"))
    m = ref["m"]                                                     # [T, L, d]
    ms = np.sqrt(np.mean(m * m, axis=2, keepdims=True))
    merr, kverr = {}, {}
    for split in (False, True):
        inp = synth.make_inputs(replace(base, split_chain=split))
        k, v, plan = gu.run_build(inp)
        mem = dv.debug_memory(plan, base.tokens)
        torch.cuda.synchronize()
        mg = mem.double().cpu().numpy().transpose(1, 0, 2)
        merr[split] = (np.abs(mg - m) / np.maximum(np.abs(m), ms)).max(axis=(0, 2))  # per layer
        gk, gv = gu.gather(k, base, toks), gu.gather(v, base, toks)
        kverr[split] = max(gu.parity(gk, ref["k"], base.head_dim)[0],
                           gu.parity(gv, ref["v"], base.head_dim)[0])
        if split:
            gu.assert_parity(gk, gv, ref["k"], ref["v"], base.head_dim,
                             f"split chain 8 layers, sigma 0.05, {path}")
        dv.free(plan)
    # the split chain's state: its bf16 rounding (unit roundoff 2^-8) and nothing more, at
    # every layer
    assert merr[True].max() <= 2.0 ** -8 * 1.01, merr[True]
    # and clearly tighter than the one-part chain's at depth
    assert merr[True][-1] < 0.5 * merr[False][-1], (merr[True], merr[False])
    assert kverr[True] < kverr[False], (kverr[True], kverr[False])


@pytest.mark.parametrize("path", PATHS)
def test_split_chain_layer_modes_and_noalloc(path):
    import torch
    cfg = synth.config("tiny", n_vis=100, w_sigma=0.05, seed=93, adapter="recurrent", split_chain=True,
                       recurrent_path=path)
    inp = synth.make_inputs(cfg)
    modes = [0, 1, 0, 2]
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
    gu.assert_parity(gu.gather(k, cfg, toks)[:, kept], gu.gather(v, cfg, toks)[:, kept],
                     ref["k"], ref["v"], cfg.head_dim, f"split chain layer modes, {path}")
    assert bool((k[3] == -5.0).all())
    k2, v2, _ = gu.run_build(inp, plan=plan, fill=-5.0, noalloc=True)
    assert torch.equal(k, k2) and torch.equal(v, v2)


@pytest.mark.parametrize("path", ["auto", "chain"])
@pytest.mark.parametrize("name", ["llava15_7b", "llava_next_7b", "qwen25vl_7b_video"])
def test_split_chain_full_size_sampled(name, path):
    # Full-size recurrent builds with the split chain, sampled tokens (every token block's edges,
    # every batch element) against the oracle. "auto": on chip for LLaVA-1.5 (r_pad 64), the
    # rearranged chain for the larger builds; "chain": on chip, or per layer at r_pad 128 and 256.
    import torch
    from dataclasses import replace
    cfg = replace(synth.CONFIGS[name], adapter="recurrent", split_chain=True, recurrent_path=path)
    inp = synth.make_inputs(cfg)
    toks = gu.sample_tokens(cfg.tokens, n=24, seed=2)
    gk, gv, ref, plan = _errors(inp, toks)
    gu.assert_parity(gk, gv, ref["k"], ref["v"], cfg.head_dim, f"{name} recurrent split chain, {path}")
    del plan
    torch.cuda.empty_cache()
