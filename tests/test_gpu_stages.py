"""Stage-wise GPU checks against the oracle: the stacked down-projection with SiLU (H), the
row sums of squares of E, and the RMS statistic of M_l, read from the build's workspace."""
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


CASES = {
    "tiny": synth.CONFIGS["tiny"],
    # 500 tokens: the rank-r GEMMs run on CTA pairs with 256-token blocks (ragged second block)
    "pairs": gu.small_config("pairs", d=768, n_layers=2, n_kv_heads=2, n_heads=4,
                             head_dim=128, rank=96, n_vis=500, batch=1, x0_sigma=0.5, seed=22),
    "ragged": gu.small_config("ragged", d=1024, n_layers=3, n_kv_heads=2, n_heads=4,
                              head_dim=128, rank=80, n_vis=300, batch=2, x0_sigma=0.5, seed=21),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_stage_outputs(name):
    import torch
    import paper_2609_34972_gb300 as dv
    cfg = CASES[name]
    inp = synth.make_inputs(cfg)
    k, v, plan = gu.run_build(inp)
    H, rstd, xx, r_pad = dv.debug_workspace(plan, cfg.tokens)
    torch.cuda.synchronize()
    ref = oracle.build_tokens(inp, np.arange(cfg.tokens), want=("h", "m"))
    x = synth.bf16_to_f32(inp.x0).astype(np.float64).reshape(cfg.tokens, cfg.d)
    # row sums of squares of E: fp32 accumulation of exact squares
    np.testing.assert_allclose(xx.double().cpu().numpy(), (x * x).sum(1), rtol=1e-5)
    # H: SiLU(x D_l) rounded to bf16; padded columns are zero
    Hn = H.double().cpu().numpy().reshape(cfg.tokens, cfg.n_layers, r_pad)
    h = ref["h"]
    assert np.all(Hn[:, :, cfg.rank:] == 0.0)
    scale = np.sqrt(np.mean(h * h))
    err = np.abs(Hn[:, :, :cfg.rank] - h) / np.maximum(np.abs(h), scale)
    assert err.max() <= 1e-2, f"H max scaled err {err.max():.3e}"
    # rstd_l = 1 / sqrt(mean(M_l^2) + eps)
    m = ref["m"]
    rs_ref = 1.0 / np.sqrt(np.mean(m * m, axis=2) + cfg.rms_eps)     # [T, L]
    rs = rstd.double().cpu().numpy().T
    np.testing.assert_allclose(rs, rs_ref, rtol=5e-3)
    dv.free(plan)


def test_stage_workspace_holds_only_planned_layers():
    # With DV_LAYER_DROP layers the plan is compacted: H and rstd hold the kept layers in order,
    # and an IDENTITY layer's statistic is that of E itself.
    import torch
    import paper_2609_34972_gb300 as dv
    cfg = CASES["ragged"]
    inp = synth.make_inputs(cfg)
    modes = [dv.DV_LAYER_DROP, dv.DV_LAYER_ADAPTER, dv.DV_LAYER_IDENTITY]
    k, v, plan = gu.run_build(inp, layer_modes=modes)
    assert plan.layers == [1, 2]
    H, rstd, xx, r_pad = dv.debug_workspace(plan, cfg.tokens)
    torch.cuda.synchronize()
    assert tuple(H.shape) == (cfg.tokens, 2 * r_pad) and tuple(rstd.shape) == (2, cfg.tokens)
    ref = oracle.build_tokens(inp, np.arange(cfg.tokens), want=("h", "m"), layers=[1])
    Hn = H.double().cpu().numpy().reshape(cfg.tokens, 2, r_pad)
    h = ref["h"][:, 0]
    scale = np.sqrt(np.mean(h * h))
    err = np.abs(Hn[:, 0, :cfg.rank] - h) / np.maximum(np.abs(h), scale)
    assert err.max() <= 1e-2, f"H max scaled err {err.max():.3e}"
    assert np.all(Hn[:, 1] == 0.0)                      # D = 0 for the identity layer
    m = ref["m"][:, 0]
    x = synth.bf16_to_f32(inp.x0).astype(np.float64).reshape(cfg.tokens, cfg.d)
    rs = rstd.double().cpu().numpy()
    np.testing.assert_allclose(rs[0], 1.0 / np.sqrt(np.mean(m * m, axis=1) + cfg.rms_eps), rtol=5e-3)
    np.testing.assert_allclose(rs[1], 1.0 / np.sqrt(np.mean(x * x, axis=1) + cfg.rms_eps), rtol=5e-3)
    dv.free(plan)
