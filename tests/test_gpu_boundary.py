"""The C ABI on a GPU: argument errors launch nothing, failure detection reports a device-side
timeout without faulting, and empty builds are no-ops."""
import ctypes

import numpy as np
import pytest

import synth
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_34972_gb300.build import build_library
    build_library()
    import paper_2609_34972_gb300 as dv
    inp = synth.make_inputs(synth.CONFIGS["tiny"])
    plan = dv.memory_plan(gu.dv_config(inp.cfg), gu.device_weights(inp))
    yield dv, inp, plan
    dv.free(plan)


def _cache(cfg, torch, S=None):
    shape = (cfg.n_layers, cfg.batch, S or cfg.n_vis, cfg.n_kv_heads, cfg.head_dim)
    return (torch.zeros(shape, dtype=torch.bfloat16, device="cuda"),
            torch.zeros(shape, dtype=torch.bfloat16, device="cuda"))


def test_device_wait_timeout_is_reported_and_context_survives(env):
    import torch
    dv, inp, plan = env
    dv.debug_wait_timeout(plan, 2000)       # 2 ms wait on a barrier nothing completes
    assert dv.plan_status(plan) == dv.DV_ERR_DEVICE_TIMEOUT
    assert dv.plan_status(plan) == dv.DV_OK  # cleared by the read
    k, v, _ = gu.run_build(inp, plan=plan)   # the context still works
    assert bool(torch.isfinite(k).all())


def test_too_many_tokens_rejected(env):
    import torch
    dv, inp, plan = env
    cfg = inp.cfg
    x0 = torch.zeros((1, cfg.n_vis + 1, cfg.d), dtype=torch.bfloat16, device="cuda")
    pos = torch.zeros((1, 1, cfg.n_vis + 1), dtype=torch.int32, device="cuda")
    k, v = _cache(cfg, torch, S=cfg.n_vis + 1)
    with pytest.raises(dv.DvError) as e:
        dv.build_visual_memory(plan, x0, pos, k, v)
    assert e.value.code == dv.DV_ERR_UNSUPPORTED_SHAPE


def test_misaligned_x0_rejected(env):
    import torch
    dv, inp, plan = env
    cfg = inp.cfg
    buf = torch.zeros(cfg.n_vis * cfg.d + 8, dtype=torch.bfloat16, device="cuda")
    x0 = buf[1:1 + cfg.n_vis * cfg.d].view(1, cfg.n_vis, cfg.d)   # 2-byte offset
    pos = torch.zeros((1, 1, cfg.n_vis), dtype=torch.int32, device="cuda")
    k, v = _cache(cfg, torch)
    with pytest.raises(dv.DvError) as e:
        dv.build_visual_memory(plan, x0, pos, k, v)
    assert e.value.code == dv.DV_ERR_ALIGNMENT
    assert bool((k == 0).all())


def test_empty_build_is_noop(env):
    import torch
    dv, inp, plan = env
    cfg = inp.cfg
    x0 = torch.zeros((1, 0, cfg.d), dtype=torch.bfloat16, device="cuda")
    pos = torch.zeros((1, 1, 0), dtype=torch.int32, device="cuda")
    k, v = _cache(cfg, torch)
    dv.build_visual_memory(plan, x0, pos, k, v)
    torch.cuda.synchronize()
    assert bool((k == 0).all()) and dv.plan_status(plan) == dv.DV_OK


def test_bad_stride_rejected(env):
    import torch
    dv, inp, plan = env
    cfg = inp.cfg
    x0 = gu.torch_bf16(inp.x0, "cuda")
    pos = torch.from_numpy(inp.pos).cuda()
    k, v = _cache(cfg, torch)
    kvc = dv.kv_cache_view(k, v)
    kvc.s_seq = kvc.s_seq + 4    # not a multiple of 8 elements
    rc = dv.lib().dv_build_visual_memory(plan.handle, ctypes.c_void_p(x0.data_ptr()), 1, cfg.n_vis,
                                         ctypes.c_void_p(pos.data_ptr()), None, 0,
                                         ctypes.byref(kvc), None)
    assert rc == dv.DV_ERR_ALIGNMENT


def test_gpu_matches_cublas_bf16_sanity(env):
    # Test-only cross-check of layouts against a library path: V with U = 0 and gamma = 1 is
    # W_V RMSNorm(E), computed here with torch (cuBLAS) in fp32 from the same bf16 inputs.
    import torch
    dv, _, _ = env
    cfg = synth.config("tiny", zero_up=True, gamma_sigma=0.0, n_vis=64)
    inp = synth.make_inputs(cfg)
    k, v, plan = gu.run_build(inp)
    x = gu.torch_bf16(inp.x0, "cuda").float().reshape(cfg.tokens, cfg.d)
    n = x * torch.rsqrt((x * x).mean(-1, keepdim=True) + cfg.rms_eps)
    for l in range(cfg.n_layers):
        ref = n @ gu.torch_bf16(inp.Wv[l], "cuda").float().T
        got = v[l, 0].reshape(cfg.n_vis, -1).float()
        assert torch.allclose(got, ref, rtol=2e-2, atol=2e-2 * ref.abs().mean().item())
    dv.free(plan)


def test_host_pipeline_matches_device_build(env):
    # The overlapped host path returns, for every submitted build, exactly the device build's K/V.
    import torch
    dv, inp, plan = env
    cfg = inp.cfg
    k_ref, v_ref, _ = gu.run_build(inp, plan=plan)
    x0_h = gu.torch_bf16(inp.x0, "cpu").pin_memory()
    pos_h = torch.from_numpy(np.ascontiguousarray(inp.pos)).pin_memory()
    x0_b = gu.torch_bf16(synth.normal_bf16(77, 0, inp.x0.shape, 0.0, 1.0), "cpu").pin_memory()
    shape = tuple(k_ref.shape)
    pipe = dv.HostPipeline(plan, tuple(x0_h.shape), tuple(pos_h.shape), shape)
    outs = [(torch.empty(shape, dtype=torch.bfloat16).pin_memory(),
             torch.empty(shape, dtype=torch.bfloat16).pin_memory()) for _ in range(4)]
    for i, (kh, vh) in enumerate(outs):
        pipe.submit(x0_h if i % 2 == 0 else x0_b, pos_h, kh, vh)
    pipe.synchronize()
    for i in (0, 2):
        assert torch.equal(outs[i][0], k_ref.cpu()) and torch.equal(outs[i][1], v_ref.cpu())
    assert not torch.equal(outs[1][0], k_ref.cpu())
    assert torch.equal(outs[1][0], outs[3][0]) and torch.equal(outs[1][1], outs[3][1])
