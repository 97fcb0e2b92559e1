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


def _host_kv(cfg, torch, fill=0.0, pinned=True):
    shape = (cfg.n_layers, cfg.batch, cfg.n_vis, cfg.n_kv_heads, cfg.head_dim)
    k = torch.full(shape, fill, dtype=torch.bfloat16)
    v = torch.full(shape, fill, dtype=torch.bfloat16)
    return (k.pin_memory(), v.pin_memory()) if pinned else (k, v)


def test_host_pipeline_matches_device_build(env):
    # dv_build_visual_memory_host through the C ABI: every submitted build returns in its host
    # buffers exactly the K/V of the device build of the same E (bit for bit), with two staging
    # sets in flight and builds of different E alternating.
    import torch
    dv, inp, plan = env
    cfg = inp.cfg
    k_ref, v_ref, _ = gu.run_build(inp, plan=plan)
    x0_b = gu.torch_bf16(synth.normal_bf16(77, 0, inp.x0.shape, 0.0, 1.0), "cuda")
    pos_d = torch.from_numpy(np.ascontiguousarray(inp.pos)).cuda()
    kb_ref, vb_ref = _cache(cfg, torch)
    dv.build_visual_memory(plan, x0_b, pos_d, kb_ref, vb_ref)
    torch.cuda.synchronize()
    x0_h = gu.torch_bf16(inp.x0, "cpu").pin_memory()
    xb_h = x0_b.cpu().pin_memory()
    pos_h = torch.from_numpy(np.ascontiguousarray(inp.pos)).pin_memory()
    pipe = dv.HostPipeline(plan, cfg.batch, cfg.n_vis, depth=2)
    outs = [_host_kv(cfg, torch, -9.0) for _ in range(5)]
    tickets = [pipe.submit(x0_h if i % 2 == 0 else xb_h, pos_h, kh, vh) for i, (kh, vh) in enumerate(outs)]
    assert tickets == list(range(5))
    for t in tickets:
        pipe.wait(t)
    for i, (kh, vh) in enumerate(outs):
        kr, vr = (k_ref, v_ref) if i % 2 == 0 else (kb_ref, vb_ref)
        assert torch.equal(kh, kr.cpu()) and torch.equal(vh, vr.cpu()), f"build {i}"
    assert dv.plan_status(plan) == dv.DV_OK
    with pytest.raises(dv.DvError):
        pipe.wait(99)                 # not issued yet
    pipe.close()


def test_host_pipeline_join_orders_a_stream(env):
    # join(stream): work enqueued on the stream afterwards sees the finished copy-out; the copy-in
    # of a build starts after the stream's earlier work (here: the host buffer the stream wrote).
    import torch
    dv, inp, plan = env
    cfg = inp.cfg
    k_ref, v_ref, _ = gu.run_build(inp, plan=plan)
    pos_h = torch.from_numpy(np.ascontiguousarray(inp.pos)).pin_memory()
    x0_h = torch.zeros((cfg.batch, cfg.n_vis, cfg.d), dtype=torch.bfloat16).pin_memory()
    x0_d = gu.torch_bf16(inp.x0, "cuda")
    kh, vh = _host_kv(cfg, torch)
    side = torch.cuda.Stream()
    pipe = dv.HostPipeline(plan, cfg.batch, cfg.n_vis, depth=1)
    with torch.cuda.stream(side):
        torch.cuda._sleep(2_000_000)                  # keep the stream busy before its copy
        x0_h.copy_(x0_d, non_blocking=True)           # E reaches the host buffer on the stream
    pipe.submit(x0_h, pos_h, kh, vh, stream=side)
    pipe.join(side)
    done = torch.cuda.Event()
    done.record(side)
    done.synchronize()
    assert torch.equal(kh, k_ref.cpu()) and torch.equal(vh, v_ref.cpu())
    pipe.close()


def test_host_pipeline_dropped_layers_and_pageable_memory():
    # With DV_LAYER_DROP layers the host rows of those layers stay untouched and the others equal
    # the device build's; pageable host buffers give the same bytes as page-locked ones.
    import torch
    import paper_2609_34972_gb300 as dv
    cfg = synth.config("tiny", batch=2, n_vis=40, seed=21)
    inp = synth.make_inputs(cfg)
    modes = [dv.DV_LAYER_ADAPTER, dv.DV_LAYER_DROP, dv.DV_LAYER_IDENTITY, dv.DV_LAYER_ADAPTER]
    k_ref, v_ref, plan = gu.run_build(inp, layer_modes=modes, fill=-5.0)
    x0_h = gu.torch_bf16(inp.x0, "cpu")
    pos_h = torch.from_numpy(np.ascontiguousarray(inp.pos))
    pipe = dv.HostPipeline(plan, cfg.batch, cfg.n_vis)
    for pinned in (True, False):
        kh, vh = _host_kv(cfg, torch, -5.0, pinned)
        xh, ph = (x0_h.pin_memory(), pos_h.pin_memory()) if pinned else (x0_h, pos_h)
        pipe.wait(pipe.submit(xh, ph, kh, vh))
        assert torch.equal(kh, k_ref.cpu()) and torch.equal(vh, v_ref.cpu()), f"pinned={pinned}"
        assert bool((kh[1] == -5.0).all()) and bool((vh[1] == -5.0).all())
    assert dv.plan_status(plan) == dv.DV_OK
    pipe.close()
    dv.free(plan)


def test_host_pipeline_rejects_shapes_beyond_the_plan(env):
    dv, inp, plan = env
    cfg = inp.cfg
    for b, n, depth, code in [(cfg.batch + 1, cfg.n_vis, 2, dv.DV_ERR_UNSUPPORTED_SHAPE),
                              (cfg.batch, cfg.n_vis + 1, 2, dv.DV_ERR_UNSUPPORTED_SHAPE),
                              (cfg.batch, cfg.n_vis, 0, dv.DV_ERR_INVALID_ARG),
                              (cfg.batch, cfg.n_vis, 5, dv.DV_ERR_INVALID_ARG)]:
        with pytest.raises(dv.DvError) as e:
            dv.HostPipeline(plan, b, n, depth=depth)
        assert e.value.code == code


@pytest.mark.parametrize("path", ["chain", "rearranged"])
def test_host_pipeline_mrope_bias_recurrent(path):
    # Three position axes (M-RoPE) and K/V bias through the host entry, with the recurrent
    # adapter (either evaluation of its chain): the host buffers equal the device build of the
    # same inputs.
    import torch
    from dataclasses import replace
    import paper_2609_34972_gb300 as dv
    cfg = gu.small_config("host_mrope", d=512, n_layers=3, n_kv_heads=2, n_heads=4, head_dim=128,
                          rank=64, n_vis=150, batch=2, rope="mrope", rope_theta=1e6,
                          mrope_section=(16, 24, 24), grid=(1, 10, 15), x0_sigma=0.5,
                          bias_sigma=0.02, w_sigma=0.05, seed=131, pos_start=15,
                          adapter="recurrent")
    cfg = replace(cfg, recurrent_path=path)
    inp = synth.make_inputs(cfg)
    k_ref, v_ref, plan = gu.run_build(inp)
    pipe = dv.HostPipeline(plan, cfg.batch, cfg.n_vis, depth=2)
    x0_h = gu.torch_bf16(inp.x0, "cpu").pin_memory()
    pos_h = torch.from_numpy(np.ascontiguousarray(inp.pos)).pin_memory()
    assert tuple(pos_h.shape) == (cfg.batch, 3, cfg.n_vis)
    kh, vh = _host_kv(cfg, torch, -1.0)
    for _ in range(2):
        t = pipe.submit(x0_h, pos_h, kh, vh)
    pipe.wait(t)
    assert torch.equal(kh, k_ref.cpu()) and torch.equal(vh, v_ref.cpu())
    assert dv.plan_status(plan) == dv.DV_OK
    pipe.close()
    dv.free(plan)
