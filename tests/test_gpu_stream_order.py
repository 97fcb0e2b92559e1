"""Stream order around the build: the build's kernels start early (programmatic dependent launch)
and wait for earlier work before they touch memory. These cases interleave builds with ordinary
stream work that writes the build's inputs right before it, reads its cache right after it, and
with a second plan whose builds share nothing but the stream. Every result must equal the one
of an isolated build bit for bit, on both K/V engines and the recurrent chain.
"""
from dataclasses import replace

import numpy as np
import pytest

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


def _isolated(inp, plan, x0, pos):
    import torch
    import paper_2609_34972_gb300 as dv
    cfg = inp.cfg
    shape = (cfg.n_layers, cfg.batch, cfg.n_vis, cfg.n_kv_heads, cfg.head_dim)
    k = torch.zeros(shape, dtype=torch.bfloat16, device="cuda")
    v = torch.zeros_like(k)
    torch.cuda.synchronize()
    dv.build_visual_memory(plan, x0, pos, k, v)
    torch.cuda.synchronize()
    return k.clone(), v.clone()


@pytest.mark.parametrize("name,kw", [
    ("so_wm", dict(n_vis=300, batch=1)),                                   # weights-as-M K/V
    ("so_tm", dict(n_vis=256, batch=2)),                                   # tokens-as-M K/V
    ("so_rec", dict(n_vis=200, batch=1, adapter="recurrent", w_sigma=0.05)),  # on-chip chain
])
def test_inputs_written_and_cache_read_by_neighbouring_stream_work(name, kw):
    import torch
    import paper_2609_34972_gb300 as dv
    cfg = gu.small_config(name, d=512, n_layers=3, n_kv_heads=2, n_heads=4, head_dim=128, rank=64,
                          x0_sigma=0.5, seed=61, pos_start=35, **kw)
    inp_a = synth.make_inputs(cfg)
    inp_b = synth.make_inputs(replace(cfg, seed=62))  # only its x0 is used (with plan a's weights)
    plan = dv.memory_plan(gu.dv_config(cfg), gu.device_weights(inp_a))
    xa = gu.torch_bf16(inp_a.x0, "cuda")
    xb = gu.torch_bf16(inp_b.x0, "cuda")
    pos = torch.from_numpy(np.ascontiguousarray(inp_a.pos)).cuda()
    ka, va = _isolated(inp_a, plan, xa, pos)
    kb, vb = _isolated(inp_a, plan, xb, pos)
    assert not torch.equal(ka, kb)

    # a second, unrelated plan whose builds run on the same stream in between
    other = synth.make_inputs(synth.config("tiny", n_vis=100, seed=63))
    plan_o = dv.memory_plan(gu.dv_config(other.cfg), gu.device_weights(other))
    xo = gu.torch_bf16(other.x0, "cuda")
    po = torch.from_numpy(np.ascontiguousarray(other.pos)).cuda()
    ko_ref, vo_ref = _isolated(other, plan_o, xo, po)
    so = (other.cfg.n_layers, other.cfg.batch, other.cfg.n_vis, other.cfg.n_kv_heads, other.cfg.head_dim)
    ko = torch.zeros(so, dtype=torch.bfloat16, device="cuda")
    vo = torch.zeros_like(ko)

    x0 = torch.empty_like(xa)
    shape = tuple(ka.shape)
    k = torch.zeros(shape, dtype=torch.bfloat16, device="cuda")
    v = torch.zeros_like(k)
    copies = []
    for i in range(12):
        src = xa if i % 2 == 0 else xb
        x0.copy_(src)                         # written by the stream right before the build
        dv.build_visual_memory(plan, x0, pos, k, v)
        copies.append((k.clone(), v.clone()))  # read by the stream right after it
        k.fill_(-1.0)                         # and overwritten before the next build
        v.fill_(-1.0)
        dv.build_visual_memory(plan_o, xo, po, ko, vo)
    torch.cuda.synchronize()
    assert dv.plan_status(plan) == dv.DV_OK and dv.plan_status(plan_o) == dv.DV_OK
    for i, (kc, vc) in enumerate(copies):
        kr, vr = (ka, va) if i % 2 == 0 else (kb, vb)
        assert torch.equal(kc, kr) and torch.equal(vc, vr), f"build {i} differs from its isolated run"
    assert torch.equal(ko, ko_ref) and torch.equal(vo, vo_ref)
    dv.free(plan_o)
    dv.free(plan)
