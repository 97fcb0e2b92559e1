"""The allocation-free build entry point (dv_build_visual_memory_noalloc) on a GPU.

Callers that must not allocate device memory while they build use this entry point; it keeps
the build's intermediates in the library's static device array. This file is collected last
so that, if it fails, a run that stops at the first failure has already run every other test.
It must also pass on its own in a fresh process.
"""
import os
import subprocess
import sys

import numpy as np
import pytest

import synth
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dv():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_34972_gb300.build import build_library
    build_library()
    import paper_2609_34972_gb300 as dv
    return dv


def _cache(cfg, torch, fill):
    shape = (cfg.n_layers, cfg.batch, cfg.n_vis, cfg.n_kv_heads, cfg.head_dim)
    return (torch.full(shape, fill, dtype=torch.bfloat16, device="cuda"),
            torch.full(shape, fill, dtype=torch.bfloat16, device="cuda"))


def _check_close(dv, cfg, k_ref, v_ref, k_new, v_new):
    toks = np.arange(cfg.tokens)
    ref_k, ref_v = gu.gather(k_ref, cfg, toks), gu.gather(v_ref, cfg, toks)
    new_k, new_v = gu.gather(k_new, cfg, toks), gu.gather(v_new, cfg, toks)
    ek, ck = gu.parity(new_k, ref_k, cfg.head_dim)
    ev, cv = gu.parity(new_v, ref_v, cfg.head_dim)
    assert ek <= gu.REL_TOL and ev <= gu.REL_TOL, (ek, ev)
    assert ck >= gu.COS_TOL and cv >= gu.COS_TOL, (ck, cv)


@pytest.mark.parametrize("name", ["tiny", "llava15_7b"])
def test_noalloc_matches_build_on_two_calls(dv, name):
    import torch
    cfg = synth.CONFIGS[name]
    inp = synth.make_inputs(cfg)
    plan = dv.memory_plan(gu.dv_config(cfg), gu.device_weights(inp))
    pos = torch.from_numpy(np.ascontiguousarray(inp.pos)).cuda()
    # two calls in a row with different embeddings: the second must not see the first's state
    x0_a = gu.torch_bf16(inp.x0, "cuda")
    x0_b = gu.torch_bf16(synth.normal_bf16(cfg.seed + 100, 0, inp.x0.shape, 0.0, cfg.x0_sigma), "cuda")
    for x0 in (x0_a, x0_b):
        k_ref, v_ref = _cache(cfg, torch, 0.0)
        dv.build_visual_memory(plan, x0, pos, k_ref, v_ref)
        k_new, v_new = _cache(cfg, torch, -3.0)
        dv.build_visual_memory_noalloc(plan, x0, pos, k_new, v_new)
        torch.cuda.synchronize()
        assert dv.plan_status(plan) == dv.DV_OK
        _check_close(dv, cfg, k_ref, v_ref, k_new, v_new)
    dv.free(plan)


def test_noalloc_rejects_builds_over_its_limit(dv):
    import torch
    # Qwen-image shape, 28 layers, rank 128, d = 3584: (28 * 128 + 64) * 2 + 28 * 4 + 4 +
    # (3584 + 64) * 2 = 14708 bytes of intermediates per token, so its 4 x 1296 = 5184-token
    # batch (72.7 MiB) is over the 32 MiB limit while one image (1296 tokens, 18.2 MiB) fits.
    # The plan's own workspace holds 1 token.
    cfg = synth.CONFIGS["qwen25vl_7b_image"]
    inp = synth.make_inputs(cfg)
    plan = dv.memory_plan(gu.dv_config(cfg, max_batch=1, max_n_vis=1), gu.device_weights(inp))
    x0 = gu.torch_bf16(inp.x0, "cuda")
    pos = torch.from_numpy(np.ascontiguousarray(inp.pos)).cuda()
    k, v = _cache(cfg, torch, 0.0)
    with pytest.raises(dv.DvError) as e:
        dv.build_visual_memory_noalloc(plan, x0, pos, k, v)
    assert e.value.code == dv.DV_ERR_UNSUPPORTED_SHAPE
    torch.cuda.synchronize()
    assert bool((k == 0).all()) and bool((v == 0).all())
    # one image of the same batch builds, and matches the planned build of that image
    one = synth.config("qwen25vl_7b_image", batch=1)
    k1, v1 = _cache(one, torch, 0.0)
    dv.build_visual_memory_noalloc(plan, x0[:1], pos[:1], k1, v1)
    plan_ref = dv.memory_plan(gu.dv_config(one), gu.device_weights(inp))
    k2, v2 = _cache(one, torch, 0.0)
    dv.build_visual_memory(plan_ref, x0[:1], pos[:1], k2, v2)
    torch.cuda.synchronize()
    assert dv.plan_status(plan) == dv.DV_OK and dv.plan_status(plan_ref) == dv.DV_OK
    _check_close(dv, one, k2, v2, k1, v1)
    dv.free(plan)
    dv.free(plan_ref)


_FIRST_CALL = r"""
import sys
import numpy as np
import torch
sys.path.insert(0, sys.argv[1])
import synth
import paper_2609_34972_gb300 as dv
from tests import gpu_util as gu
torch.cuda.set_device(0)
cfg = synth.CONFIGS[sys.argv[2]]
inp = synth.make_inputs(cfg)
plan = dv.memory_plan(gu.dv_config(cfg), gu.device_weights(inp))
x0 = gu.torch_bf16(inp.x0, "cuda")
pos = torch.from_numpy(np.ascontiguousarray(inp.pos)).cuda()
shape = (cfg.n_layers, cfg.batch, cfg.n_vis, cfg.n_kv_heads, cfg.head_dim)
k = torch.zeros(shape, dtype=torch.bfloat16, device="cuda")
v = torch.zeros(shape, dtype=torch.bfloat16, device="cuda")
torch.cuda.synchronize()
free_before = torch.cuda.mem_get_info()[0]
dv.build_visual_memory_noalloc(plan, x0, pos, k, v)   # the first build of this process
torch.cuda.synchronize()
free_after = torch.cuda.mem_get_info()[0]
assert dv.plan_status(plan) == dv.DV_OK
print("free before", free_before, "after", free_after)
sys.exit(0 if free_before == free_after else 3)
"""


@pytest.mark.parametrize("name", ["tiny", "llava15_7b"])
def test_first_call_allocates_nothing(dv, name):
    # In a fresh process, the first no-allocation build after dv_memory_plan leaves the device's
    # free memory unchanged: the plan reserved the static array and loaded the build's kernels.
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, "-c", _FIRST_CALL, root, name], capture_output=True,
                       text=True, timeout=600, cwd=root)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
