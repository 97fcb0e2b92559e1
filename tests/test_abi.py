"""The C-ABI library without a GPU: it builds for sm_103a, loads, exports every entry point
declared in include/dv.h, and rejects bad configurations before touching the device."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def dv():
    from paper_2609_34972_gb300.build import build_library
    build_library()
    import paper_2609_34972_gb300 as dv
    return dv


def _declared():
    src = open(os.path.join(ROOT, "include", "dv.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(dv_[a-z_]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(dv):
    names = _declared()
    assert "dv_memory_plan" in names and "dv_build_visual_memory" in names and "dv_free" in names
    lib = dv.lib()
    for n in names:
        assert hasattr(lib, n), f"{n} declared in dv.h but not exported"
    assert sorted(dv.EXPORTED) == names


def test_error_strings(dv):
    for code in range(0, 8):
        assert dv.error_string(code) and dv.error_string(code) != "unknown status"
    assert dv.error_string(99) == "unknown status"


def test_null_arguments_rejected(dv):
    lib = dv.lib()
    assert lib.dv_memory_plan(None, None, None, None) == dv.DV_ERR_INVALID_ARG
    h = ctypes.c_void_p()
    assert lib.dv_memory_plan(None, None, None, ctypes.byref(h)) == dv.DV_ERR_INVALID_ARG
    assert lib.dv_build_visual_memory(None, None, 1, 1, None, None, 0, None, None) == dv.DV_ERR_INVALID_ARG
    assert lib.dv_plan_status(None) == dv.DV_ERR_INVALID_ARG
    assert lib.dv_debug_copy_memory(None, 0, None, None) == dv.DV_ERR_INVALID_ARG
    lib.dv_free(None)  # no-op
    pipe = ctypes.c_void_p(7)
    assert lib.dv_host_pipeline_create(None, 1, 1, 2, ctypes.byref(pipe)) == dv.DV_ERR_INVALID_ARG
    assert pipe.value is None                       # set to NULL on error
    assert lib.dv_host_pipeline_create(None, 1, 1, 2, None) == dv.DV_ERR_INVALID_ARG
    assert lib.dv_build_visual_memory_host(None, None, None, None, None, None, None) == dv.DV_ERR_INVALID_ARG
    assert lib.dv_host_pipeline_wait(None, 0) == dv.DV_ERR_INVALID_ARG
    assert lib.dv_host_pipeline_join(None, None) == dv.DV_ERR_INVALID_ARG
    lib.dv_host_pipeline_free(None)  # no-op
    with pytest.raises(ValueError):
        dv.make_config(512, 4, 8, 64, 16, adapter="stacked")


@pytest.mark.parametrize("field,value,code", [
    ("d", 100, 2), ("d", 0, 1), ("rank", 0, 1), ("rank", 300, 2), ("head_dim", 96, 2),
    ("n_layers", -1, 1), ("act", 3, 1), ("rope", 5, 1), ("max_batch", 0, 1),
    ("rope_theta", -1.0, 1), ("rms_eps", -1e-6, 1), ("n_kv_heads", 129, 2),
    ("adapter", 2, 1), ("adapter", -1, 1), ("rope", 3, 1), ("k_norm", 2, 1),
    ("k_norm_eps", -1.0, 1), ("split_chain", 2, 1), ("split_chain", 1, 1),
    ("recurrent_path", 3, 1), ("recurrent_path", -1, 1), ("recurrent_path", 2, 1),
])
def test_bad_config_rejected_before_device(dv, field, value, code):
    cfg = dv.make_config(512, 4, 8, 64, 16, max_batch=1, max_n_vis=64)
    setattr(cfg, field, value)
    w = dv.DvWeights(*([ctypes.c_void_p(256)] * 5 + [None, None, None]))
    h = ctypes.c_void_p()
    assert dv.lib().dv_memory_plan(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(h)) == code
    assert not h.value


@pytest.mark.parametrize("d,split,path,code", [
    (576, 0, "rearranged", 2),   # the rearranged chain's slices need d % 128 == 0
    (512, 0, "bogus", None),     # refused by the binding
])
def test_recurrent_path_rules(dv, d, split, path, code):
    if code is None:
        with pytest.raises(ValueError):
            dv.make_config(d, 4, 8, 64, 16, adapter="recurrent", recurrent_path=path)
        return
    cfg = dv.make_config(d, 4, 8, 64, 16, max_batch=1, max_n_vis=64, adapter="recurrent",
                         split_chain=bool(split), recurrent_path=path)
    w = dv.DvWeights(*([ctypes.c_void_p(256)] * 5 + [None, None, None]))
    h = ctypes.c_void_p()
    assert dv.lib().dv_memory_plan(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(h)) == code
    assert not h.value


def test_mrope_sections_must_cover_half_head(dv):
    cfg = dv.make_config(512, 4, 8, 128, 16, rope="mrope", mrope_section=(16, 24, 20),
                         max_batch=1, max_n_vis=64)
    w = dv.DvWeights(*([ctypes.c_void_p(256)] * 5 + [None, None, None]))
    h = ctypes.c_void_p()
    assert dv.lib().dv_memory_plan(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(h)) == 2


@pytest.mark.parametrize("sections", [(16, 24, 24), (20, 22, 22), (10, 27, 27)])
def test_interleaved_mrope_sections_must_match_the_layout(dv, sections):
    # The interleaved layout over 64 pairs gives h the pairs j = 1 mod 3 below 3 s_h and w the
    # pairs j = 2 mod 3 below 3 s_w. These sections sum to 64 but the layout cannot give each
    # axis its count (e.g. (16, 24, 24) would need pair 71), so the plan is refused before
    # any device work. (24, 20, 20), the Qwen3-VL layout, is accepted on the GPU.
    cfg = dv.make_config(512, 4, 8, 128, 16, rope="mrope_interleaved", mrope_section=sections,
                         max_batch=1, max_n_vis=64)
    w = dv.DvWeights(*([ctypes.c_void_p(256)] * 5 + [None, None, None, None]))
    h = ctypes.c_void_p()
    rc = dv.lib().dv_memory_plan(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(h))
    assert rc == dv.DV_ERR_UNSUPPORTED_SHAPE and not h.value


def test_k_norm_needs_its_gain(dv):
    cfg = dv.make_config(512, 4, 8, 64, 16, max_batch=1, max_n_vis=64, k_norm=True)
    w = dv.DvWeights(*([ctypes.c_void_p(256)] * 5 + [None, None, None, None]))
    h = ctypes.c_void_p()
    assert dv.lib().dv_memory_plan(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(h)) == 1


def test_missing_weights_rejected(dv):
    cfg = dv.make_config(512, 4, 8, 64, 16, max_batch=1, max_n_vis=64, has_kv_bias=True)
    w = dv.DvWeights(*([ctypes.c_void_p(256)] * 5 + [None, None, None]))   # bias asked for, not given
    h = ctypes.c_void_p()
    assert dv.lib().dv_memory_plan(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(h)) == 1


def test_binding_fails_loudly_without_library(dv, monkeypatch):
    monkeypatch.setattr(dv, "_lib", None)
    monkeypatch.setattr(dv, "LIB_PATH", "/nonexistent/libdv.so")
    with pytest.raises(RuntimeError):
        dv.lib()


def test_kv_width_must_be_multiple_of_128(dv):
    # The K/V kernel pairs 128 K channels with the same 128 V channels per CTA pair.
    cfg = dv.make_config(512, 4, 3, 64, 16, max_batch=1, max_n_vis=64)   # kv = 192
    w = dv.DvWeights(*([ctypes.c_void_p(256)] * 5 + [None, None, None]))
    h = ctypes.c_void_p()
    assert dv.lib().dv_memory_plan(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(h)) == 2


@pytest.mark.parametrize("modes", [[0, 3, 0, 0], [2, 2, 2, 2]])
def test_bad_layer_modes_rejected(dv, modes):
    # an unknown mode, or every layer dropped, is an argument error found before the device
    cfg = dv.make_config(512, 4, 8, 64, 16, max_batch=1, max_n_vis=64)
    arr = (ctypes.c_ubyte * 4)(*modes)
    w = dv.DvWeights(*([ctypes.c_void_p(256)] * 5 + [None, None, ctypes.cast(arr, ctypes.c_void_p)]))
    h = ctypes.c_void_p()
    assert dv.lib().dv_memory_plan(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(h)) == 1


def test_text_attention_validates_before_device(dv):
    lib = dv.lib()
    kvc = dv.DvKVCache(256, 512, 8 * 64 * 100, 8 * 64 * 100, 8 * 64, 64)
    p = ctypes.c_void_p(1024)
    args = lambda **kw: [kw.get("q", p), kw.get("batch", 1), kw.get("hq", 8), kw.get("hkv", 8),
                         kw.get("nt", 4), kw.get("hd", 64), ctypes.byref(kw.get("cache", kvc)),
                         kw.get("layer", 0), kw.get("max_keys", 100), p, p,
                         ctypes.c_float(kw.get("scale", 0.125)), kw.get("out", p), None]
    assert lib.dv_text_attention(*args(batch=0)) == dv.DV_OK          # empty: nothing to do
    assert lib.dv_text_attention(*args(q=None)) == dv.DV_ERR_INVALID_ARG
    assert lib.dv_text_attention(*args(hq=6, hkv=4)) == dv.DV_ERR_INVALID_ARG
    assert lib.dv_text_attention(*args(scale=0.0)) == dv.DV_ERR_INVALID_ARG
    assert lib.dv_text_attention(*args(hd=96)) == dv.DV_ERR_UNSUPPORTED_SHAPE
    assert lib.dv_text_attention(*args(q=ctypes.c_void_p(1026))) == dv.DV_ERR_ALIGNMENT
    bad = dv.DvKVCache(256, 512, 8 * 64 * 100, 8 * 64 * 100, 8 * 64 + 4, 64)
    assert lib.dv_text_attention(*args(cache=bad)) == dv.DV_ERR_ALIGNMENT
