"""Helpers for the GPU tests: move seeded inputs to the device, run the C-ABI build through the
Python binding, gather cache rows, and apply the parity bar against the oracle.

Parity bar (bf16 inputs, fp32 accumulation): for every K and V element,
    |gpu - oracle| / max(|oracle|, rms of the oracle's head row) <= 2e-2,
the plain relative error |gpu - oracle| / |oracle| <= 2e-2 wherever |oracle| is at least its
head row's rms (reported beside it), and per (token, layer) the cosine between the GPU and
oracle kv vectors is >= 0.9999, separately for K and V.
"""
from __future__ import annotations

import json
import os

import numpy as np

import synth

REL_TOL = 2e-2
COS_TOL = 0.9999


def torch_bf16(bits, device):
    import torch
    a = np.ascontiguousarray(bits, dtype=np.uint16)
    return torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).to(device)


def device_weights(inp, device="cuda"):
    w = {n: torch_bf16(getattr(inp, n), device) for n in ("D", "U", "gamma", "Wk", "Wv")}
    if inp.bk is not None:
        w["bk"] = torch_bf16(inp.bk, device)
        w["bv"] = torch_bf16(inp.bv, device)
    if getattr(inp, "kgamma", None) is not None:
        w["kgamma"] = torch_bf16(inp.kgamma, device)
    return w


def dv_config(cfg, max_batch=None, max_n_vis=None):
    import paper_2609_34972_gb300 as dv
    return dv.make_config(cfg.d, cfg.n_layers, cfg.n_kv_heads, cfg.head_dim, cfg.rank,
                          rope=cfg.rope, rope_theta=cfg.rope_theta,
                          mrope_section=cfg.mrope_section, rms_eps=cfg.rms_eps,
                          max_batch=max_batch or cfg.batch, max_n_vis=max_n_vis or cfg.n_vis,
                          has_kv_bias=cfg.bias_sigma > 0, adapter=cfg.adapter,
                          k_norm=cfg.k_norm, k_norm_eps=cfg.k_norm_eps,
                          split_chain=getattr(cfg, "split_chain", False),
                          recurrent_path=getattr(cfg, "recurrent_path", "auto"))


def run_build(inp, plan=None, seq_len=None, batch_cache=None, slot=None, slot0=0, fill=0.0,
              layer_modes=None, noalloc=False):
    """Plan (unless given) and build into a fresh [L, B_c, S, H, D_h] cache; returns (k, v, plan)."""
    import torch
    import paper_2609_34972_gb300 as dv
    cfg = inp.cfg
    dev = torch.device("cuda")
    if plan is None:
        plan = dv.memory_plan(dv_config(cfg), device_weights(inp, dev), layer_modes=layer_modes)
    S = seq_len or cfg.n_vis
    Bc = batch_cache or cfg.batch
    shape = (cfg.n_layers, Bc, S, cfg.n_kv_heads, cfg.head_dim)
    k = torch.full(shape, fill, dtype=torch.bfloat16, device=dev)
    v = torch.full(shape, fill, dtype=torch.bfloat16, device=dev)
    x0 = torch_bf16(inp.x0, dev)
    pos = torch.from_numpy(np.ascontiguousarray(inp.pos)).to(dev)
    sl = None if slot is None else torch.from_numpy(np.ascontiguousarray(slot, np.int32)).to(dev)
    build = dv.build_visual_memory_noalloc if noalloc else dv.build_visual_memory
    build(plan, x0, pos, k, v, slot=sl, slot0=slot0)
    torch.cuda.synchronize()
    assert dv.plan_status(plan) == dv.DV_OK
    return k, v, plan


def gather(cache, cfg, tokens, slot=None, slot0=0):
    """fp64 [n, L, kv] rows of the cache for flat token ids (b * n_vis + i)."""
    import torch
    tokens = np.asarray(tokens)
    b = tokens // cfg.n_vis
    i = tokens % cfg.n_vis
    s = slot.reshape(-1)[tokens] if slot is not None else slot0 + i
    idx_b = torch.as_tensor(b, device=cache.device)
    idx_s = torch.as_tensor(s, device=cache.device)
    rows = cache[:, idx_b, idx_s]                       # [L, n, H, D]
    return rows.permute(1, 0, 2, 3).reshape(len(tokens), cfg.n_layers, -1).double().cpu().numpy()


def parity(g, o, head_dim):
    """(max scaled error, min cosine) of GPU g against oracle o, both [n, L, kv]."""
    e = parity_stats(g, o, head_dim)
    return e["scaled"], e["cos"]


def parity_stats(g, o, head_dim):
    """Error figures of GPU g against oracle o, both [n, L, kv]:
    scaled  max |g - o| / max(|o|, rms of o's head row)  (the bar)
    raw     max |g - o| / |o| over the elements with |o| >= their head row's rms (the plain
            relative error where it is meaningful; these elements' scaled error is the same)
    cos     min per-(token, layer) cosine over the kv vector
    small   fraction of elements with |o| < rms, where the scaled error is the looser one."""
    n, L, kv = o.shape
    oh = o.reshape(n, L, kv // head_dim, head_dim)
    gh = g.reshape(n, L, kv // head_dim, head_dim)
    rms = np.sqrt(np.mean(oh * oh, axis=-1, keepdims=True))
    diff = np.abs(gh - oh)
    err = diff / np.maximum(np.abs(oh), rms)
    big = np.abs(oh) >= rms
    raw = float((diff[big] / np.abs(oh[big])).max()) if big.any() else 0.0
    cos = np.sum(g * o, axis=-1) / (np.linalg.norm(g, axis=-1) * np.linalg.norm(o, axis=-1))
    return {"scaled": float(err.max()), "raw": raw, "cos": float(cos.min()),
            "small": float(1.0 - big.mean())}


def assert_parity(gk, gv, ok, ov, head_dim, label="", rel_tol=REL_TOL, cos_tol=COS_TOL):
    sk = parity_stats(gk, ok, head_dim)
    sv = parity_stats(gv, ov, head_dim)
    ek, ck, ev, cv = sk["scaled"], sk["cos"], sv["scaled"], sv["cos"]
    msg = (f"{label}: K max err {ek:.3e} (raw {sk['raw']:.3e}) min cos {ck:.7f}; "
           f"V max err {ev:.3e} (raw {sv['raw']:.3e}) min cos {cv:.7f}")
    log = os.environ.get("DV_PARITY_LOG")
    if log:
        with open(log, "a") as f:
            f.write(json.dumps({"case": label, "k_max_err": ek, "k_raw_err": sk["raw"],
                                "k_min_cos": ck, "k_small_frac": sk["small"], "v_max_err": ev,
                                "v_raw_err": sv["raw"], "v_min_cos": cv,
                                "v_small_frac": sv["small"], "n_tokens": int(ok.shape[0])}) + "\n")
    assert np.all(np.isfinite(gk)) and np.all(np.isfinite(gv)), msg
    assert ek <= rel_tol and ev <= rel_tol, msg
    assert sk["raw"] <= rel_tol and sv["raw"] <= rel_tol, msg
    assert ck >= cos_tol and cv >= cos_tol, msg
    return ek, ev, ck, cv


def sample_tokens(T, n=48, seed=0):
    """Tokens spread over every 128-row tile, always including both ends and tile borders."""
    rng = np.random.default_rng(seed)
    fixed = {0, 1, T - 1, T - 2, min(127, T - 1), min(128, T - 1), (T - 1) // 128 * 128}
    picks = set(int(x) for x in rng.integers(0, T, size=n)) | fixed
    return np.array(sorted(p for p in picks if 0 <= p < T), dtype=np.int64)


def small_config(name, **kw):
    base = synth.CONFIGS["tiny"]
    from dataclasses import replace
    return replace(base, name=name, **kw)
