"""Writes ``oracle_builds.json``: sampled K/V cache values of three small seeded builds, as the
fp64 oracle computes them.

The stored values come from the oracle alone (the embedding adapter of Sec. 3.1 Eqs. 4-5, the
recurrent adapter of Sec. 3.1 Eq. 6, then Sec. 3.2 Eq. 7: RMSNorm, the K/V projection and RoPE
at the original visual positions). The cases cover both adapters, both head widths, 1-D RoPE
and interleaved M-RoPE, the K/V bias and the per-head K norm. Each case records a SHA-256 of its
seeded inputs, so a change of the input generator shows up as such and not as a parity failure.

Run from the repository root:  python tests/golden/make_golden.py
"""
from __future__ import annotations

import dataclasses
import hashlib
import json
import os
import sys

import numpy as np

_ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
if _ROOT not in sys.path:
    sys.path.insert(0, _ROOT)

import oracle  # noqa: E402
import synth   # noqa: E402

OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "oracle_builds.json")


def cases():
    """(case name, config, sampled flat token ids, sampled KV heads, sampled channels per head)."""
    tiny = synth.CONFIGS["tiny"]
    qwen3_like = dataclasses.replace(
        tiny, name="qwen3_like", d=512, n_layers=3, n_heads=4, n_kv_heads=2, head_dim=128,
        rank=24, n_vis=64, batch=2, rope="mrope_interleaved", rope_theta=5e6,
        mrope_section=(24, 20, 20), grid=(1, 8, 8), x0_sigma=0.5, bias_sigma=0.02,
        k_norm=True, seed=7, pos_start=15)
    ch64 = [0, 1, 31, 32, 33, 63]            # both rotary halves, pair partners 0/32 and 1/33
    ch128 = [0, 1, 63, 64, 65, 127]
    return [
        ("tiny_embedding", tiny, [0, 29, 63], [0, 3, 7], ch64),
        ("tiny_recurrent", dataclasses.replace(tiny, name="tiny_recurrent", adapter="recurrent"), [0, 29, 63], [0, 3, 7], ch64),
        ("qwen3_like", qwen3_like, [0, 45, 64, 127], [0, 1], ch128),
    ]


def input_digest(inp) -> str:
    h = hashlib.sha256()
    for name in ("x0", "D", "U", "gamma", "Wk", "Wv", "bk", "bv", "kgamma", "pos"):
        a = getattr(inp, name)
        h.update(name.encode())
        if a is not None:
            h.update(np.ascontiguousarray(a).tobytes())
    return h.hexdigest()


def sample(cfg, out, heads, channels):
    """Per (token, layer, head): the head row's rms and the values at the sampled channels."""
    n, L, _ = out.shape
    rows = out.reshape(n, L, cfg.n_kv_heads, cfg.head_dim)[:, :, heads]
    rms = np.sqrt(np.mean(rows * rows, axis=-1))
    return rms, rows[..., channels]


def main():
    doc = {"source": "fp64 oracle: Sec. 3.1 Eqs. 4-6 and Sec. 3.2 Eq. 7; written by make_golden.py",
           "cases": []}
    for name, cfg, toks, heads, chans in cases():
        inp = synth.make_inputs(cfg)
        ref = oracle.build_tokens(inp, np.asarray(toks))
        k_rms, k_val = sample(cfg, ref["k"], heads, chans)
        v_rms, v_val = sample(cfg, ref["v"], heads, chans)
        doc["cases"].append({
            "name": name,
            "config": {f.name: getattr(cfg, f.name) for f in dataclasses.fields(cfg)
                       if f.name != "description"},
            "inputs_sha256": input_digest(inp), "tokens": toks, "heads": heads, "channels": chans,
            "k_rms": k_rms.tolist(), "k": k_val.tolist(), "v_rms": v_rms.tolist(), "v": v_val.tolist(),
        })
    with open(OUT, "w") as f:
        json.dump(doc, f, indent=None, separators=(",", ":"))
        f.write("\n")
    print(f"wrote {OUT} ({os.path.getsize(OUT)} bytes)")


if __name__ == "__main__":
    main()
