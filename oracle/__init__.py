"""ORACLE — TEST INFRASTRUCTURE ONLY.

ctypes access to ``oracle.c``, the plain fp64 CPU statement of the visual-memory build
with the embedding adapter (Sec. 3.1 Eqs. 4-5) or the recurrent adapter (Sec. 3.1 Eq. 6),
then Sec. 3.2 Eq. 7 with RMSNorm per App. K and RoPE at the original visual positions.
Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may
import this module. It imports nothing from the
CUDA path, and the CUDA path imports nothing from it.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
# A test may point this module at another build of oracle.c (the mutation tests do).
_LIB_OVERRIDE = os.environ.get("DV_ORACLE_LIB")
_lib = None


class _Cfg(ctypes.Structure):
    _fields_ = [("d", ctypes.c_int), ("n_layers", ctypes.c_int), ("n_kv_heads", ctypes.c_int),
                ("head_dim", ctypes.c_int), ("rank", ctypes.c_int), ("rope", ctypes.c_int),
                ("rope_theta", ctypes.c_double), ("mrope_section", ctypes.c_int * 3),
                ("rms_eps", ctypes.c_double), ("recurrent", ctypes.c_int),
                ("k_norm", ctypes.c_int), ("k_norm_eps", ctypes.c_double)]

_ROPE_MODES = {"1d": 0, "mrope": 1, "mrope_interleaved": 2}


def build(force: bool = False) -> str:
    """Compile ``oracle.c`` (plain C11, OpenMP, fp64) into ``liboracle.so``."""
    src = os.path.join(_HERE, "oracle.c")
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(src):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
                               "-ffp-contract=off", src, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        if _LIB_OVERRIDE:
            lib = ctypes.CDLL(_LIB_OVERRIDE)
        else:
            build()
            lib = ctypes.CDLL(_LIB_PATH)
        vp, i32, i64, dbl = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_double
        lib.oracle_silu.argtypes = [dbl]
        lib.oracle_silu.restype = dbl
        lib.oracle_adapter_row.argtypes = [i32, i32, vp, vp, vp, vp, vp, vp]
        lib.oracle_rmsnorm_row.argtypes = [i32, vp, vp, dbl, vp]
        lib.oracle_project_row.argtypes = [i32, i32, vp, vp, vp, vp]
        lib.oracle_rope_head.argtypes = [i32, dbl, i32, vp, vp, vp]
        lib.oracle_head_rmsnorm.argtypes = [i32, vp, dbl, vp]
        lib.oracle_build_tokens.argtypes = [ctypes.POINTER(_Cfg), vp, i32, vp, vp, vp, vp, vp,
                                            vp, vp, vp, vp, vp, i64, vp, i32, vp, vp, vp, vp, vp]
        lib.oracle_build_tokens.restype = i32
        lib.oracle_num_threads.restype = i32
        lib.oracle_text_attention.argtypes = [i32, i32, i32, i32, i32, i32, vp, vp, vp, vp, vp,
                                              dbl, vp]
        lib.oracle_text_attention.restype = i32
        _lib = lib
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data


def _u16(a):
    return None if a is None else np.ascontiguousarray(a, dtype=np.uint16)


def _f64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


def num_threads() -> int:
    return int(_load().oracle_num_threads())


def silu(u: float) -> float:
    return float(_load().oracle_silu(float(u)))


def adapter_row(x, Dl, Ul):
    """(z, h, m) of the adapter for one row x[d]; Dl bf16 bits [r][d], Ul bf16 bits [d][r]."""
    x = _f64(x)
    Dl, Ul = _u16(Dl), _u16(Ul)
    r, d = Dl.shape
    z, h, m = np.empty(r), np.empty(r), np.empty(d)
    _load().oracle_adapter_row(d, r, _p(x), _p(Dl), _p(Ul), _p(z), _p(h), _p(m))
    return z, h, m


def rmsnorm_row(m, gamma, eps: float):
    m, gamma = _f64(m), _f64(gamma)
    n = np.empty_like(m)
    _load().oracle_rmsnorm_row(m.shape[0], _p(m), _p(gamma), float(eps), _p(n))
    return n


def project_row(W, b, n):
    """W bf16 bits [kv][d], b bf16 bits [kv] or None, n[d] double."""
    W, b, n = _u16(W), _u16(b), _f64(n)
    out = np.empty(W.shape[0])
    _load().oracle_project_row(W.shape[1], W.shape[0], _p(W), _p(b), _p(n), _p(out))
    return out


def rope_head(x, pos3, theta: float, mrope=False, section=(0, 0, 0)):
    """RoPE of one head. ``mrope``: False / "1d", True / "mrope" (contiguous sections) or
    "mrope_interleaved"."""
    x = _f64(x).copy()
    p3 = np.zeros(3)
    p3[:len(np.atleast_1d(pos3))] = np.atleast_1d(pos3)
    sec = (ctypes.c_int * 3)(*section)
    mode = _ROPE_MODES[mrope] if isinstance(mrope, str) else int(bool(mrope))
    _load().oracle_rope_head(x.shape[0], float(theta), mode, ctypes.addressof(sec), _p(p3), _p(x))
    return x


def head_rmsnorm(x, gain, eps: float):
    """Per-head K normalisation of one head x[D_h] with bf16-bit gain [D_h]."""
    x = _f64(x).copy()
    g = _u16(gain)
    _load().oracle_head_rmsnorm(x.shape[0], _p(g), float(eps), _p(x))
    return x


def build_tokens(inp, tokens=None, want=("k", "v"), layers=None):
    """Run the whole build for the given flat token ids (default: every token) and layers
    (default: all, in order).

    ``inp`` carries ``cfg`` (d, n_layers, n_kv_heads, head_dim, rank, rope, rope_theta,
    mrope_section, rms_eps, n_vis, adapter, k_norm, k_norm_eps) and the bf16-bit arrays x0, D,
    U, gamma, Wk, Wv, bk, bv, kgamma and int32 pos [B][P][N_v]. Returns a dict of fp64 arrays: k, v [n][Ls][kv], m, n [n][Ls][d],
    h [n][Ls][r] (Ls = number of evaluated layers), for the names in ``want``.
    """
    cfg = inp.cfg
    c = _Cfg(cfg.d, cfg.n_layers, cfg.n_kv_heads, cfg.head_dim, cfg.rank,
             _ROPE_MODES[cfg.rope], float(cfg.rope_theta),
             (ctypes.c_int * 3)(*cfg.mrope_section), float(cfg.rms_eps),
             1 if getattr(cfg, "adapter", "embedding") == "recurrent" else 0,
             1 if getattr(cfg, "k_norm", False) else 0, float(getattr(cfg, "k_norm_eps", 1e-6)))
    B = inp.x0.shape[0]
    if tokens is None:
        tokens = np.arange(B * cfg.n_vis, dtype=np.int64)
    tokens = np.ascontiguousarray(tokens, dtype=np.int64)
    lay = None if layers is None else np.ascontiguousarray(layers, dtype=np.int32)
    nt, kv = tokens.shape[0], cfg.n_kv_heads * cfg.head_dim
    L = cfg.n_layers if lay is None else lay.shape[0]
    out = {}
    shapes = {"k": (nt, L, kv), "v": (nt, L, kv), "m": (nt, L, cfg.d), "h": (nt, L, cfg.rank),
              "n": (nt, L, cfg.d)}
    for name in want:
        out[name] = np.empty(shapes[name])
    arrs = [_u16(inp.x0), np.ascontiguousarray(inp.pos, dtype=np.int32), _u16(inp.D), _u16(inp.U),
            _u16(inp.gamma), _u16(inp.Wk), _u16(inp.Wv), _u16(inp.bk), _u16(inp.bv),
            _u16(getattr(inp, "kgamma", None))]
    rc = _load().oracle_build_tokens(
        ctypes.byref(c), _p(arrs[0]), cfg.n_vis, _p(arrs[1]), _p(arrs[2]), _p(arrs[3]),
        _p(arrs[4]), _p(arrs[5]), _p(arrs[6]), _p(arrs[7]), _p(arrs[8]), _p(arrs[9]), _p(tokens), nt,
        _p(lay), 0 if lay is None else int(lay.shape[0]), _p(out.get("k")), _p(out.get("v")), _p(out.get("m")), _p(out.get("h")), _p(out.get("n")))
    if rc != 0:
        raise ValueError("oracle_build_tokens rejected its arguments")
    return out


def text_attention(q, k, v, n_keys, q_slot, scale: float):
    """Causal text-query attention over cache slots (Sec. 3.2): q [B][Hq][Nt][D], k, v
    [B][S][Hkv][D] (fp64-convertible), n_keys int [B], q_slot int [B][Nt]. Returns fp64
    [B][Hq][Nt][D]."""
    q, k, v = _f64(q), _f64(k), _f64(v)
    B, Hq, Nt, D = q.shape
    S, Hkv = k.shape[1], k.shape[2]
    nk = np.ascontiguousarray(n_keys, dtype=np.int32)
    qs = np.ascontiguousarray(q_slot, dtype=np.int32)
    out = np.empty_like(q)
    rc = _load().oracle_text_attention(B, Hq, Hkv, Nt, S, D, _p(q), _p(k), _p(v), _p(nk), _p(qs),
                                       float(scale), _p(out))
    if rc != 0:
        raise ValueError("oracle_text_attention rejected its arguments")
    return out
