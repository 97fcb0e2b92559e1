"""Seeded synthetic workloads for the visual-memory build.

This module draws inputs only. It holds none of the method's arithmetic: the
oracle (``oracle/``) and the CUDA path (``paper_2609_34972_gb300``) both take
what it returns as their inputs, and it imports neither of them.

Workload shapes follow the five synthetic configurations the library is
measured on (LLaVA- and Qwen2.5-VL-shaped backbones, whose visual embeddings
stand in for the image and video benchmarks the paper evaluates on, Sec. 4.1).
No dataset item, model weight or trained adapter is used: every tensor is drawn
from the counter-based generator in ``gen.c``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass, field, replace

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "libdvgen.so")
_lib = None

# Counter streams, one per tensor, so that changing one shape never shifts another tensor.
STREAM_X0, STREAM_D, STREAM_U, STREAM_GAMMA, STREAM_WK, STREAM_WV, STREAM_BK, STREAM_BV = range(8)
STREAM_KGAMMA = 8


def build(force: bool = False) -> str:
    """Compile ``gen.c`` into ``libdvgen.so`` (plain C, OpenMP, no FP contraction)."""
    src = os.path.join(_HERE, "gen.c")
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(src):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
                               "-ffp-contract=off", src, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB_PATH)
        u64, i64, dbl = ctypes.c_uint64, ctypes.c_int64, ctypes.c_double
        vp = ctypes.c_void_p
        lib.dvgen_normal_bf16.argtypes = [u64, u64, u64, i64, dbl, dbl, vp]
        lib.dvgen_normal_f64.argtypes = [u64, u64, u64, i64, dbl, dbl, vp]
        lib.dvgen_ar1_frames_bf16.argtypes = [u64, u64, i64, i64, dbl, dbl, vp]
        lib.dvgen_bf16_to_f32.argtypes = [vp, i64, vp]
        lib.dvgen_f64_to_bf16.argtypes = [dbl]
        lib.dvgen_f64_to_bf16.restype = ctypes.c_uint16
        lib.dvgen_key.argtypes = [u64, u64]
        lib.dvgen_key.restype = u64
        _lib = lib
    return _lib


def normal_bf16(seed: int, stream: int, shape, mean: float = 0.0, sigma: float = 1.0,
                offset: int = 0) -> np.ndarray:
    """bf16 bit patterns (uint16) of ``mean + sigma * N(0,1)`` drawn at counters offset.."""
    n = int(np.prod(shape))
    out = np.empty(n, dtype=np.uint16)
    _load().dvgen_normal_bf16(seed, stream, offset, n, mean, sigma, out.ctypes.data)
    return out.reshape(shape)


def normal_f64(seed: int, stream: int, shape, mean: float = 0.0, sigma: float = 1.0,
               offset: int = 0) -> np.ndarray:
    n = int(np.prod(shape))
    out = np.empty(n, dtype=np.float64)
    _load().dvgen_normal_f64(seed, stream, offset, n, mean, sigma, out.ctypes.data)
    return out.reshape(shape)


def ar1_frames_bf16(seed: int, stream: int, n_frames: int, per_frame: int, rho: float,
                    scale: float) -> np.ndarray:
    out = np.empty(n_frames * per_frame, dtype=np.uint16)
    _load().dvgen_ar1_frames_bf16(seed, stream, n_frames, per_frame, rho, scale, out.ctypes.data)
    return out


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32."""
    bits = np.ascontiguousarray(bits, dtype=np.uint16)
    return (bits.astype(np.uint32) << 16).view(np.float32)


def f64_to_bf16(values) -> np.ndarray:
    """Round doubles to bf16 bit patterns with the generator's rule (f64 -> f32 -> bf16, RNE)."""
    f = np.ascontiguousarray(values, dtype=np.float64).astype(np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    r = ((u + 0x7FFF + lsb) >> 16).astype(np.uint16)
    nan = np.isnan(f)
    if nan.any():
        r[nan] = 0x7FC0
    return r


# --------------------------------------------------------------------------------------------
# Workload configurations
# --------------------------------------------------------------------------------------------

@dataclass(frozen=True)
class Config:
    name: str
    d: int
    n_layers: int
    n_heads: int          # query heads of the backbone (informational: the build writes K/V only)
    n_kv_heads: int
    head_dim: int
    rank: int
    n_vis: int
    batch: int
    rope: str             # "1d", "mrope" (contiguous sections) or "mrope_interleaved"
    rope_theta: float
    mrope_section: tuple = (0, 0, 0)
    rms_eps: float = 1e-6
    x0_sigma: float = 0.5
    w_sigma: float = 0.02
    gamma_sigma: float = 0.02   # gamma = 1 + N(0, gamma_sigma); 0 gives gamma = 1 exactly
    bias_sigma: float = 0.0     # > 0: K/V bias ~ N(0, bias_sigma); 0: no bias
    zero_up: bool = False       # zero-initialised up-projection (adapter starts as the identity)
    seed: int = 0
    pos_start: int = 0
    grid: tuple = ()            # (frames, rows, cols) of the visual grid, M-RoPE only
    ar1_rho: float = 0.0        # > 0: frame-correlated x0 (video), per token-in-frame element
    adapter: str = "embedding"  # "embedding" (Sec. 3.1 Eq. 5) or "recurrent" (Sec. 3.1 Eq. 6)
    k_norm: bool = False        # per-head RMSNorm of K before RoPE (Qwen3-VL backbones)
    k_norm_eps: float = 1e-6
    k_norm_sigma: float = 0.1   # per-head K-norm gain = 1 + N(0, k_norm_sigma)
    split_chain: bool = False   # recurrent adapter: hi + lo bf16 operands in the chain's GEMMs
    recurrent_path: str = "auto"  # recurrent adapter: "auto", "chain" or "rearranged"
    description: str = ""

    @property
    def kv(self) -> int:
        return self.n_kv_heads * self.head_dim

    @property
    def tokens(self) -> int:
        return self.batch * self.n_vis

    @property
    def n_pos(self) -> int:
        return 1 if self.rope == "1d" else 3

    def flops(self) -> float:
        """Plain-definition FLOPs of one build: 4*d*r + 4*d*kv per token and layer."""
        return float(self.tokens) * self.n_layers * (4.0 * self.d * self.rank + 4.0 * self.d * self.kv)

    def min_bytes(self) -> float:
        """Least HBM traffic of one build: weights once, x0 in, positions in, K/V out."""
        w = self.n_layers * (2 * self.d * self.rank + self.d + 2 * self.kv * self.d) * 2
        return float(w + self.tokens * self.d * 2 + self.tokens * self.n_pos * 4
                     + self.tokens * self.n_layers * 2 * self.kv * 2)


CONFIGS = {
    "tiny": Config(
        name="tiny", d=512, n_layers=4, n_heads=8, n_kv_heads=8, head_dim=64, rank=16,
        n_vis=64, batch=1, rope="1d", rope_theta=10000.0, rms_eps=1e-6, x0_sigma=1.0,
        seed=0, pos_start=5,
        description="d=512, L=4, 8x64 MHA, r=16, N_v=64, batch 1, 1-D RoPE at positions 5..68"),
    "llava15_7b": Config(
        name="llava15_7b", d=4096, n_layers=32, n_heads=32, n_kv_heads=32, head_dim=128,
        rank=64, n_vis=576, batch=1, rope="1d", rope_theta=10000.0, rms_eps=1e-5,
        x0_sigma=0.5, seed=1, pos_start=35,
        description="LLaVA-1.5-7B-shaped: d=4096, L=32, 32x128 MHA, r=64, N_v=576 (24x24), "
                    "batch 1, 1-D RoPE at positions 35..610"),
    "llava_next_7b": Config(
        name="llava_next_7b", d=4096, n_layers=32, n_heads=32, n_kv_heads=32, head_dim=128,
        rank=128, n_vis=2880, batch=8, rope="1d", rope_theta=10000.0, rms_eps=1e-5,
        x0_sigma=0.5, seed=2, pos_start=35,
        description="LLaVA-NeXT-7B-shaped: d=4096, L=32, 32x128 MHA, r=128, N_v=2880 "
                    "(5 tiles x 576), batch 8, 1-D RoPE at positions 35..2914"),
    "qwen25vl_7b_image": Config(
        name="qwen25vl_7b_image", d=3584, n_layers=28, n_heads=28, n_kv_heads=4, head_dim=128,
        rank=128, n_vis=1296, batch=4, rope="mrope", rope_theta=1e6, mrope_section=(16, 24, 24),
        rms_eps=1e-6, x0_sigma=0.5, seed=3, pos_start=15, grid=(1, 36, 36),
        description="Qwen2.5-VL-7B-shaped image: d=3584, L=28, GQA 28/4x128, r=128, N_v=1296 "
                    "(36x36), batch 4, M-RoPE [16,24,24] over a 1x36x36 grid"),
    "qwen3vl_4b_image": Config(
        name="qwen3vl_4b_image", d=2560, n_layers=36, n_heads=32, n_kv_heads=8, head_dim=128,
        rank=128, n_vis=1024, batch=4, rope="mrope_interleaved", rope_theta=5e6,
        mrope_section=(24, 20, 20), rms_eps=1e-6, x0_sigma=0.5, seed=5, pos_start=15,
        grid=(1, 32, 32), k_norm=True,
        description="Qwen3-VL-4B-shaped image (the paper's default backbone): d=2560, L=36, "
                    "GQA 32/8x128, r=128, N_v=1024 (32x32), batch 4, interleaved M-RoPE "
                    "[24,20,20], per-head K RMSNorm"),
    "qwen25vl_7b_video": Config(
        name="qwen25vl_7b_video", d=3584, n_layers=28, n_heads=28, n_kv_heads=4, head_dim=128,
        rank=256, n_vis=16384, batch=1, rope="mrope", rope_theta=1e6, mrope_section=(16, 24, 24),
        rms_eps=1e-6, x0_sigma=0.5, seed=4, pos_start=15, grid=(32, 16, 32), ar1_rho=0.9,
        description="Qwen2.5-VL-7B-shaped video: d=3584, L=28, GQA 28/4x128, r=256, N_v=16384 "
                    "(32 frames x 16x32), batch 1, M-RoPE over a 32x16x32 grid, frame-correlated x0"),
}

CONFIG_ORDER = ["tiny", "llava15_7b", "llava_next_7b", "qwen25vl_7b_image", "qwen25vl_7b_video",
                "qwen3vl_4b_image"]


def config(name: str, **overrides) -> Config:
    return replace(CONFIGS[name], **overrides)


def positions(cfg: Config) -> np.ndarray:
    """int32 [B][P][N_v] visual positions (P = 1 for 1-D RoPE, 3 for M-RoPE (t, h, w)).

    1-D: token i of every batch element sits at pos_start + i.
    M-RoPE: token i is (frame f, row y, col x) of the visual grid in raster order and sits at
    (pos_start + f, pos_start + y, pos_start + x); for a single image f = 0.
    """
    B, N = cfg.batch, cfg.n_vis
    if cfg.rope == "1d":
        p = cfg.pos_start + np.arange(N, dtype=np.int64)
        return np.ascontiguousarray(np.broadcast_to(p, (B, 1, N)).astype(np.int32))
    frames, rows, cols = cfg.grid if cfg.grid else (1, 1, N)
    if frames * rows * cols != N:
        raise ValueError(f"grid {cfg.grid} does not hold {N} tokens")
    i = np.arange(N, dtype=np.int64)
    f, y, x = i // (rows * cols), (i // cols) % rows, i % cols
    p = np.stack([f, y, x]) + cfg.pos_start
    return np.ascontiguousarray(np.broadcast_to(p, (B, 3, N)).astype(np.int32))


@dataclass
class Inputs:
    """bf16 tensors as uint16 bit patterns, in the layouts the C-ABI takes."""
    cfg: Config
    x0: np.ndarray      # [B][N_v][d]
    D: np.ndarray       # [L][r][d]   down-projection, [out][in]
    U: np.ndarray       # [L][d][r]   up-projection, [out][in]
    gamma: np.ndarray   # [L][d]      RMSNorm weight
    Wk: np.ndarray      # [L][kv][d]
    Wv: np.ndarray      # [L][kv][d]
    bk: np.ndarray | None = None  # [L][kv]
    bv: np.ndarray | None = None
    pos: np.ndarray = field(default=None)  # int32 [B][P][N_v]
    kgamma: np.ndarray | None = None  # [L][head_dim] per-head K-norm gain (k_norm configs)


def make_x0(cfg: Config) -> np.ndarray:
    B, N, d = cfg.batch, cfg.n_vis, cfg.d
    if cfg.ar1_rho > 0.0:
        frames = cfg.grid[0]
        per_frame = (N // frames) * d
        out = np.empty((B, N * d), dtype=np.uint16)
        for b in range(B):
            out[b] = ar1_frames_bf16(cfg.seed, STREAM_X0 + 100 * b, frames, per_frame,
                                     cfg.ar1_rho, cfg.x0_sigma)
        return out.reshape(B, N, d)
    return normal_bf16(cfg.seed, STREAM_X0, (B, N, d), 0.0, cfg.x0_sigma)


def make_inputs(cfg: Config, with_x0: bool = True) -> Inputs:
    L, r, d, kv = cfg.n_layers, cfg.rank, cfg.d, cfg.kv
    s = cfg.seed
    D = normal_bf16(s, STREAM_D, (L, r, d), 0.0, cfg.w_sigma)
    if cfg.zero_up:
        U = np.zeros((L, d, r), dtype=np.uint16)
    else:
        U = normal_bf16(s, STREAM_U, (L, d, r), 0.0, cfg.w_sigma)
    if cfg.gamma_sigma > 0:
        gamma = normal_bf16(s, STREAM_GAMMA, (L, d), 1.0, cfg.gamma_sigma)
    else:
        gamma = np.full((L, d), 0x3F80, dtype=np.uint16)  # bf16 1.0
    Wk = normal_bf16(s, STREAM_WK, (L, kv, d), 0.0, cfg.w_sigma)
    Wv = normal_bf16(s, STREAM_WV, (L, kv, d), 0.0, cfg.w_sigma)
    bk = bv = None
    if cfg.bias_sigma > 0:
        bk = normal_bf16(s, STREAM_BK, (L, kv), 0.0, cfg.bias_sigma)
        bv = normal_bf16(s, STREAM_BV, (L, kv), 0.0, cfg.bias_sigma)
    kgamma = None
    if cfg.k_norm:
        kgamma = normal_bf16(s, STREAM_KGAMMA, (L, cfg.head_dim), 1.0, cfg.k_norm_sigma)
    x0 = make_x0(cfg) if with_x0 else None
    return Inputs(cfg=cfg, x0=x0, D=D, U=U, gamma=gamma, Wk=Wk, Wv=Wv, bk=bk, bv=bv,
                  pos=positions(cfg), kgamma=kgamma)
