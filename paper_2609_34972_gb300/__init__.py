"""Python binding of the GB300 visual-memory build (``include/dv.h``).

Argument marshalling only: every step of the build runs in the CUDA kernels of ``libdv.so``.
PyTorch supplies device memory and the CUDA stream. There is no CPU fallback: if the library
is missing, every call raises.

    plan = memory_plan(cfg, weights)               # once per weight set
    build_visual_memory(plan, x0, pos, k_cache, v_cache)   # the hot path
    free(plan)

Tensor layouts (bf16 unless stated, all on the current CUDA device):
    x0      [B, N_v, d]          visual embeddings E (Sec. 2 Eq. 1)
    pos     int32 [B, P, N_v]    P = 1 (1-D RoPE) or 3 (M-RoPE t, h, w)
    weights D [L, r, d], U [L, d, r], gamma [L, d], Wk, Wv [L, kv, d], bk, bv [L, kv] (optional),
            kgamma [L, D_h] (per-head K-norm gain, with k_norm)
    k/v cache [L, B_c, S, H_kv, D_h] or any strided view with D_h contiguous
"""
from __future__ import annotations

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libdv.so")

DV_OK = 0
DV_ERR_INVALID_ARG = 1
DV_ERR_UNSUPPORTED_SHAPE = 2
DV_ERR_ALIGNMENT = 3
DV_ERR_OOM = 4
DV_ERR_CUDA = 5
DV_ERR_DEVICE_TIMEOUT = 6
DV_ERR_UNSUPPORTED_DEVICE = 7
DV_ACT_SILU = 0
DV_ROPE_1D = 0
DV_ROPE_MROPE = 1
DV_ROPE_MROPE_INTERLEAVED = 2
_ROPE = {"1d": DV_ROPE_1D, "mrope": DV_ROPE_MROPE, "mrope_interleaved": DV_ROPE_MROPE_INTERLEAVED}
DV_LAYER_ADAPTER = 0
DV_LAYER_IDENTITY = 1
DV_LAYER_DROP = 2
DV_ADAPTER_EMBEDDING = 0
DV_ADAPTER_RECURRENT = 1
DV_RECURRENT_AUTO = 0
DV_RECURRENT_CHAIN = 1
DV_RECURRENT_REARRANGED = 2
_RECURRENT_PATH = {"auto": DV_RECURRENT_AUTO, "chain": DV_RECURRENT_CHAIN,
                   "rearranged": DV_RECURRENT_REARRANGED}

EXPORTED = ["dv_memory_plan", "dv_build_visual_memory", "dv_plan_status", "dv_free",
            "dv_error_string", "dv_timing_enable", "dv_timing_read", "dv_kernels_per_build",
            "dv_debug_wait_timeout", "dv_debug_copy_workspace", "dv_build_visual_memory_noalloc",
            "dv_debug_copy_memory", "dv_kv_engine", "dv_text_attention", "dv_text_attention_status",
            "dv_host_pipeline_create", "dv_build_visual_memory_host", "dv_host_pipeline_wait",
            "dv_host_pipeline_join", "dv_host_pipeline_free"]
N_STAGES = 4
STAGE_NAMES = ["down_proj_silu", "row_sumsq", "rms_stats", "kv_proj_rope_store"]
# Stage names of a recurrent-adapter build (stage 0 is empty there).
STAGE_NAMES_RECURRENT = ["none", "adapter_chain", "rms_stats", "kv_proj_rope_store"]


class DvConfig(ctypes.Structure):
    _fields_ = [("d", ctypes.c_int), ("n_layers", ctypes.c_int), ("n_kv_heads", ctypes.c_int),
                ("head_dim", ctypes.c_int), ("rank", ctypes.c_int), ("act", ctypes.c_int),
                ("rope", ctypes.c_int), ("rope_theta", ctypes.c_float),
                ("mrope_section", ctypes.c_int * 3), ("rms_eps", ctypes.c_float),
                ("max_batch", ctypes.c_int), ("max_n_vis", ctypes.c_int),
                ("has_kv_bias", ctypes.c_int), ("adapter", ctypes.c_int),
                ("k_norm", ctypes.c_int), ("k_norm_eps", ctypes.c_float),
                ("split_chain", ctypes.c_int), ("recurrent_path", ctypes.c_int)]


class DvWeights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("D", "U", "gamma", "Wk", "Wv", "bk", "bv",
                                               "layer_mode", "k_norm_gamma")]


class DvKVCache(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("s_layer", ctypes.c_longlong),
                ("s_batch", ctypes.c_longlong), ("s_seq", ctypes.c_longlong),
                ("s_head", ctypes.c_longlong)]


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded ``libdv.so``; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"CUDA library {LIB_PATH} is missing: run "
                               "`python -c 'import __graft_entry__ as g; g.build()'` first")
        L = ctypes.CDLL(LIB_PATH)
        vp, i32 = ctypes.c_void_p, ctypes.c_int
        L.dv_memory_plan.argtypes = [ctypes.POINTER(DvConfig), ctypes.POINTER(DvWeights), vp,
                                     ctypes.POINTER(vp)]
        L.dv_build_visual_memory.argtypes = [vp, vp, i32, i32, vp, vp, i32,
                                             ctypes.POINTER(DvKVCache), vp]
        L.dv_plan_status.argtypes = [vp]
        L.dv_free.argtypes = [vp]
        L.dv_free.restype = None
        L.dv_error_string.argtypes = [i32]
        L.dv_error_string.restype = ctypes.c_char_p
        L.dv_timing_enable.argtypes = [vp, i32]
        L.dv_timing_read.argtypes = [vp, ctypes.POINTER(ctypes.c_double), i32,
                                     ctypes.POINTER(i32)]
        L.dv_kernels_per_build.argtypes = [vp]
        L.dv_debug_wait_timeout.argtypes = [vp, i32, vp]
        L.dv_debug_copy_workspace.argtypes = [vp, i32, vp, vp, vp, ctypes.POINTER(i32), vp]
        L.dv_build_visual_memory_noalloc.argtypes = [vp, vp, i32, i32, vp, vp, i32,
                                                     ctypes.POINTER(DvKVCache), vp]
        L.dv_debug_copy_memory.argtypes = [vp, i32, vp, vp]
        L.dv_kv_engine.argtypes = [vp, ctypes.c_longlong]
        L.dv_text_attention.argtypes = [vp, i32, i32, i32, i32, i32, ctypes.POINTER(DvKVCache),
                                        i32, i32, vp, vp, ctypes.c_float, vp, vp]
        L.dv_text_attention_status.argtypes = []
        L.dv_host_pipeline_create.argtypes = [vp, i32, i32, i32, ctypes.POINTER(vp)]
        L.dv_build_visual_memory_host.argtypes = [vp, vp, vp, vp, vp, vp,
                                                  ctypes.POINTER(ctypes.c_longlong)]
        L.dv_host_pipeline_wait.argtypes = [vp, ctypes.c_longlong]
        L.dv_host_pipeline_join.argtypes = [vp, vp]
        L.dv_host_pipeline_free.argtypes = [vp]
        L.dv_host_pipeline_free.restype = None
        for name in ("dv_memory_plan", "dv_build_visual_memory", "dv_plan_status",
                     "dv_timing_enable", "dv_timing_read", "dv_kernels_per_build",
                     "dv_debug_wait_timeout", "dv_debug_copy_workspace",
                     "dv_build_visual_memory_noalloc", "dv_debug_copy_memory", "dv_kv_engine",
                     "dv_text_attention", "dv_text_attention_status", "dv_host_pipeline_create",
                     "dv_build_visual_memory_host", "dv_host_pipeline_wait",
                     "dv_host_pipeline_join"):
            getattr(L, name).restype = i32
        _lib = L
    return _lib


class DvError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: {error_string(code)} (status {code})")


def error_string(code: int) -> str:
    return lib().dv_error_string(int(code)).decode()


def _check(code: int, where: str):
    if code != DV_OK:
        raise DvError(code, where)


def _stream_handle(stream):
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(int(stream.cuda_stream))


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def make_config(d, n_layers, n_kv_heads, head_dim, rank, rope="1d", rope_theta=10000.0,
                mrope_section=(0, 0, 0), rms_eps=1e-6, max_batch=1, max_n_vis=1,
                has_kv_bias=False, adapter="embedding", k_norm=False,
                k_norm_eps=1e-6, split_chain=False, recurrent_path="auto") -> DvConfig:
    """``adapter``: "embedding" (M_l = A_l(E), Sec. 3.1 Eq. 5) or "recurrent"
    (M_l = A_l(M_{l-1}), Sec. 3.1 Eq. 6). ``rope``: "1d", "mrope" (contiguous sections) or
    "mrope_interleaved". ``k_norm``: per-head RMSNorm of K before RoPE (weights["kgamma"]).
    ``split_chain`` (recurrent only): the chain's GEMMs read hi + lo bf16 operands.
    ``recurrent_path`` (recurrent only): "auto", "chain" (the paper's order) or "rearranged"."""
    if adapter not in ("embedding", "recurrent"):
        raise ValueError(f"unknown adapter {adapter!r}")
    if rope not in _ROPE:
        raise ValueError(f"unknown rope {rope!r}")
    if recurrent_path not in _RECURRENT_PATH:
        raise ValueError(f"unknown recurrent_path {recurrent_path!r}")
    return DvConfig(int(d), int(n_layers), int(n_kv_heads), int(head_dim), int(rank),
                    DV_ACT_SILU, _ROPE[rope],
                    float(rope_theta), (ctypes.c_int * 3)(*mrope_section), float(rms_eps),
                    int(max_batch), int(max_n_vis), int(bool(has_kv_bias)),
                    DV_ADAPTER_RECURRENT if adapter == "recurrent" else DV_ADAPTER_EMBEDDING,
                    int(bool(k_norm)), float(k_norm_eps), int(bool(split_chain)),
                    _RECURRENT_PATH[recurrent_path])


class Plan:
    """Owns a ``dv_plan*``: repacked weights, workspace and TMA descriptors on one device."""

    def __init__(self, handle: ctypes.c_void_p, cfg: DvConfig, layers=None):
        self.handle = handle
        self.cfg = cfg
        # cache layers the plan builds (all but the DV_LAYER_DROP ones), in order
        self.layers = list(range(cfg.n_layers)) if layers is None else list(layers)

    @property
    def alive(self) -> bool:
        return bool(self.handle and self.handle.value)

    def __del__(self):
        try:
            free(self)
        except Exception:
            pass


def memory_plan(cfg: DvConfig, weights: dict, stream=None, layer_modes=None) -> Plan:
    """Plan a build for ``cfg`` from device weights (dict of torch tensors, see module doc).
    ``layer_modes``: optional sequence of DV_LAYER_* per layer (App. J adapter skipping)."""
    modes = None
    if layer_modes is not None:
        if len(layer_modes) != cfg.n_layers:
            raise ValueError("layer_modes needs one entry per layer")
        modes = (ctypes.c_ubyte * cfg.n_layers)(*[int(m) for m in layer_modes])
    w = DvWeights(*[_ptr(weights.get(n)) for n in ("D", "U", "gamma", "Wk", "Wv", "bk", "bv")],
                  ctypes.cast(modes, ctypes.c_void_p) if modes is not None else None,
                  _ptr(weights.get("kgamma")))
    h = ctypes.c_void_p()
    _check(lib().dv_memory_plan(ctypes.byref(cfg), ctypes.byref(w), _stream_handle(stream),
                                ctypes.byref(h)), "dv_memory_plan")
    kept = None if layer_modes is None else [l for l, m in enumerate(layer_modes)
                                             if int(m) != DV_LAYER_DROP]
    return Plan(h, cfg, kept)


def kv_cache_view(k, v) -> DvKVCache:
    """Describe two [L, B, S, H, D_h] (strided, D_h contiguous) bf16 tensors for the C ABI."""
    if k.dim() != 5 or v.dim() != 5 or k.stride() != v.stride() or k.stride(4) != 1:
        raise ValueError("k and v must be 5-D [L, B, S, H, D_h] views with equal strides, D_h contiguous")
    s = k.stride()
    return DvKVCache(k.data_ptr(), v.data_ptr(), s[0], s[1], s[2], s[3])


def _n_pos(cfg: DvConfig) -> int:
    return 1 if cfg.rope == DV_ROPE_1D else 3


def _check_tensor(name, t, dtype, device=None, shape=None, contiguous=True):
    import torch
    if not isinstance(t, torch.Tensor):
        raise ValueError(f"{name} must be a torch tensor")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if device is not None and t.device != device:
        raise ValueError(f"{name} must be on {device}, got {t.device}")
    if contiguous and not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")


def validate_build(cfg: DvConfig, x0, pos, k_cache, v_cache, slot=None, slot0: int = 0,
                   device=None):
    """Checks of a build's tensors against the plan's configuration, made before the C call.
    A wrong d or an undersized cache would make the kernels read or write out of bounds, and an
    int64 position tensor would be read as wrong positions, so they raise ValueError here; the
    C ABI itself checks pointers, alignment, strides and the plan's token limit. ``device``
    defaults to the current CUDA device (the one the C ABI builds on). Returns (B, N_v)."""
    import torch
    if device is None:
        device = torch.device("cuda", torch.cuda.current_device())
    if not isinstance(x0, torch.Tensor) or x0.dim() != 3:
        raise ValueError("x0 must be a 3-D [B, N_v, d] tensor")
    B, N = int(x0.shape[0]), int(x0.shape[1])
    _check_tensor("x0", x0, torch.bfloat16, device, (B, N, cfg.d))
    _check_tensor("pos", pos, torch.int32, device, (B, _n_pos(cfg), N))
    for name, c in (("k_cache", k_cache), ("v_cache", v_cache)):
        _check_tensor(name, c, torch.bfloat16, device, contiguous=False)
        if c.dim() != 5:
            raise ValueError(f"{name} must be 5-D [L, B_c, S, H_kv, D_h]")
        if (c.shape[0] < cfg.n_layers or c.shape[1] < B or c.shape[3] != cfg.n_kv_heads
                or c.shape[4] != cfg.head_dim):
            raise ValueError(f"{name} of shape {tuple(c.shape)} cannot hold {cfg.n_layers} layers x "
                             f"{B} batch rows x {cfg.n_kv_heads} heads x {cfg.head_dim}")
    if k_cache.shape != v_cache.shape:
        raise ValueError("k_cache and v_cache must have the same shape")
    S = int(k_cache.shape[2])
    if int(slot0) < 0:
        raise ValueError("slot0 must be >= 0")
    if slot is None:
        if B * N > 0 and int(slot0) + N > S:
            raise ValueError(f"slots {slot0}..{int(slot0) + N - 1} exceed the cache's {S} slots")
    else:
        _check_tensor("slot", slot, torch.int32, device, (B, N))
        if B * N > 0:
            lo, hi = int(slot.min()), int(slot.max())   # synchronises: slots are checked, not trusted
            if lo < 0 or hi >= S:
                raise ValueError(f"slot values {lo}..{hi} outside the cache's {S} slots")
    return B, N


def build_visual_memory(plan: Plan, x0, pos, k_cache, v_cache, slot=None, slot0: int = 0,
                        stream=None) -> None:
    """Enqueue one build on ``stream`` (default: torch's current stream). Asynchronous, except
    that explicit ``slot`` values are range-checked on the host first (a synchronisation)."""
    B, N = validate_build(plan.cfg, x0, pos, k_cache, v_cache, slot, slot0)
    kvc = kv_cache_view(k_cache, v_cache)
    _check(lib().dv_build_visual_memory(plan.handle, _ptr(x0), B, N, _ptr(pos), _ptr(slot),
                                        int(slot0), ctypes.byref(kvc), _stream_handle(stream)),
           "dv_build_visual_memory")


def build_visual_memory_noalloc(plan: Plan, x0, pos, k_cache, v_cache, slot=None,
                                slot0: int = 0, stream=None) -> None:
    """Same build as ``build_visual_memory`` for callers that must not allocate device memory:
    the intermediates live in the library's static 32 MiB device array, not in the plan's
    workspace. All such calls on a device share that array, so calls must not overlap on the
    GPU; builds whose intermediates exceed 32 MiB raise DvError (unsupported shape)."""
    B, N = validate_build(plan.cfg, x0, pos, k_cache, v_cache, slot, slot0)
    kvc = kv_cache_view(k_cache, v_cache)
    _check(lib().dv_build_visual_memory_noalloc(plan.handle, _ptr(x0), B, N, _ptr(pos), _ptr(slot),
                                                int(slot0), ctypes.byref(kvc),
                                                _stream_handle(stream)),
           "dv_build_visual_memory_noalloc")


def plan_status(plan: Plan) -> int:
    """Synchronise and read (and clear) the plan's device status word."""
    return int(lib().dv_plan_status(plan.handle))


def free(plan: Plan) -> None:
    if plan is not None and plan.alive:
        lib().dv_free(plan.handle)
        plan.handle = ctypes.c_void_p()


def kernels_per_build(plan: Plan) -> int:
    return int(lib().dv_kernels_per_build(plan.handle))


def timing_enable(plan: Plan, on: bool = True) -> None:
    _check(lib().dv_timing_enable(plan.handle, int(bool(on))), "dv_timing_enable")


def timing_read(plan: Plan):
    """(per-stage summed milliseconds, number of builds) since timing_enable."""
    ms = (ctypes.c_double * N_STAGES)()
    n = ctypes.c_int()
    _check(lib().dv_timing_read(plan.handle, ms, N_STAGES, ctypes.byref(n)), "dv_timing_read")
    return list(ms), n.value


def debug_wait_timeout(plan: Plan, timeout_us: int, stream=None) -> None:
    _check(lib().dv_debug_wait_timeout(plan.handle, int(timeout_us), _stream_handle(stream)),
           "dv_debug_wait_timeout")


def debug_workspace(plan: Plan, tokens: int, stream=None):
    """(H [tokens, L*r_pad] bf16, rstd [L, tokens] fp32, xx [tokens] fp32) of the last build;
    L counts the planned layers (``plan.layers``), which excludes dropped ones."""
    import torch
    r_pad = ctypes.c_int()
    _check(lib().dv_debug_copy_workspace(plan.handle, 0, None, None, None, ctypes.byref(r_pad),
                                         None), "dv_debug_copy_workspace")
    L = len(plan.layers)
    H = torch.empty((tokens, L * r_pad.value), dtype=torch.bfloat16, device="cuda")
    rstd = torch.empty((L, tokens), dtype=torch.float32, device="cuda")
    xx = torch.empty((tokens,), dtype=torch.float32, device="cuda")
    _check(lib().dv_debug_copy_workspace(plan.handle, int(tokens), _ptr(H), _ptr(rstd), _ptr(xx),
                                         None, _stream_handle(stream)), "dv_debug_copy_workspace")
    return H, rstd, xx, r_pad.value


def debug_memory(plan: Plan, tokens: int, stream=None):
    """bf16 M_l of every planned layer of the last (recurrent) build: [L_planned, tokens, d]."""
    import torch
    mem = torch.empty((len(plan.layers), tokens, plan.cfg.d), dtype=torch.bfloat16, device="cuda")
    _check(lib().dv_debug_copy_memory(plan.handle, int(tokens), _ptr(mem), _stream_handle(stream)),
           "dv_debug_copy_memory")
    return mem


def text_attention(q, k_cache, v_cache, layer: int, n_keys, q_slot, scale: float, out=None,
                   stream=None):
    """Causal attention of text queries over one layer of the cache (Sec. 3.2).

    q: bf16 [B, Hq, Nt, D_h] (rotated); k_cache / v_cache: the [L, B_c, S, H_kv, D_h] cache views
    the build writes; n_keys int32 [B]; q_slot int32 [B, Nt]. Returns bf16 [B, Hq, Nt, D_h]."""
    import torch
    B, Hq, Nt, D = (int(x) for x in q.shape)
    kvc = kv_cache_view(k_cache, v_cache)
    if out is None:
        out = torch.empty((B, Hq, Nt, D), dtype=torch.bfloat16, device=q.device)
    _check(lib().dv_text_attention(_ptr(q), B, Hq, int(k_cache.shape[3]), Nt, D, ctypes.byref(kvc),
                                   int(layer), int(k_cache.shape[2]), _ptr(n_keys), _ptr(q_slot),
                                   float(scale), _ptr(out), _stream_handle(stream)),
           "dv_text_attention")
    return out


def text_attention_status() -> int:
    return int(lib().dv_text_attention_status())


KV_KERNELS = {1: "dv_kv_pair_kernel (weights as M, 2-SM UMMA)",
              2: "dv_pair_tm_kernel<EPI_KV> (256-token blocks as M, 2-SM UMMA)"}


def kv_kernel(plan: Plan, tokens: int) -> str:
    """Name of the kernel that computes K/V in a build of ``tokens`` tokens."""
    return KV_KERNELS.get(int(lib().dv_kv_engine(plan.handle, int(tokens))), "none")


def stage_names(plan: Plan):
    """Names of the four timed stages of a build with this plan."""
    return STAGE_NAMES_RECURRENT if plan.cfg.adapter == DV_ADAPTER_RECURRENT else STAGE_NAMES


class HostPipeline:
    """End-to-end builds from host memory through the C ABI (``dv_host_pipeline_*``,
    ``dv_build_visual_memory_host``): every ``submit`` copies one batch's E and positions to the
    device, builds, and copies the built K/V back into the caller's host buffers, with the
    copy-out of one build overlapping the next build (``depth`` device staging sets).

    Host tensors (CPU, contiguous; page-locked for the copies to overlap):
        x0 bf16 [B, N_v, d], pos int32 [B, P, N_v], k / v bf16 [L, B, N_v, H_kv, D_h]
    ``submit`` returns a ticket; ``wait(ticket)`` blocks until that build's K/V are in its
    host buffers, ``join(stream)`` orders later work on ``stream`` after every submitted build.
    """

    def __init__(self, plan: Plan, batch: int, n_vis: int, depth: int = 2):
        self.plan = plan
        self.batch, self.n_vis = int(batch), int(n_vis)
        h = ctypes.c_void_p()
        _check(lib().dv_host_pipeline_create(plan.handle, self.batch, self.n_vis, int(depth),
                                             ctypes.byref(h)), "dv_host_pipeline_create")
        self.handle = h

    def _check_host(self, x0, pos, k, v):
        import torch
        cfg, B, N = self.plan.cfg, self.batch, self.n_vis
        cpu = torch.device("cpu")
        _check_tensor("x0", x0, torch.bfloat16, cpu, (B, N, cfg.d))
        _check_tensor("pos", pos, torch.int32, cpu, (B, _n_pos(cfg), N))
        shape = (cfg.n_layers, B, N, cfg.n_kv_heads, cfg.head_dim)
        _check_tensor("k", k, torch.bfloat16, cpu, shape)
        _check_tensor("v", v, torch.bfloat16, cpu, shape)

    def submit(self, x0, pos, k, v, stream=None) -> int:
        if not self.plan.alive or not (self.handle and self.handle.value):
            raise ValueError("the pipeline or its plan has been freed")
        self._check_host(x0, pos, k, v)
        t = ctypes.c_longlong()
        _check(lib().dv_build_visual_memory_host(self.handle, _ptr(x0), _ptr(pos), _ptr(k), _ptr(v),
                                                 _stream_handle(stream), ctypes.byref(t)),
               "dv_build_visual_memory_host")
        return t.value

    def wait(self, ticket: int) -> None:
        _check(lib().dv_host_pipeline_wait(self.handle, int(ticket)), "dv_host_pipeline_wait")

    def join(self, stream=None) -> None:
        _check(lib().dv_host_pipeline_join(self.handle, _stream_handle(stream)), "dv_host_pipeline_join")

    def close(self) -> None:
        if self.handle and self.handle.value:
            lib().dv_host_pipeline_free(self.handle)
            self.handle = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
