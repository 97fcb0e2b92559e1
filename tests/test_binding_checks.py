"""The Python binding refuses bad build arguments before the C call (CPU only).

A wrong hidden size, an undersized cache or slots past its end would make the kernels read or
write out of bounds on the GPU, and int64 positions (torch.arange's default) would be read as
wrong positions, so ``validate_build`` raises ValueError for each of them. The checks run here
on CPU tensors by naming the CPU as the build device."""
import pytest

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def dv():
    import paper_2609_34972_gb300 as dv
    return dv


CPU = torch.device("cpu")
L, B, N, D, H, HD = 4, 2, 24, 512, 8, 64


def _args(dv, rope="1d", **kw):
    cfg = dv.make_config(D, L, H, HD, 16, rope=rope,
                         mrope_section=(8, 12, 12) if rope != "1d" else (0, 0, 0),
                         max_batch=B, max_n_vis=N)
    P = 1 if rope == "1d" else 3
    a = dict(x0=torch.zeros((B, N, D), dtype=torch.bfloat16),
             pos=torch.zeros((B, P, N), dtype=torch.int32),
             k_cache=torch.zeros((L, B, N, H, HD), dtype=torch.bfloat16),
             v_cache=torch.zeros((L, B, N, H, HD), dtype=torch.bfloat16),
             slot=None, slot0=0)
    a.update(kw)
    return cfg, a


def _validate(dv, cfg, a):
    return dv.validate_build(cfg, a["x0"], a["pos"], a["k_cache"], a["v_cache"], a["slot"],
                             a["slot0"], device=CPU)


def test_good_arguments_pass(dv):
    cfg, a = _args(dv)
    assert _validate(dv, cfg, a) == (B, N)
    cfg, a = _args(dv, rope="mrope")
    assert _validate(dv, cfg, a) == (B, N)
    # a larger cache with an offset, and explicit slots in range
    big = torch.zeros((L, B + 1, N + 9, H, HD), dtype=torch.bfloat16)
    cfg, a = _args(dv, k_cache=big, v_cache=big.clone(), slot0=9)
    assert _validate(dv, cfg, a) == (B, N)
    slot = torch.arange(N, dtype=torch.int32).repeat(B, 1) + 3
    cfg, a = _args(dv, k_cache=big, v_cache=big.clone(), slot=slot)
    assert _validate(dv, cfg, a) == (B, N)


@pytest.mark.parametrize("what,value", [
    ("x0", torch.zeros((B, N, D + 64), dtype=torch.bfloat16)),                  # wrong d
    ("x0", torch.zeros((B, N, D), dtype=torch.float16)),                        # wrong dtype
    ("x0", torch.zeros((B, D, N), dtype=torch.bfloat16).transpose(1, 2)),       # not contiguous
    ("x0", torch.zeros((B * N, D), dtype=torch.bfloat16)),                      # not 3-D
    ("pos", torch.zeros((B, 1, N), dtype=torch.int64)),                         # int64 positions
    ("pos", torch.zeros((B, N), dtype=torch.int32)),                            # missing axis dim
    ("pos", torch.zeros((B, 3, N), dtype=torch.int32)),                         # M-RoPE pos for 1-D
    ("k_cache", torch.zeros((L - 1, B, N, H, HD), dtype=torch.bfloat16)),       # too few layers
    ("k_cache", torch.zeros((L, B - 1, N, H, HD), dtype=torch.bfloat16)),       # too few batch rows
    ("k_cache", torch.zeros((L, B, N - 1, H, HD), dtype=torch.bfloat16)),       # too few slots
    ("k_cache", torch.zeros((L, B, N, H // 2, HD), dtype=torch.bfloat16)),      # wrong head count
    ("k_cache", torch.zeros((L, B, N, H, HD * 2), dtype=torch.bfloat16)),       # wrong head width
    ("v_cache", torch.zeros((L, B, N, H, HD), dtype=torch.float32)),            # wrong dtype
    ("slot0", 1),                                                               # slots past the end
    ("slot0", -1),
    ("slot", torch.zeros((B, N), dtype=torch.int64)),                           # int64 slots
    ("slot", torch.full((B, N), N, dtype=torch.int32)),                         # slot == S
    ("slot", torch.full((B, N), -2, dtype=torch.int32)),                        # negative slot
    ("slot", torch.zeros((B, N - 1), dtype=torch.int32)),                       # wrong shape
])
def test_bad_argument_raises(dv, what, value):
    cfg, a = _args(dv, **{what: value})
    with pytest.raises(ValueError):
        _validate(dv, cfg, a)


def test_mrope_needs_three_position_axes(dv):
    cfg, a = _args(dv, rope="mrope", pos=torch.zeros((B, 1, N), dtype=torch.int32))
    with pytest.raises(ValueError):
        _validate(dv, cfg, a)


def test_cuda_tensors_expected_by_default_device(dv):
    # Without a device argument the build device is the current CUDA device, so CPU tensors
    # are refused (on a machine without CUDA the lookup of that device itself fails).
    cfg, a = _args(dv)
    with pytest.raises((ValueError, RuntimeError, AssertionError)):
        dv.validate_build(cfg, a["x0"], a["pos"], a["k_cache"], a["v_cache"])


def test_host_pipeline_checks_host_buffers(dv):
    # The end-to-end wrapper takes exact dense host layouts: [L, B, N_v, H, D_h] K/V.
    cfg, a = _args(dv)
    pipe = object.__new__(dv.HostPipeline)     # no device pipeline: only the argument checks
    pipe.plan = type("P", (), {"cfg": cfg})()
    pipe.batch, pipe.n_vis = B, N
    pipe.handle = None
    kv = torch.zeros((L, B, N, H, HD), dtype=torch.bfloat16)
    pipe._check_host(a["x0"], a["pos"], kv, kv.clone())
    with pytest.raises(ValueError):
        pipe._check_host(a["x0"], a["pos"].long(), kv, kv.clone())
    with pytest.raises(ValueError):
        pipe._check_host(a["x0"], a["pos"], kv[:, :, :-1].clone(), kv.clone())
    with pytest.raises(ValueError):
        pipe._check_host(a["x0"][:, :-1].clone(), a["pos"], kv, kv.clone())
