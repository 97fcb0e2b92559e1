"""The seeded input generator: determinism, distribution, rounding, workload recipes."""
import numpy as np
import pytest

import synth


def test_deterministic_and_counter_based():
    a = synth.normal_bf16(3, 5, (1000,), 0.0, 1.0)
    b = synth.normal_bf16(3, 5, (1000,), 0.0, 1.0)
    assert np.array_equal(a, b)
    # counter-based: a window drawn at an offset equals the same slice of a longer draw
    c = synth.normal_bf16(3, 5, (400,), 0.0, 1.0, offset=600)
    assert np.array_equal(a[600:], c)
    assert not np.array_equal(a, synth.normal_bf16(3, 6, (1000,), 0.0, 1.0))
    assert not np.array_equal(a, synth.normal_bf16(4, 5, (1000,), 0.0, 1.0))


def test_normal_moments():
    x = synth.normal_f64(11, 0, (400_000,), 0.0, 1.0)
    assert abs(x.mean()) < 0.01 and abs(x.std() - 1.0) < 0.01
    assert abs(np.mean(x ** 4) - 3.0) < 0.05                      # Gaussian kurtosis
    w = synth.bf16_to_f32(synth.normal_bf16(11, 1, (400_000,), 0.0, 0.02)).astype(float)
    assert abs(w.std() - 0.02) < 0.0005


def test_bf16_rounding_matches_torch():
    torch = pytest.importorskip("torch")
    v = synth.normal_f64(12, 0, (100_000,), 0.0, 3.0).astype(np.float32)
    ours = synth.f64_to_bf16(v)
    ref = torch.from_numpy(v).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)
    c = synth.normal_bf16(12, 0, (100_000,), 0.0, 3.0)
    assert np.array_equal(c, synth.f64_to_bf16(synth.normal_f64(12, 0, (100_000,), 0.0, 3.0)))


def test_ar1_frames_correlation():
    n_frames, per = 32, 20_000
    x = synth.bf16_to_f32(synth.ar1_frames_bf16(4, 0, n_frames, per, 0.9, 1.0)).astype(float)
    x = x.reshape(n_frames, per)
    rho = np.mean([np.corrcoef(x[f], x[f + 1])[0, 1] for f in range(n_frames - 1)])
    assert abs(rho - 0.9) < 0.01
    assert abs(x.std() - 1.0) < 0.02


def test_positions():
    p = synth.positions(synth.CONFIGS["tiny"])
    assert p.shape == (1, 1, 64) and p[0, 0, 0] == 5 and p[0, 0, -1] == 68
    p = synth.positions(synth.CONFIGS["llava15_7b"])
    assert p[0, 0, 0] == 35 and p[0, 0, -1] == 610
    p = synth.positions(synth.CONFIGS["llava_next_7b"])
    assert p.shape == (8, 1, 2880) and p[7, 0, -1] == 2914
    c4 = synth.CONFIGS["qwen25vl_7b_image"]
    p = synth.positions(c4)
    assert p.shape == (4, 3, 1296)
    assert np.all(p[:, 0] == 15) and p[0, 1, 36] == 16 and p[0, 2, 37] == 16 and p[0, 2, 35] == 50
    c5 = synth.CONFIGS["qwen25vl_7b_video"]
    p = synth.positions(c5)
    assert p.shape == (1, 3, 16384) and p[0, 0, -1] == 15 + 31 and p[0, 1, 512] == 15
    assert p[0, 2, 31] == 15 + 31 and p[0, 1, 32] == 16


def test_config_workload_figures():
    c2 = synth.CONFIGS["llava15_7b"]
    assert c2.tokens == 576 and c2.kv == 4096
    assert c2.flops() == pytest.approx(1.256e12, rel=2e-3)
    c5 = synth.CONFIGS["qwen25vl_7b_video"]
    assert c5.kv == 512 and c5.flops() == pytest.approx(5.051e12, rel=2e-3)
