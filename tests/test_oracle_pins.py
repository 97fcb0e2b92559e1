"""Pins of the fp64 oracle to what the paper and the mathematics fix (CPU only).

Each test targets a mistake the oracle could plausibly make (a dropped term, a wrong sign,
a transposed operand, a wrong index), using closed forms, invariants, hand-derived tiny
examples and special cases that reduce to a library routine. None of them re-types the
oracle's formula and compares the oracle with itself.
"""
import dataclasses
import math

import numpy as np
import pytest

import oracle
import synth
from synth import Config, Inputs, f64_to_bf16 as bf


def _tiny_cfg(**kw):
    base = dict(name="hand", d=4, n_layers=1, n_heads=1, n_kv_heads=1, head_dim=4, rank=2,
                n_vis=1, batch=1, rope="1d", rope_theta=10000.0, rms_eps=0.0)
    base.update(kw)
    return Config(**base)


def _inputs(cfg, x0, D, U, gamma, Wk, Wv, pos, bk=None, bv=None):
    return Inputs(cfg=cfg, x0=bf(np.asarray(x0, float)), D=bf(np.asarray(D, float)),
                  U=bf(np.asarray(U, float)), gamma=bf(np.asarray(gamma, float)),
                  Wk=bf(np.asarray(Wk, float)), Wv=bf(np.asarray(Wv, float)),
                  bk=None if bk is None else bf(np.asarray(bk, float)),
                  bv=None if bv is None else bf(np.asarray(bv, float)),
                  pos=np.asarray(pos, dtype=np.int32))


# ---------------------------------------------------------------- SiLU (Sec. 3.1 Eq. 4)

def test_silu_closed_forms():
    # sigmoid(ln 3) = 3/4 and sigmoid(-ln 3) = 1/4, so SiLU(+-ln 3) = (3/4) ln 3, -(1/4) ln 3.
    ln3 = math.log(3.0)
    assert oracle.silu(ln3) == pytest.approx(0.75 * ln3, rel=1e-15)
    assert oracle.silu(-ln3) == pytest.approx(-0.25 * ln3, rel=1e-15)
    assert oracle.silu(0.0) == 0.0
    # u*s(u) - (-u)*s(-u) = u (s(u) + s(-u)) = u for every u.
    for u in (0.1, 1.7, 5.0, 20.0):
        assert oracle.silu(u) - oracle.silu(-u) == pytest.approx(u, rel=1e-14)
    assert oracle.silu(40.0) == pytest.approx(40.0, rel=1e-15)
    assert abs(oracle.silu(-40.0)) < 1e-15


# ---------------------------------------------------------------- adapter (Sec. 3.1 Eqs. 4-5)

def test_adapter_hand_example():
    # x = [1, 2, 0, -1]; D_l (d x r) picks x_0 and x_1, so z = [1, 2].
    # U_l (r x d) sends h_0 to channel 1 and h_1 / 2 to channel 2.
    x = np.array([1.0, 2.0, 0.0, -1.0])
    D_stored = bf(np.array([[1, 0, 0, 0], [0, 1, 0, 0]], float))          # [r][d]
    U_stored = bf(np.array([[0, 0], [1, 0], [0, 0.5], [0, 0]], float))     # [d][r]
    z, h, m = oracle.adapter_row(x, D_stored, U_stored)
    s1, s2 = 1.0 / (1.0 + math.exp(-1.0)), 1.0 / (1.0 + math.exp(-2.0))
    np.testing.assert_allclose(z, [1.0, 2.0], rtol=0, atol=0)
    np.testing.assert_allclose(h, [s1, 2 * s2], rtol=1e-15)
    np.testing.assert_allclose(m, [1.0, 2.0 + s1, 0.5 * 2 * s2, -1.0], rtol=1e-15)


def _random_inputs(**kw):
    cfg = synth.config("tiny", **kw)
    return cfg, synth.make_inputs(cfg)


def test_zero_up_projection_is_identity():
    # U_l initialised to zero makes A_l the identity (Sec. 3.1): M_l = E exactly.
    cfg, inp = _random_inputs(zero_up=True, n_vis=16)
    out = oracle.build_tokens(inp, want=("m",))
    x = synth.bf16_to_f32(inp.x0).astype(np.float64).reshape(cfg.tokens, 1, cfg.d)
    assert np.array_equal(out["m"], np.broadcast_to(x, out["m"].shape))


def test_zero_down_projection_is_identity():
    # D_l = 0 gives z = 0, SiLU(0) = 0, so the residual update vanishes and M_l = E.
    cfg, inp = _random_inputs(n_vis=16)
    inp.D[:] = 0
    out = oracle.build_tokens(inp, want=("m", "h"))
    x = synth.bf16_to_f32(inp.x0).astype(np.float64).reshape(cfg.tokens, 1, cfg.d)
    assert np.all(out["h"] == 0.0)
    assert np.array_equal(out["m"], np.broadcast_to(x, out["m"].shape))


def test_update_rank_at_most_r():
    # rank(Delta_l(X)) <= r (Sec. 3.1): the update of N_v > r tokens spans at most r directions.
    cfg, inp = _random_inputs(n_vis=64, rank=16, x0_sigma=1.0, w_sigma=0.2)
    out = oracle.build_tokens(inp, want=("m",))
    x = synth.bf16_to_f32(inp.x0).astype(np.float64).reshape(cfg.tokens, cfg.d)
    for l in range(cfg.n_layers):
        delta = out["m"][:, l, :] - x                      # [N_v, d]
        s = np.linalg.svd(delta, compute_uv=False)
        assert s[cfg.rank] < 1e-9 * s[0]                   # nothing beyond r directions
        assert s[cfg.rank - 1] > 1e-6 * s[0]               # and generically exactly r


def test_stacked_down_projection_equals_per_layer():
    # Every layer's down-projection reads only E (Sec. 3.1 Eq. 5), so the L products x D_l are
    # the column blocks of one product x [D_1 ... D_L]; checked against a library matmul.
    cfg, inp = _random_inputs(n_vis=8)
    out = oracle.build_tokens(inp, want=("h",))
    x = synth.bf16_to_f32(inp.x0).astype(np.float64).reshape(cfg.tokens, cfg.d)
    Dcat = synth.bf16_to_f32(inp.D).astype(np.float64).reshape(cfg.n_layers * cfg.rank, cfg.d)
    z = x @ Dcat.T                                          # [T, L*r], one stacked product
    h = z / (1.0 + np.exp(-z))
    np.testing.assert_allclose(out["h"].reshape(cfg.tokens, -1), h, rtol=1e-12, atol=1e-14)


def test_layers_independent_given_embeddings():
    # The memories are conditionally independent across layers given E (Sec. 3.1): changing
    # layer 2's weights leaves every other layer's K and V bit-identical.
    cfg, inp = _random_inputs(n_vis=8)
    a = oracle.build_tokens(inp, want=("k", "v"))
    inp.U[2] = synth.normal_bf16(99, 0, inp.U[2].shape, 0.0, 0.05)
    inp.Wk[2] = synth.normal_bf16(99, 1, inp.Wk[2].shape, 0.0, 0.05)
    b = oracle.build_tokens(inp, want=("k", "v"))
    for l in (0, 1, 3):
        assert np.array_equal(a["k"][:, l], b["k"][:, l]) and np.array_equal(a["v"][:, l], b["v"][:, l])
    assert not np.array_equal(a["k"][:, 2], b["k"][:, 2])


# ---------------------------------------------------------------- RMSNorm (LN_l, Eq. 7; App. K)

def test_rmsnorm_constant_vector_with_eps():
    # m = c * 1: mean(m^2) = c^2, so n = gamma * c / sqrt(c^2 + eps).
    d, c, eps = 8, -3.0, 0.5
    gamma = np.array([2.0, 1.0, 0.5, -1.0, 3.0, 1.0, 1.0, 0.25])
    n = oracle.rmsnorm_row(np.full(d, c), gamma, eps)
    np.testing.assert_allclose(n, gamma * c / math.sqrt(c * c + eps), rtol=1e-15)


def test_rmsnorm_hand_example():
    # m = [1, 2, 2, 4]: mean of squares 25/4, root 5/2, so n = m / 2.5 exactly.
    n = oracle.rmsnorm_row(np.array([1.0, 2.0, 2.0, 4.0]), np.ones(4), 0.0)
    np.testing.assert_allclose(n, [0.4, 0.8, 0.8, 1.6], rtol=1e-15)


def test_rmsnorm_scale_invariance_and_library():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(0)
    m, g = rng.normal(size=256), rng.normal(size=256)
    n1 = oracle.rmsnorm_row(m, g, 0.0)
    n2 = oracle.rmsnorm_row(37.5 * m, g, 0.0)
    np.testing.assert_allclose(n1, n2, rtol=1e-13)
    ref = torch.nn.functional.rms_norm(torch.tensor(m)[None], (256,), torch.tensor(g), eps=1e-6)[0]
    np.testing.assert_allclose(oracle.rmsnorm_row(m, g, 1e-6), ref.numpy(), rtol=1e-13)


# ---------------------------------------------------------------- projection (Eq. 7)

def test_projection_matches_library_matmul():
    rng = np.random.default_rng(1)
    W = bf(rng.normal(size=(24, 40)))                       # kv != d catches a transposition
    b = bf(rng.normal(size=24))
    n = rng.normal(size=40)
    out = oracle.project_row(W, b, n)
    Wf, bfv = synth.bf16_to_f32(W).astype(float), synth.bf16_to_f32(b).astype(float)
    np.testing.assert_allclose(out, Wf @ n + bfv, rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(oracle.project_row(W, None, n), Wf @ n, rtol=1e-12, atol=1e-13)


# ---------------------------------------------------------------- RoPE at the visual positions

def _basis(D, j):
    e = np.zeros(D)
    e[j] = 1.0
    return e


def test_rope_position_zero_is_identity():
    x = np.random.default_rng(2).normal(size=128)
    np.testing.assert_array_equal(oracle.rope_head(x, 0, 10000.0), x)


def test_rope_basis_closed_form():
    # D = 8, theta = 10^4: inverse frequencies 10^4^(-2j/8) = 10^-j = 1, 0.1, 0.01, 0.001.
    # Rotate-half: e_j -> cos(a) e_j + sin(a) e_{j+4};  e_{j+4} -> -sin(a) e_j + cos(a) e_{j+4}.
    p = 7
    for j, f in enumerate([1.0, 0.1, 0.01, 0.001]):
        a = p * f
        y = oracle.rope_head(_basis(8, j), p, 10000.0)
        want = np.zeros(8)
        want[j], want[j + 4] = math.cos(a), math.sin(a)
        np.testing.assert_allclose(y, want, atol=1e-15)
        y = oracle.rope_head(_basis(8, j + 4), p, 10000.0)
        want = np.zeros(8)
        want[j], want[j + 4] = -math.sin(a), math.cos(a)
        np.testing.assert_allclose(y, want, atol=1e-15)


def test_rope_norm_and_relative_position():
    rng = np.random.default_rng(3)
    q, k = rng.normal(size=128), rng.normal(size=128)
    for p in (1, 35, 610, 2914):
        y = oracle.rope_head(q, p, 10000.0)
        # each pair (j, j + 64) keeps its length
        np.testing.assert_allclose(y[:64] ** 2 + y[64:] ** 2, q[:64] ** 2 + q[64:] ** 2, rtol=1e-12)
    for m_, n_ in ((3, 10), (100, 35), (0, 2914)):
        lhs = oracle.rope_head(q, m_, 1e6) @ oracle.rope_head(k, n_, 1e6)
        rhs = q @ oracle.rope_head(k, n_ - m_, 1e6)
        assert lhs == pytest.approx(rhs, rel=1e-10, abs=1e-10)


def test_mrope_equal_axes_is_1d():
    x = np.random.default_rng(4).normal(size=128)
    for p in (0, 15, 51):
        np.testing.assert_allclose(oracle.rope_head(x, (p, p, p), 1e6, True, (16, 24, 24)),
                                   oracle.rope_head(x, p, 1e6), rtol=0, atol=0)


def test_mrope_section_mapping():
    # D = 16 (8 pairs), sections (2, 3, 3): pairs 0-1 follow t, 2-4 follow h, 5-7 follow w.
    sec, theta = (2, 3, 3), 10000.0
    owner = [0, 0, 1, 1, 1, 2, 2, 2]
    for axis in range(3):
        pos = [0, 0, 0]
        pos[axis] = 5
        for j in range(8):
            y = oracle.rope_head(_basis(16, j), pos, theta, True, sec)
            a = 5 * theta ** (-2.0 * j / 16) if owner[j] == axis else 0.0
            assert y[j] == pytest.approx(math.cos(a), abs=1e-15)
            assert y[j + 8] == pytest.approx(math.sin(a), abs=1e-15)


# ---------------------------------------------------------------- the whole build, by hand

def test_end_to_end_hand_example():
    # d = 4, r = 2, one layer, one K/V head of width 4, 1-D position p = 1, eps = 0.
    # Adapter as in test_adapter_hand_example: m = [1, 2 + h0, h1 / 2, -1].
    # gamma = 1, W_K = I, W_V = cyclic shift (v_c = n_{c+1 mod 4}), theta = 10^4 so the two
    # pairs (0, 2), (1, 3) turn by 1 and 0.01 rad. V is not rotated.
    cfg = _tiny_cfg()
    Wv = np.roll(np.eye(4), 1, axis=1)                       # row c picks n_{c+1}
    inp = _inputs(cfg, x0=[[[1, 2, 0, -1]]], D=[[[1, 0, 0, 0], [0, 1, 0, 0]]],
                  U=[[[0, 0], [1, 0], [0, 0.5], [0, 0]]], gamma=[[1, 1, 1, 1]],
                  Wk=[np.eye(4)], Wv=[Wv], pos=[[[1]]])
    out = oracle.build_tokens(inp, want=("k", "v", "m", "n"))
    h0 = 1.0 / (1.0 + math.exp(-1.0))
    h1 = 2.0 / (1.0 + math.exp(-2.0))
    m = np.array([1.0, 2.0 + h0, 0.5 * h1, -1.0])
    n = m / math.sqrt(np.mean(m * m))
    c1, s1, c2, s2 = math.cos(1.0), math.sin(1.0), math.cos(0.01), math.sin(0.01)
    k = [n[0] * c1 - n[2] * s1, n[1] * c2 - n[3] * s2, n[2] * c1 + n[0] * s1, n[3] * c2 + n[1] * s2]
    v = [n[1], n[2], n[3], n[0]]
    np.testing.assert_allclose(out["m"][0, 0], m, rtol=1e-15)
    np.testing.assert_allclose(out["n"][0, 0], n, rtol=1e-14)
    np.testing.assert_allclose(out["k"][0, 0], k, rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(out["v"][0, 0], v, rtol=1e-13, atol=1e-15)


def test_bias_is_added_before_rope():
    # With W_K = 0 the key is the rotated bias: k = RoPE(b_K); the value is the plain bias.
    cfg = _tiny_cfg()
    inp = _inputs(cfg, x0=[[[1, 2, 0, -1]]], D=np.zeros((1, 2, 4)), U=np.zeros((1, 4, 2)),
                  gamma=[[1, 1, 1, 1]], Wk=np.zeros((1, 4, 4)), Wv=np.zeros((1, 4, 4)),
                  pos=[[[3]]], bk=[[0.5, 0, -1, 0]], bv=[[0.25, 0, 0, 1]])
    out = oracle.build_tokens(inp)
    a, b_ = 3.0, 0.03
    want_k = [0.5 * math.cos(a) + 1.0 * math.sin(a), 0.0, -1.0 * math.cos(a) + 0.5 * math.sin(a), 0.0]
    np.testing.assert_allclose(out["k"][0, 0], want_k, atol=1e-15)
    np.testing.assert_allclose(out["v"][0, 0], [0.25, 0, 0, 1], atol=0)
    del b_


def test_unit_gain_zero_update_reduces_to_norm_projection_rope():
    # U = 0 and gamma = 1: K = RoPE(W_K RMSNorm(E)), assembled here from library routines
    # (numpy matmul, elementwise cos/sin) for a 2-head, 3-layer, batch-2 M-RoPE case.
    cfg = synth.Config(name="e2e", d=64, n_layers=3, n_heads=4, n_kv_heads=2, head_dim=16,
                       rank=8, n_vis=12, batch=2, rope="mrope", rope_theta=1e6,
                       mrope_section=(2, 3, 3), rms_eps=1e-6, x0_sigma=1.0, gamma_sigma=0.0,
                       zero_up=True, seed=7, pos_start=15, grid=(1, 3, 4))
    inp = synth.make_inputs(cfg)
    out = oracle.build_tokens(inp)
    x = synth.bf16_to_f32(inp.x0).astype(float).reshape(cfg.tokens, cfg.d)
    nrm = x / np.sqrt(np.mean(x * x, axis=1, keepdims=True) + cfg.rms_eps)
    pos = inp.pos.transpose(0, 2, 1).reshape(cfg.tokens, 3).astype(float)
    j = np.arange(8)
    axis = np.array([0, 0, 1, 1, 1, 2, 2, 2])
    ang = pos[:, axis] * (1e6 ** (-2.0 * j / 16))[None]       # [T, 8]
    c, s = np.cos(ang), np.sin(ang)
    for l in range(cfg.n_layers):
        Wk = synth.bf16_to_f32(inp.Wk[l]).astype(float)
        Wv = synth.bf16_to_f32(inp.Wv[l]).astype(float)
        k = (nrm @ Wk.T).reshape(cfg.tokens, 2, 16)
        k1, k2 = k[..., :8], k[..., 8:]
        kr = np.concatenate([k1 * c[:, None] - k2 * s[:, None], k2 * c[:, None] + k1 * s[:, None]], -1)
        np.testing.assert_allclose(out["k"][:, l], kr.reshape(cfg.tokens, -1), rtol=1e-11, atol=1e-12)
        np.testing.assert_allclose(out["v"][:, l], nrm @ Wv.T, rtol=1e-11, atol=1e-12)


def test_token_subset_matches_full_run():
    # Sampled evaluation (used at full sizes) equals the same rows of a full run.
    cfg, inp = _random_inputs(n_vis=20, batch=2)
    full = oracle.build_tokens(inp)
    sel = np.array([39, 0, 21, 5])
    part = oracle.build_tokens(inp, sel)
    assert np.array_equal(full["k"][sel], part["k"]) and np.array_equal(full["v"][sel], part["v"])


def test_each_batch_element_uses_its_own_positions():
    # Two batch elements with identical embeddings but different positions: the values agree,
    # and the keys differ by exactly the rotation over the position gap (RoPE composes:
    # R(p_b) k = R(p_b - p_a) R(p_a) k).
    cfg = synth.config("tiny", n_vis=6, batch=2)
    inp = synth.make_inputs(cfg)
    inp.x0[1] = inp.x0[0]
    inp.pos = inp.pos.copy()
    inp.pos[1, 0] = inp.pos[0, 0] + 40
    out = oracle.build_tokens(inp)
    kv, Dh = cfg.kv, cfg.head_dim
    for i in range(6):
        a, b = i, 6 + i
        np.testing.assert_array_equal(out["v"][a], out["v"][b])
        for l in range(cfg.n_layers):
            for h in range(cfg.n_kv_heads):
                ka = out["k"][a, l, h * Dh:(h + 1) * Dh]
                kb = out["k"][b, l, h * Dh:(h + 1) * Dh]
                np.testing.assert_allclose(oracle.rope_head(ka, 40, cfg.rope_theta), kb,
                                           rtol=1e-9, atol=1e-12)


def test_layer_subset_matches_full_run():
    cfg, inp = _random_inputs(n_vis=6)
    full = oracle.build_tokens(inp)
    part = oracle.build_tokens(inp, np.array([4, 1]), layers=[3, 0])
    assert np.array_equal(part["k"][0, 0], full["k"][4, 3]) and np.array_equal(part["k"][1, 1], full["k"][1, 0])
    assert np.array_equal(part["v"][0, 1], full["v"][4, 0])


# ---------------------------------------------------------------- recurrent adapter (Sec. 3.1 Eq. 6)

def _silu_by_hand(u):
    return u / (1.0 + math.exp(-u))


def test_recurrent_two_layer_hand_example():
    # E = [a, b, 0, 0]. Layer 1: D_1 reads channel 0, U_1 writes u * h_1 to channel 2, so
    # M_1 = [a, b, u SiLU(a), 0]. Layer 2: D_2 reads channel 2 (zero in E, so only the chained
    # state M_1 feeds it), U_2 writes w * h_2 to channel 3:
    # M_2 = [a, b, u SiLU(a), w SiLU(u SiLU(a))].
    a, b, u, w = 1.0, 2.0, 0.5, 2.0
    cfg = _tiny_cfg(n_layers=2, rank=1, adapter="recurrent")
    D = [[[1, 0, 0, 0]], [[0, 0, 1, 0]]]                           # [L][r][d]
    U = [[[0], [0], [u], [0]], [[0], [0], [0], [w]]]               # [L][d][r]
    eye = np.eye(4)
    inp = _inputs(cfg, [[[a, b, 0, 0]]], D, U, [[1] * 4] * 2, [eye] * 2, [eye] * 2, [[[0]]])
    out = oracle.build_tokens(inp, want=("m", "h"))
    h1 = _silu_by_hand(a)
    h2 = _silu_by_hand(u * h1)
    np.testing.assert_allclose(out["h"][0, :, 0], [h1, h2], rtol=1e-15)
    np.testing.assert_allclose(out["m"][0, 0], [a, b, u * h1, 0.0], rtol=1e-15, atol=0)
    np.testing.assert_allclose(out["m"][0, 1], [a, b, u * h1, w * h2], rtol=1e-15, atol=0)


def test_recurrent_single_layer_equals_embedding():
    # With L = 1, M_1 = A_1(M_0) = A_1(E) for both variants (Eqs. 5 and 6).
    cfg, inp = _random_inputs(n_vis=8, n_layers=1)
    emb = oracle.build_tokens(inp, want=("k", "v", "m"))
    inp_r = dataclasses.replace(inp, cfg=synth.config("tiny", n_vis=8, n_layers=1,
                                                      adapter="recurrent"))
    rec = oracle.build_tokens(inp_r, want=("k", "v", "m"))
    for n in ("k", "v", "m"):
        assert np.array_equal(emb[n], rec[n])


def test_recurrent_zero_up_keeps_embeddings():
    # U_l = 0 makes every A_l the identity, so M_l = E at every depth of the chain.
    cfg = synth.config("tiny", zero_up=True, n_vis=16, adapter="recurrent")
    inp = synth.make_inputs(cfg)
    out = oracle.build_tokens(inp, want=("m",))
    x = synth.bf16_to_f32(inp.x0).astype(np.float64).reshape(cfg.tokens, 1, cfg.d)
    assert np.array_equal(out["m"], np.broadcast_to(x, out["m"].shape))


def test_recurrent_frozen_after_first_layer_matches_embedding_of_first_adapter():
    # U_l = 0 for l >= 2 freezes the chain at M_1 = A_1(E). The embedding variant with A_1
    # copied into every layer also gives M_l = A_1(E), so K/V agree at every layer.
    cfg = synth.config("tiny", n_vis=8, adapter="recurrent", w_sigma=0.1)
    inp = synth.make_inputs(cfg)
    inp.U[1:] = 0
    rec = oracle.build_tokens(inp, want=("k", "v"))
    emb_cfg = synth.config("tiny", n_vis=8, w_sigma=0.1)
    D1 = np.broadcast_to(inp.D[0], inp.D.shape).copy()
    U1 = np.broadcast_to(inp.U[0], inp.U.shape).copy()
    emb = oracle.build_tokens(dataclasses.replace(inp, cfg=emb_cfg, D=D1, U=U1))
    np.testing.assert_allclose(rec["k"], emb["k"], rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(rec["v"], emb["v"], rtol=1e-12, atol=1e-14)


def test_recurrent_updates_lie_in_each_layers_up_span():
    # M_l - M_{l-1} = phi(M_{l-1} D_l) U_l: every token's step at layer l lies in the row space
    # of U_l (r directions), and the accumulated change M_l - E spans at most l * r directions.
    cfg = synth.config("tiny", n_vis=64, rank=4, adapter="recurrent", w_sigma=0.2, x0_sigma=1.0)
    inp = synth.make_inputs(cfg)
    out = oracle.build_tokens(inp, want=("m",))
    x = synth.bf16_to_f32(inp.x0).astype(np.float64).reshape(cfg.tokens, cfg.d)
    prev = x
    for l in range(cfg.n_layers):
        Ul = synth.bf16_to_f32(inp.U[l]).astype(np.float64)          # [d][r]
        q, _ = np.linalg.qr(Ul)                                        # basis of its columns
        step = out["m"][:, l] - prev
        resid = step - (step @ q) @ q.T
        assert np.abs(resid).max() <= 1e-12 * max(np.abs(step).max(), 1e-300)
        assert np.abs(step).max() > 1e-6
        s = np.linalg.svd(out["m"][:, l] - x, compute_uv=False)
        if (l + 1) * cfg.rank < len(s):
            assert s[(l + 1) * cfg.rank] < 1e-9 * s[0]
        prev = out["m"][:, l]


def test_recurrent_layer_subset_matches_full_run():
    # Selected layers still see the whole chain before them.
    cfg = synth.config("tiny", n_vis=6, adapter="recurrent")
    inp = synth.make_inputs(cfg)
    full = oracle.build_tokens(inp)
    part = oracle.build_tokens(inp, np.array([4, 1]), layers=[3, 1])
    assert np.array_equal(part["k"][0, 0], full["k"][4, 3]) and np.array_equal(part["k"][1, 1], full["k"][1, 1])
    assert np.array_equal(part["v"][0, 1], full["v"][4, 1])


# ---------------------------------------------------------------- Qwen3-VL backbone variant
# Per-head RMSNorm of K before RoPE and the interleaved M-RoPE frequency layout.

def test_k_norm_hand_example_norm_before_rope():
    # x0 = [1, 0, 0, 0], eps = 0: RMSNorm gives n = [2, 0, 0, 0]. W_K = 2 I: k = [4, 0, 0, 0]
    # (head rms 2), normalised to [2, 0, 0, 0], times the gain g = [2, 1, 1, 1]: [4, 0, 0, 0].
    # Then RoPE at p = 1 turns pair (0, 2) by 1 rad: K = [4 cos 1, 0, 4 sin 1, 0]. (Rotating
    # first and normalising after would give [4 cos 1, 0, 2 sin 1, 0].) V = 2 n is not normed.
    cfg = _tiny_cfg(k_norm=True, k_norm_eps=0.0)
    inp = _inputs(cfg, x0=[[[1, 0, 0, 0]]], D=np.zeros((1, 2, 4)), U=np.zeros((1, 4, 2)),
                  gamma=[[1, 1, 1, 1]], Wk=[2 * np.eye(4)], Wv=[2 * np.eye(4)], pos=[[[1]]])
    inp.kgamma = bf(np.array([[2.0, 1.0, 1.0, 1.0]]))
    out = oracle.build_tokens(inp)
    np.testing.assert_allclose(out["k"][0, 0], [4 * math.cos(1.0), 0, 4 * math.sin(1.0), 0],
                               rtol=1e-14, atol=1e-15)
    np.testing.assert_allclose(out["v"][0, 0], [4.0, 0, 0, 0], rtol=0, atol=0)


def test_k_norm_closed_form_rms_and_head_independence():
    # Gain 1 and position 0: every key head has rms 1 (eps 0). Scaling the W_K rows of head 0
    # by 4 leaves every head unchanged (each head is normed on its own).
    cfg = synth.config("tiny", n_vis=8, pos_start=0, k_norm=True, k_norm_eps=0.0, k_norm_sigma=0.0)
    inp = synth.make_inputs(cfg)
    inp.pos[:] = 0
    a = oracle.build_tokens(inp)
    kh = a["k"].reshape(cfg.tokens, cfg.n_layers, cfg.n_kv_heads, cfg.head_dim)
    np.testing.assert_allclose(np.sqrt(np.mean(kh * kh, axis=-1)), 1.0, rtol=1e-12)
    Wk = synth.bf16_to_f32(inp.Wk).astype(np.float64)
    Wk[:, :cfg.head_dim] *= 4.0                                 # head 0 of every layer, exact in bf16
    inp.Wk = bf(Wk)
    b = oracle.build_tokens(inp)
    np.testing.assert_allclose(b["k"], a["k"], rtol=1e-12, atol=1e-14)
    np.testing.assert_array_equal(b["v"], a["v"])


def test_k_norm_leaves_values_alone():
    cfg = synth.config("tiny", n_vis=8, k_norm=True)
    inp = synth.make_inputs(cfg)
    plain = oracle.build_tokens(dataclasses.replace(inp, cfg=synth.config("tiny", n_vis=8)))
    normed = oracle.build_tokens(inp)
    np.testing.assert_array_equal(plain["v"], normed["v"])
    assert not np.allclose(plain["k"], normed["k"])


def test_interleaved_mrope_equal_axes_is_1d():
    x = np.random.default_rng(5).normal(size=128)
    for p in (0, 15, 51):
        np.testing.assert_allclose(oracle.rope_head(x, (p, p, p), 5e6, "mrope_interleaved",
                                                    (24, 20, 20)),
                                   oracle.rope_head(x, p, 5e6), rtol=0, atol=0)


def test_interleaved_mrope_mapping():
    # D = 16 (8 pairs), sections (t, h, w) = (4, 2, 2): h takes j = 1, 4 (j = 1 mod 3, j < 6),
    # w takes j = 2, 5 (j = 2 mod 3, j < 6), t takes j = 0, 3, 6, 7.
    sec, theta = (4, 2, 2), 10000.0
    owner = [0, 1, 2, 0, 1, 2, 0, 0]
    for axis in range(3):
        pos = [0, 0, 0]
        pos[axis] = 5
        for j in range(8):
            y = oracle.rope_head(_basis(16, j), pos, theta, "mrope_interleaved", sec)
            a = 5 * theta ** (-2.0 * j / 16) if owner[j] == axis else 0.0
            assert y[j] == pytest.approx(math.cos(a), abs=1e-15)
            assert y[j + 8] == pytest.approx(math.sin(a), abs=1e-15)


# ---------------------------------------------------------------- consumer: text-query attention
# Sec. 3.2: text queries attend causally to [K^v; K^t], [V^v; V^t] (slots in sequence order).

def test_attention_single_visible_key_returns_its_value():
    rng = np.random.default_rng(10)
    q = rng.normal(size=(1, 2, 3, 8))
    k = rng.normal(size=(1, 5, 1, 8))
    v = rng.normal(size=(1, 5, 1, 8))
    out = oracle.text_attention(q, k, v, [5], [[0, 0, 0]], 0.3)
    np.testing.assert_array_equal(out, np.broadcast_to(v[0, 0, 0], out.shape))


def test_attention_two_keys_hand_example_and_no_visible_key():
    # q = e_0, keys 2 e_0 and 0, scale 1/2: scores 1 and 0, weights e/(e+1), 1/(e+1).
    q = np.zeros((1, 1, 2, 4)); q[0, 0, :, 0] = 1.0
    k = np.zeros((1, 3, 1, 4)); k[0, 0, 0, 0] = 2.0
    v = np.zeros((1, 3, 1, 4)); v[0, 0, 0] = [1, 0, 0, 0]; v[0, 1, 0] = [0, 3, 0, 0]
    out = oracle.text_attention(q, k, v, [3], [[1, -1]], 0.5)
    e = math.e
    np.testing.assert_allclose(out[0, 0, 0], [e / (e + 1), 3 / (e + 1), 0, 0], rtol=1e-15)
    np.testing.assert_array_equal(out[0, 0, 1], 0.0)      # slot -1: nothing visible


def test_attention_is_causal_and_respects_key_count():
    # Changing what lies after a query's slot (or past n_keys) leaves its output unchanged.
    rng = np.random.default_rng(11)
    q = rng.normal(size=(2, 2, 4, 16))
    k = rng.normal(size=(2, 12, 2, 16))
    v = rng.normal(size=(2, 12, 2, 16))
    n_keys, q_slot = [12, 9], [[3, 5, 8, 11], [2, 4, 8, 10]]
    a = oracle.text_attention(q, k, v, n_keys, q_slot, 0.25)
    k2, v2 = k.copy(), v.copy()
    k2[0, 9:] += 5.0
    v2[0, 9:] -= 3.0
    k2[1, 9:] *= -2.0                                       # past n_keys of batch 1
    b = oracle.text_attention(q, k2, v2, n_keys, q_slot, 0.25)
    np.testing.assert_array_equal(a[0, :, :3], b[0, :, :3])
    np.testing.assert_array_equal(a[1], b[1])
    assert not np.allclose(a[0, :, 3], b[0, :, 3])


def test_attention_grouped_heads_share_their_kv_head():
    # Hq = 4 over Hkv = 2: heads 0, 1 read kv head 0 and heads 2, 3 kv head 1.
    rng = np.random.default_rng(12)
    q = np.broadcast_to(rng.normal(size=(1, 1, 2, 8)), (1, 4, 2, 8)).copy()
    k = rng.normal(size=(1, 6, 2, 8))
    v = rng.normal(size=(1, 6, 2, 8))
    out = oracle.text_attention(q, k, v, [6], [[4, 5]], 0.35)
    np.testing.assert_array_equal(out[0, 0], out[0, 1])
    np.testing.assert_array_equal(out[0, 2], out[0, 3])
    assert not np.allclose(out[0, 0], out[0, 2])


def test_attention_matches_library_routine():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(13)
    B, Hq, Hkv, Nt, S, D = 2, 4, 2, 5, 20, 16
    q = rng.normal(size=(B, Hq, Nt, D))
    k = rng.normal(size=(B, S, Hkv, D))
    v = rng.normal(size=(B, S, Hkv, D))
    n_keys, q_slot = [20, 15], [[14, 15, 16, 18, 19], [3, 7, 9, 12, 14]]
    got = oracle.text_attention(q, k, v, n_keys, q_slot, 0.25)
    kk = torch.from_numpy(k).permute(0, 2, 1, 3).repeat_interleave(Hq // Hkv, dim=1)
    vv = torch.from_numpy(v).permute(0, 2, 1, 3).repeat_interleave(Hq // Hkv, dim=1)
    s = torch.arange(S)
    mask = torch.stack([(s[None, :] <= torch.tensor(q_slot[b])[:, None]) & (s[None, :] < n_keys[b])
                        for b in range(B)])[:, None]
    ref = torch.nn.functional.scaled_dot_product_attention(torch.from_numpy(q), kk, vv,
                                                           attn_mask=mask, scale=0.25)
    np.testing.assert_allclose(got, ref.numpy(), rtol=1e-12, atol=1e-13)
