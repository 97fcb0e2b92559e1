"""GPU parity over a seeded random sweep of small configurations, each compared element by
element with the fp64 oracle over every token.

The sweep draws what the ABI accepts and the engines branch on: hidden sizes with odd and even
K-slab counts, every rank padding (r_pad 64, 128, 192, 256), both head widths and several KV
head counts, token counts that pick the 1-SM or the 2-SM rank-r engine and either K/V engine
(ragged tails included), 1-D, contiguous and interleaved M-RoPE, K/V bias, the per-head K
norm, both adapters, and per-layer modes (adapter, identity, dropped). The draw is fixed by the
seed, so a failure names a reproducible case. Weights are drawn with the workloads' sigma (0.02):
with larger recurrent adapters the chain's bf16 operands (M_l, h_l) let the error grow with depth
(1.2e-2 at layer 0 to 2.2e-2 at layer 5 for sigma 0.05 in one drawn case), a property of bf16
GEMMs in the chain rather than of one kernel.
"""
from dataclasses import replace

import numpy as np
import pytest

import oracle
import synth
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu

N_CASES = 24


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_34972_gb300.build import build_library
    build_library()


def _draw(i):
    rs = np.random.RandomState(1000 + i)
    hd = int(rs.choice([64, 128]))
    n_kv = int(rs.choice([2, 4, 6, 8])) if hd == 64 else int(rs.choice([1, 2, 3, 4]))
    d = int(rs.choice([64, 128, 192, 256, 320, 448, 512, 640, 768, 1024]))
    L = int(rs.randint(1, 7))
    rank = int(rs.randint(1, 257))
    batch = int(rs.choice([1, 2, 3]))
    rope = str(rs.choice(["1d", "mrope", "mrope_interleaved"]))
    grid, sec = (), (0, 0, 0)
    if rope == "1d":
        n_vis = int(rs.randint(1, 400))
    else:
        frames, rows, cols = int(rs.choice([1, 2])), int(rs.randint(1, 20)), int(rs.randint(1, 20))
        n_vis, grid = frames * rows * cols, (frames, rows, cols)
        if rope == "mrope":
            sec = (16, 24, 24) if hd == 128 else (8, 12, 12)
        else:
            sec = (24, 20, 20) if hd == 128 else (12, 10, 10)
    adapter = "recurrent" if rs.rand() < 0.3 else "embedding"
    cfg = gu.small_config(
        f"sweep{i}", d=d, n_layers=L, n_kv_heads=n_kv, n_heads=n_kv * int(rs.choice([1, 2])),
        head_dim=hd, rank=rank, n_vis=n_vis, batch=batch, rope=rope,
        rope_theta=float(rs.choice([1e4, 1e6])), mrope_section=sec, grid=grid,
        x0_sigma=0.5, w_sigma=0.02,
        bias_sigma=0.02 if rs.rand() < 0.4 else 0.0, k_norm=bool(rs.rand() < 0.3),
        adapter=adapter, seed=2000 + i, pos_start=int(rs.randint(0, 50)))
    modes = None
    if L > 1 and rs.rand() < 0.35:
        modes = [int(m) for m in rs.choice([0, 0, 1, 2], size=L)]
        if all(m == 2 for m in modes):
            modes[0] = 0
    return cfg, modes


@pytest.mark.parametrize("i", range(N_CASES))
def test_random_configuration(i):
    cfg, modes = _draw(i)
    inp = synth.make_inputs(cfg)
    k, v, plan = gu.run_build(inp, fill=-7.0, layer_modes=modes)
    ref_inp = inp
    kept = list(range(cfg.n_layers))
    if modes is not None:
        D, U = inp.D.copy(), inp.U.copy()
        for l, m in enumerate(modes):
            if m != 0:  # identity and dropped layers pass M unchanged (the adapter is zero)
                D[l] = 0
                U[l] = 0
        ref_inp = replace(inp, D=D, U=U)
        kept = [l for l, m in enumerate(modes) if m != 2]
    toks = np.arange(cfg.tokens)
    ref = oracle.build_tokens(ref_inp, toks, layers=kept)
    gk = gu.gather(k, cfg, toks)[:, kept]
    gv = gu.gather(v, cfg, toks)[:, kept]
    label = (f"sweep {i}: d={cfg.d} L={cfg.n_layers} kv={cfg.n_kv_heads}x{cfg.head_dim} r={cfg.rank} "
             f"T={cfg.batch}x{cfg.n_vis} {cfg.rope} bias={cfg.bias_sigma > 0} knorm={cfg.k_norm} "
             f"{cfg.adapter} modes={modes}")
    gu.assert_parity(gk, gv, ref["k"], ref["v"], cfg.head_dim, label)
    if modes is not None:
        for l, m in enumerate(modes):
            if m == 2:
                assert bool((k[l] == -7.0).all()) and bool((v[l] == -7.0).all()), f"{label}: layer {l} written"
