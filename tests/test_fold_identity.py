"""The rearrangement of the recurrent adapter's chain that the GPU path computes (CPU only).

With rows of M, D_l [r][d] and U_l [d][r], the chain of Sec. 3.1 Eq. 6 is M_0 = E,
M_l = M_{l-1} + h_l U_l^T with h_l = SiLU(M_{l-1} D_l^T). Unrolling M_{l-1} gives
    z_l = E D_l^T + sum_{j<l} h_j (D_l U_j)^T,    M_l = E + sum_{j<=l} h_j U_j^T,
so the down-projection input of every layer follows from E and the earlier r-wide h_j through
the r x r products D_l U_j, and M_l is a running sum over the layers. These tests check both
identities against the fp64 oracle's own chain (its h_l and M_l), in fp64 with numpy, on a few
tokens: the rearrangement is exact algebra, so they agree to rounding.
"""
import numpy as np
import pytest

import oracle
import synth


def _f64(bits):
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


@pytest.mark.parametrize("n_layers,rank,w_sigma,seed", [(6, 16, 0.05, 3), (12, 40, 0.02, 4)])
def test_rearranged_chain_matches_the_oracle(n_layers, rank, w_sigma, seed):
    cfg = synth.config("tiny", n_layers=n_layers, rank=rank, n_vis=24, w_sigma=w_sigma, seed=seed,
                       adapter="recurrent")
    inp = synth.make_inputs(cfg)
    toks = np.array([0, 5, 11, 23])
    ref = oracle.build_tokens(inp, toks, want=("h", "m"))
    E = _f64(inp.x0).reshape(cfg.tokens, cfg.d)[toks]           # [n][d]
    D, U = _f64(inp.D), _f64(inp.U)                             # [L][r][d], [L][d][r]
    h, m = ref["h"], ref["m"]                                   # [n][L][r], [n][L][d]
    L = cfg.n_layers
    for l in range(L):
        z = E @ D[l].T
        for j in range(l):
            z = z + h[:, j] @ (D[l] @ U[j]).T                   # Q_lj = D_l U_j
        np.testing.assert_allclose(z / (1.0 + np.exp(-z)), h[:, l], rtol=1e-10, atol=1e-12)
        M = E + sum(h[:, j] @ U[j].T for j in range(l + 1))
        np.testing.assert_allclose(M, m[:, l], rtol=1e-10, atol=1e-12)


def test_rearrangement_sees_the_chain_order():
    # A planted reordering (the layers' products taken as D_j U_l instead of D_l U_j) must fail:
    # the identity depends on which layer's D meets which layer's U.
    cfg = synth.config("tiny", n_layers=4, rank=16, n_vis=8, w_sigma=0.1, seed=5, adapter="recurrent")
    inp = synth.make_inputs(cfg)
    toks = np.array([0, 3])
    h = oracle.build_tokens(inp, toks, want=("h",))["h"]
    E = _f64(inp.x0).reshape(cfg.tokens, cfg.d)[toks]
    D, U = _f64(inp.D), _f64(inp.U)
    l = 3
    good = E @ D[l].T + sum(h[:, j] @ (D[l] @ U[j]).T for j in range(l))
    bad = E @ D[l].T + sum(h[:, j] @ (D[j] @ U[l]).T for j in range(l))
    hl = h[:, l]
    assert np.abs(good / (1.0 + np.exp(-good)) - hl).max() < 1e-12
    assert np.abs(bad / (1.0 + np.exp(-bad)) - hl).max() > 1e-6
