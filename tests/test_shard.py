"""Splitting one workload over ranks (paper_2609_34972_gb300.shard), on CPU.

Tokens are independent and, given E, so are the layers (Sec. 3.1, Eq. 5), so a batch splits by
tokens (no collective) or by layers (E broadcast from rank 0). The partition logic is checked
directly, and then end to end with two gloo ranks: each rank computes its share with the oracle
(standing in for its GPU's build), rank 0 gathers the shares, and every (token, layer) must be
owned by exactly one rank and equal the unsplit build bit for bit.
"""
import os
import pickle
import socket
import sys
from dataclasses import replace

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

from paper_2609_34972_gb300 import shard as sh  # noqa: E402


@pytest.mark.parametrize("n,world", [(10, 3), (7, 7), (0, 2), (23040, 8), (5, 1)])
def test_even_range_partitions_in_order(n, world):
    parts = [sh.even_range(n, world, r) for r in range(world)]
    assert parts[0][0] == 0 and parts[-1][1] == n
    for (a0, a1), (b0, b1) in zip(parts, parts[1:]):
        assert a1 == b0
    sizes = [b - a for a, b in parts]
    assert max(sizes) - min(sizes) <= 1


def test_bad_splits_raise():
    with pytest.raises(ValueError):
        sh.even_range(4, 0, 0)
    with pytest.raises(ValueError):
        sh.even_range(4, 2, 2)
    with pytest.raises(ValueError):
        sh.layer_shard(3, 4, 0)          # 4 ranks, 3 layers: some rank gets none
    with pytest.raises(ValueError):
        sh.layer_modes(4, 2, 0, base=[2, 2, 0, 0])   # rank 0's layers are all dropped


@pytest.mark.parametrize("batch,n_vis,world", [(8, 2880, 3), (2, 5, 4), (1, 576, 2), (3, 7, 1)])
def test_token_shards_cover_the_batch(batch, n_vis, world):
    seen = []
    for r in range(world):
        part = sh.token_shard(batch, n_vis, world, r)
        for b, i0, i1 in part.segments():
            assert 0 <= b < batch and 0 <= i0 < i1 <= n_vis
            seen.extend(b * n_vis + np.arange(i0, i1))
        assert sum(i1 - i0 for _, i0, i1 in part.segments()) == part.tokens
    assert seen == list(range(batch * n_vis))


def test_shard_positions_follow_the_tokens():
    rng = np.random.default_rng(3)
    pos = rng.integers(0, 1000, size=(3, 3, 11)).astype(np.int32)
    part = sh.token_shard(3, 11, 2, 1)            # flat tokens 16..32
    got = sh.shard_positions(pos, part)
    assert got.shape == (1, 3, part.tokens) and got.dtype == np.int32
    flat = pos.transpose(0, 2, 1).reshape(33, 3)  # [token][axis]
    assert np.array_equal(got[0].T, flat[part.start:part.stop])


def test_layer_modes_partition_the_layers():
    L, world = 32, 3
    modes = [sh.layer_modes(L, world, r) for r in range(world)]
    for l in range(L):
        owners = [r for r in range(world) if modes[r][l] != sh.DV_LAYER_DROP]
        assert len(owners) == 1
    base = [1] * 4 + [0] * 24 + [2] * 4          # identity, adapter, dropped (App. J)
    m = [sh.layer_modes(L, 2, r, base) for r in range(2)]
    assert m[0][:4] == [1] * 4 and m[1][28:] == [2] * 4 and m[1][:16] == [2] * 16


def test_check_cover_finds_gaps_and_overlaps():
    T, L = 6, 4
    ok = [(range(0, 3), range(L)), (range(3, 6), range(L))]
    assert (sh.check_cover(ok, T, L)[3:] == 1).all()
    with pytest.raises(ValueError):
        sh.check_cover([(range(0, 4), range(L)), (range(3, 6), range(L))], T, L)   # overlap
    with pytest.raises(ValueError):
        sh.check_cover([(range(0, 3), range(L)), (range(4, 6), range(L))], T, L)   # gap
    with pytest.raises(ValueError):
        sh.check_cover([([0, 0, 1, 2, 3, 4, 5], range(L))], T, L)                 # duplicate


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _split_worker(rank, world, port, out_dir):
    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), OMP_NUM_THREADS="1")
    import oracle
    import synth
    from paper_2609_34972_gb300 import shard as sh
    dist.init_process_group("gloo", rank=rank, world_size=world)
    cfg = synth.config("tiny", batch=3, n_vis=40, seed=9, bias_sigma=0.02)
    inp = synth.make_inputs(cfg)

    # token split: this rank's flat tokens as one batch element at their own positions
    part = sh.token_shard(cfg.batch, cfg.n_vis, world, rank)
    x0_flat = inp.x0.reshape(cfg.tokens, cfg.d)
    sub = replace(inp, cfg=replace(cfg, batch=1, n_vis=part.tokens),
                  x0=np.ascontiguousarray(x0_flat[part.start:part.stop][None]),
                  pos=sh.shard_positions(inp.pos, part))
    tok = oracle.build_tokens(sub)
    tok_share = (np.arange(part.start, part.stop), np.arange(cfg.n_layers), tok["k"], tok["v"])

    # layer split: E arrives by broadcast from rank 0 (the other ranks start from zeros); its bf16
    # bit patterns travel as bytes
    nbytes = inp.x0.size * 2
    x0 = torch.from_numpy(np.ascontiguousarray(inp.x0).reshape(-1).view(np.uint8).copy()) if rank == 0 \
        else torch.zeros(nbytes, dtype=torch.uint8)
    dist.broadcast(x0, src=0)
    first, stop = sh.layer_shard(cfg.n_layers, world, rank)
    modes = sh.layer_modes(cfg.n_layers, world, rank)
    layers = [l for l, m in enumerate(modes) if m != sh.DV_LAYER_DROP]
    assert layers == list(range(first, stop))
    got = replace(inp, x0=x0.numpy().view(np.uint16).reshape(inp.x0.shape))
    lay = oracle.build_tokens(got, layers=layers)
    lay_share = (np.arange(cfg.tokens), np.array(layers), lay["k"], lay["v"])

    shares = [None] * world if rank == 0 else None
    dist.gather_object((tok_share, lay_share), shares, dst=0)
    if rank == 0:
        with open(os.path.join(out_dir, "shares.pkl"), "wb") as f:
            pickle.dump(shares, f)
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_token_and_layer_splits_reassemble_the_build_gloo(tmp_path, world):
    mp = pytest.importorskip("torch.multiprocessing")
    import oracle
    import synth
    mp.spawn(_split_worker, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    shares = pickle.load(open(tmp_path / "shares.pkl", "rb"))
    cfg = synth.config("tiny", batch=3, n_vis=40, seed=9, bias_sigma=0.02)
    full = oracle.build_tokens(synth.make_inputs(cfg))
    for which in (0, 1):                          # 0: token split, 1: layer split
        parts = [s[which] for s in shares]
        sh.check_cover([(t, l) for t, l, _, _ in parts], cfg.tokens, cfg.n_layers)
        k = np.full_like(full["k"], np.nan)
        v = np.full_like(full["v"], np.nan)
        for t, l, pk, pv in parts:
            k[np.ix_(t, l)] = pk
            v[np.ix_(t, l)] = pv
        assert np.array_equal(k, full["k"]) and np.array_equal(v, full["v"]), which
