"""Splitting one visual-memory build over several GPUs, one process per GPU.

Visual tokens are independent of each other, and given E every layer's memory is independent
of every other layer's (Sec. 3.1: M_l = A_l(E), Eq. 5), so one workload splits two ways with no
exchange of results:

- tokens: rank r builds the flat token rows [r T / N, (r + 1) T / N) of the batch (T = B N_v,
  flat id b N_v + i) into a cache of its own; no collective.
- layers: rank r builds the cache layers [r L / N, (r + 1) L / N) of every token, planning the
  other layers as DV_LAYER_DROP; each step rank 0 broadcasts E, the only collective.

This module holds the host-side partition logic only (ranges, layer modes, the gathered
positions of a token shard, and the check that a partition covers every (token, layer) once);
the builds themselves run through the C ABI on each rank's GPU. The recurrent adapter (Eq. 6)
chains the layers, so it splits by tokens only.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

from . import DV_LAYER_ADAPTER, DV_LAYER_DROP


def even_range(n: int, world: int, rank: int) -> tuple[int, int]:
    """[start, stop) of rank's share of n items split as evenly as possible, in rank order."""
    if world < 1 or not 0 <= rank < world or n < 0:
        raise ValueError(f"bad split: n={n}, world={world}, rank={rank}")
    return rank * n // world, (rank + 1) * n // world


@dataclass(frozen=True)
class TokenShard:
    """A rank's contiguous run of flat token ids [start, stop) of a [B, N_v] batch."""
    start: int
    stop: int
    n_vis: int

    @property
    def tokens(self) -> int:
        return self.stop - self.start

    def segments(self):
        """(batch element, first i, stop i) runs of the shard, in order."""
        out, t = [], self.start
        while t < self.stop:
            b, i = divmod(t, self.n_vis)
            e = min(self.stop, (b + 1) * self.n_vis)
            out.append((b, i, i + e - t))
            t = e
        return out


def token_shard(batch: int, n_vis: int, world: int, rank: int) -> TokenShard:
    start, stop = even_range(batch * n_vis, world, rank)
    return TokenShard(start, stop, n_vis)


def shard_positions(pos: np.ndarray, shard: TokenShard) -> np.ndarray:
    """int32 [1, P, n] positions of the shard's tokens, gathered from pos [B, P, N_v]: the shard
    is built as one batch element of n tokens, each at its own original position(s)."""
    pos = np.asarray(pos)
    if pos.ndim != 3 or pos.shape[2] != shard.n_vis:
        raise ValueError("pos must be [B, P, N_v]")
    parts = [pos[b, :, i0:i1] for b, i0, i1 in shard.segments()]
    if not parts:
        return np.zeros((1, pos.shape[1], 0), dtype=np.int32)
    return np.ascontiguousarray(np.concatenate(parts, axis=1)[None].astype(np.int32))


def layer_shard(n_layers: int, world: int, rank: int) -> tuple[int, int]:
    first, stop = even_range(n_layers, world, rank)
    if stop <= first:
        raise ValueError(f"{n_layers} layers cannot give each of {world} ranks a layer")
    return first, stop


def layer_modes(n_layers: int, world: int, rank: int, base=None) -> list[int]:
    """DV_LAYER_* per cache layer for this rank: its own layers keep their mode (default
    DV_LAYER_ADAPTER), every other layer is DV_LAYER_DROP (no weights, no K/V on this rank)."""
    first, stop = layer_shard(n_layers, world, rank)
    base = [DV_LAYER_ADAPTER] * n_layers if base is None else [int(m) for m in base]
    if len(base) != n_layers:
        raise ValueError("base modes need one entry per layer")
    modes = [base[l] if first <= l < stop else DV_LAYER_DROP for l in range(n_layers)]
    if all(m == DV_LAYER_DROP for m in modes):
        raise ValueError(f"rank {rank} has no layer to build")
    return modes


def check_cover(owned, n_tokens: int, n_layers: int) -> np.ndarray:
    """Every (token, layer) of the workload owned by exactly one rank. ``owned`` lists, per
    rank, (token ids, layer ids) it builds. Returns the [T, L] owner map; raises ValueError on
    a gap or an overlap."""
    owner = np.full((n_tokens, n_layers), -1, dtype=np.int64)
    for r, (toks, lays) in enumerate(owned):
        toks = np.asarray(toks, dtype=np.int64)
        lays = np.asarray(lays, dtype=np.int64)
        if len(np.unique(toks)) != len(toks) or len(np.unique(lays)) != len(lays):
            raise ValueError(f"rank {r} lists a token or a layer twice")
        sub = owner[np.ix_(toks, lays)]
        if (sub != -1).any():
            raise ValueError(f"rank {r} overlaps another rank's (token, layer) entries")
        owner[np.ix_(toks, lays)] = r
    if (owner == -1).any():
        t, l = np.argwhere(owner == -1)[0]
        raise ValueError(f"(token {t}, layer {l}) is built by no rank")
    return owner
