"""Population-parallel discovery over several processes (one GPU each).

The path shards with no exchange: each rank discovers the connection lists of
its own contiguous genome range (emr_partition_genomes balances the ranges by
the packed cost estimates; emr.pack_population(pop, genomes=(g0, g1)) packs
one range). The only collective is the optional gather of every rank's counts
and lists to the rank that assembles the substrate networks, here over
torch.distributed (NCCL with device tensors, gloo with host tensors).
Concatenated in rank order, the ranges' lists are the whole population's lists
(pair r = g * S + s), identical to a single-process run.
"""
from __future__ import annotations

import numpy as np
import torch
import torch.distributed as dist

from . import emr


def genome_ranges(pack_full: np.ndarray, query, world: int) -> np.ndarray:
    """Genome range boundaries of the world's ranks: int32 [world + 1]."""
    return emr.partition_genomes(pack_full, query, world)


def range_sources(sources, g0: int, g1: int):
    """The query slots of genomes [g0, g1): shared slots unchanged, per-genome rows sliced."""
    if not sources.per_genome:
        return sources
    from .workloads import Sources
    return Sources(a=sources.a[g0:g1], b=sources.b[g0:g1], side=sources.side[g0:g1],
                   count=None if sources.count is None else sources.count[g0:g1])


def gather_lists(counts: torch.Tensor, idx: torch.Tensor, w: torch.Tensor, dst: int = 0, group=None):
    """Gather every rank's lists to rank dst. counts: int64 [pairs of this rank]; idx (int32) and
    w (float32): this rank's entries in pair order (pair k's list is counts[k] entries after
    those of pairs 0..k-1). On dst returns (counts, offsets, idx, w) of all ranks concatenated in
    rank order (offsets: int64 [pairs + 1], exclusive prefix of counts); None elsewhere. All
    tensors on one device: host for gloo, the rank's GPU for NCCL."""
    rank, world = dist.get_rank(group), dist.get_world_size(group)
    dev = counts.device
    size = torch.tensor([counts.numel(), idx.numel()], dtype=torch.int64, device=dev)
    sizes = [torch.empty_like(size) for _ in range(world)]
    dist.all_gather(sizes, size, group=group)
    sizes = [tuple(int(v) for v in s.cpu()) for s in sizes]
    max_p = max(1, max(s[0] for s in sizes))
    max_e = max(1, max(s[1] for s in sizes))

    def padded(t, n):
        out = torch.zeros(n, dtype=t.dtype, device=dev)
        out[:t.numel()] = t.reshape(-1)
        return out

    parts = {}
    for name, t, n in (("counts", counts, max_p), ("idx", idx, max_e), ("w", w, max_e)):
        buf = padded(t, n)
        lst = [torch.empty_like(buf) for _ in range(world)] if rank == dst else None
        dist.gather(buf, lst, dst=dst, group=group)
        parts[name] = lst
    if rank != dst:
        return None
    cnt = torch.cat([parts["counts"][k][:sizes[k][0]] for k in range(world)])
    ix = torch.cat([parts["idx"][k][:sizes[k][1]] for k in range(world)])
    wv = torch.cat([parts["w"][k][:sizes[k][1]] for k in range(world)])
    off = torch.zeros(cnt.numel() + 1, dtype=torch.int64, device=dev)
    off[1:] = torch.cumsum(cnt, 0)
    return cnt, off, ix, wv
