"""Running the path on several GPUs as independent replicas.

Every image (and every candidate-group episode) is independent through
selection, compaction and prefill, so a global batch splits across ranks with
no exchange on the data path.  This module holds the host-side pieces: the
partition of a batch's images over ranks, balanced by the tokens each image
brings, and the max-over-ranks reduction used for timing.
"""
from __future__ import annotations

import heapq
from typing import List, Sequence


def shard_images(n_vis: Sequence[int], n_txt: Sequence[int], world: int, rank: int) -> List[int]:
    """Image indices of `rank` when the batch is spread over `world` ranks.

    Longest-processing-time-first greedy on the per-image token count
    N_b + L_b (the selector encoder's sequence length, which also bounds the
    prefill length); ties broken by image index so every rank computes the same
    partition.  Returns the indices in ascending order."""
    if world < 1 or not (0 <= rank < world):
        raise ValueError("need 0 <= rank < world")
    if len(n_vis) != len(n_txt):
        raise ValueError("n_vis and n_txt differ in length")
    order = sorted(range(len(n_vis)), key=lambda b: (-(int(n_vis[b]) + int(n_txt[b])), b))
    heap = [(0, r) for r in range(world)]
    owner = {}
    for b in order:
        load, r = heapq.heappop(heap)
        owner[b] = r
        heapq.heappush(heap, (load + int(n_vis[b]) + int(n_txt[b]), r))
    return sorted(b for b, r in owner.items() if r == rank)


def max_over_ranks(value: float, device=None) -> float:
    """The maximum of `value` over the ranks of the default process group (the
    value itself when torch.distributed is not initialised)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return float(value)
    if device is None:
        device = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())
