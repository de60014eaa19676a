"""Token sharding across ranks (one process per GPU).

Tokens are independent through the routed FFN stack (every step of a routed
block is per token; the depth memory is per token), so a batch splits into
contiguous token shards with replicated weights and no collective on the data
path.  Only the final hidden states (and optional routing statistics) are
gathered, outside the timed stack.
"""

from __future__ import annotations

from typing import List, Tuple


def shard_range(n_tokens: int, rank: int, world: int) -> Tuple[int, int]:
    """Contiguous, balanced shard [start, start + count) of n_tokens for `rank`."""
    if world < 1 or not (0 <= rank < world):
        raise ValueError(f"bad rank {rank} of world {world}")
    if n_tokens < 0:
        raise ValueError("n_tokens must be >= 0")
    base, extra = divmod(n_tokens, world)
    start = rank * base + min(rank, extra)
    return start, base + (1 if rank < extra else 0)


def shard_sizes(n_tokens: int, world: int) -> List[int]:
    return [shard_range(n_tokens, r, world)[1] for r in range(world)]


def gather_shards(pg_all_gather, local, n_tokens: int, world: int):
    """Reassemble per-rank [count_r, ...] torch tensors into [n_tokens, ...].

    pg_all_gather(list_of_outputs, input) is torch.distributed.all_gather (any
    backend); shards are padded to the largest shard for the collective.
    """
    import torch
    sizes = shard_sizes(n_tokens, world)
    cap = max(sizes) if sizes else 0
    pad = torch.zeros((cap,) + tuple(local.shape[1:]), dtype=local.dtype, device=local.device)
    pad[: local.shape[0]] = local
    outs = [torch.empty_like(pad) for _ in range(world)]
    pg_all_gather(outs, pad)
    return torch.cat([o[:s] for o, s in zip(outs, sizes)], dim=0)
