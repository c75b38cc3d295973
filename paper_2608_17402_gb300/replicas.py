"""Host-side logic of the multi-GPU benchmark: one process per GPU, tokens sharded.

The layer is independent per token (Eqs. 1-7 involve no cross-token term), so a
batch splits across ranks by contiguous token ranges with no data-path
collective: each rank runs the whole layer on its own tokens.  The only
communication is timing: every rank's measured time is reduced with MAX, so that
the reported step time is that of the slowest rank.  Works with the gloo (CPU)
and nccl (GPU) backends.
"""
from __future__ import annotations

import torch
import torch.distributed as dist


def token_shard(T: int, rank: int, world: int) -> tuple[int, int]:
    """Contiguous range ``[start, stop)`` of the T tokens owned by ``rank``.

    Shards differ in size by at most one token; their concatenation in rank order
    is ``range(T)``."""
    if world < 1 or not 0 <= rank < world or T < 0:
        raise ValueError(f"bad shard request T={T} rank={rank} world={world}")
    base, extra = divmod(T, world)
    start = rank * base + min(rank, extra)
    return start, start + base + (1 if rank < extra else 0)


def max_over_ranks(values, device=None):
    """Element-wise maximum of ``values`` (a sequence of floats) over all ranks.

    Without an initialised process group (a single process) the values come back
    unchanged.  ``device`` must be a CUDA device for the nccl backend."""
    vals = [float(v) for v in values]
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return vals
    t = torch.tensor(vals, dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t.cpu()]
