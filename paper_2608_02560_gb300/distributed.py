"""Row-sharded retrieval across ranks (one process per GPU).

Every rank holds a contiguous block of the index's rows (`shard_rows`). For a batch of
queries each rank computes its shard's best key per query on its GPU
(`precog_retrieve_keys`), one all-reduce MAX over the int64 keys combines the shards --
the exchange step of the sharded path -- and every rank decodes the same result
(`precog_decode_keys`): the exact top-1 of the whole index, ties to the lowest global row,
as `precog_retrieve` would return on the unsharded index. The state bank can be sharded
the same way; the rank that owns the winning row then serves its state.
"""
from __future__ import annotations

from . import precog_decode_keys, precog_retrieve_keys


def shard_rows(M: int, world: int, rank: int):
    """(row_offset, rows) of rank's block when M rows are split as evenly as possible."""
    base, extra = divmod(M, world)
    rows = base + (1 if rank < extra else 0)
    offset = rank * base + min(rank, extra)
    return offset, rows


def combine_keys(keys, group=None):
    """Combine the shards' keys in place: the signed maximum over ranks (keys are ordered
    as int64 by score, then lower row), a no-op without a process group of several ranks."""
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized() and dist.get_world_size(group) > 1:
        dist.all_reduce(keys, op=dist.ReduceOp.MAX, group=group)
    return keys


def sharded_retrieve(index_shard, queries, row_offset: int, best_idx, best_score=None, group=None,
                     workspace=None):
    """Exact top-1 over the row-sharded index (this rank's rows start at ``row_offset``);
    every rank receives the same global rows and scores. Runs on torch's current stream,
    which the collective also uses."""
    import torch
    keys = torch.empty(queries.shape[0], dtype=torch.int64, device=queries.device)
    precog_retrieve_keys(index_shard, queries, row_offset, keys, workspace=workspace)
    combine_keys(keys, group)
    precog_decode_keys(keys, best_idx, best_score)
    return best_idx
