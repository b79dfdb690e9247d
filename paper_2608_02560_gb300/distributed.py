"""Row-sharded retrieval across ranks (one process per GPU).

Every rank holds a contiguous block of the index's rows (`shard_rows`). For a batch of
queries each rank computes its shard's best key per query on its GPU
(`precog_retrieve_keys`), one all-reduce MAX over the int64 keys combines the shards --
the exchange step of the sharded path -- and every rank decodes the same result
(`precog_decode_keys`): the exact top-1 of the whole index, ties to the lowest global row,
as `precog_retrieve` would return on the unsharded index. The state bank is sharded the
same way (`gather_owned_states`): the rank that owns a winning row copies it from its own
memory, the others contribute zeros, and one all-reduce SUM hands every rank the
injected states; no rank reads another's memory.
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


def gather_owned_states(bank_shard, row_offset: int, best_idx, out, group=None):
    """The injected states of a row-sharded bank: ``out[q] = bank[best_idx[q]]`` on every
    rank, ``bank_shard`` holding this rank's rows ``row_offset ..``. The owner of a row
    copies it from its own memory, the other ranks write zeros, and one all-reduce SUM over
    ``out`` combines the ranks (adding zeros leaves every value as it is, up to the sign
    of a zero). A row of -1 (nothing comparable) gives the zero state, as injecting -1
    does. Runs on torch's current stream; no host synchronisation."""
    import torch
    import torch.distributed as dist
    rows = bank_shard.shape[0]
    flat = out.view(out.shape[0], -1)
    if rows == 0:
        flat.zero_()
    else:
        local = best_idx - row_offset
        owned = (local >= 0) & (local < rows)
        picked = bank_shard.view(rows, -1).index_select(0, local.clamp(0, rows - 1))
        flat.copy_(torch.where(owned[:, None], picked, torch.zeros((), dtype=picked.dtype,
                                                                    device=picked.device)))
    if dist.is_available() and dist.is_initialized() and dist.get_world_size(group) > 1:
        dist.all_reduce(out, op=dist.ReduceOp.SUM, group=group)
    return out
