"""The multi-rank host logic of bench.py on CPU: two gloo ranks on 127.0.0.1. Each rank
encodes its own corpus shard (different chunks, same shape; no exchange on the data path),
the timed region is the slowest rank's time, and the reported rate counts the units of all
ranks. No GPU is touched."""
import os
import socket

import pytest


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, queue):
    import torch
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        import synth
        seed = bench.shard_seed(rank)
        inp = synth.device_scan_inputs(64, 16, 16, seed, 0, torch.device("cpu"), with_C=False)
        x = inp["x"].float()
        gathered = [torch.empty_like(x) for _ in range(world)]
        dist.all_gather(gathered, x)
        distinct = not torch.equal(gathered[0], gathered[1])
        slowest = bench.reduce_max(1.0 + rank, world, torch.device("cpu"))
        rate = bench.whole_job_rate(1000, world, 5, slowest)
        queue.put((rank, seed, distinct, slowest, rate, tuple(x.shape)))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_shard_and_reduce():
    mp = pytest.importorskip("torch.multiprocessing")
    ctx = mp.get_context("spawn")
    queue = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, queue)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=180)
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    res = sorted(queue.get(timeout=10) for _ in range(2))
    (r0, s0, d0, t0, v0, sh0), (r1, s1, d1, t1, v1, sh1) = res
    assert (r0, r1) == (0, 1) and s0 != s1            # each rank its own shard
    assert sh0 == sh1 and d0 and d1                   # same shape, different chunks
    assert t0 == t1 == 2.0                            # both ranks report the slowest time
    assert v0 == v1 == 2 * 1000 * 5 / 2.0             # units of all ranks / slowest time


def test_single_rank_helpers():
    import bench
    assert bench.shard_seed(0) == 0 and bench.shard_seed(3) == 3000
    assert bench.reduce_max(4.5, 1, None) == 4.5
    assert bench.whole_job_rate(10, 1, 3, 2.0) == 15.0


def _key(score, row):
    """The documented shard key, written out independently: ordered score bits << 32 |
    (2^32 - 1 - row), top bit flipped so that keys order as int64 (None: no row)."""
    import numpy as np
    if score is None:
        return -(1 << 63)
    u = int(np.array([score + 0.0], dtype=np.float32).view(np.uint32)[0])
    ordered = (~u & 0xffffffff) if u & 0x80000000 else (u | 0x80000000)
    k = ((ordered << 32) | (0xffffffff - row)) ^ (1 << 63)
    return k - (1 << 64) if k >= (1 << 63) else k


def _key_row(k):
    if k == -(1 << 63):
        return -1
    return 0xffffffff - ((k + (1 << 64)) % (1 << 64) & 0xffffffff)


# per query: (rank 0's best, rank 1's best) as (score, global row) or None
_SHARD_BEST = [((0.9, 10), (0.8, 150)),        # the higher score wins
               ((0.7, 20), (0.7, 120)),        # a tie: the lower global row
               (None, (-0.5, 199)),            # one empty shard, a negative score
               (None, None),                   # no comparable row anywhere
               ((-0.0, 5), (0.0, 101))]        # -0 and +0 are the same score


def _combine_main(rank, world, port, queue):
    import torch
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        from paper_2608_02560_gb300.distributed import combine_keys, shard_rows
        keys = torch.tensor([_key(*b[rank]) if b[rank] else _key(None, 0) for b in _SHARD_BEST],
                            dtype=torch.int64)
        combine_keys(keys)
        queue.put((rank, [_key_row(int(k)) for k in keys], shard_rows(200, world, rank)))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_combine_shard_keys():
    """Row-sharded retrieval's exchange step: an all-reduce MAX over the shards' int64 keys
    picks the higher score, then the lower global row, across ranks."""
    mp = pytest.importorskip("torch.multiprocessing")
    ctx = mp.get_context("spawn")
    queue = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_combine_main, args=(r, 2, port, queue)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=180)
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    res = sorted(queue.get(timeout=10) for _ in range(2))
    (_, rows0, sh0), (_, rows1, sh1) = res
    assert rows0 == rows1 == [10, 20, 199, -1, 5]
    assert sh0 == (0, 100) and sh1 == (100, 100)


@pytest.mark.parametrize("M,world", [(0, 1), (0, 3), (1, 4), (7, 2), (10000, 3), (1_000_000, 8), (5, 8)])
def test_shard_rows_tile_the_index(M, world):
    """The ranks' row blocks are contiguous, in rank order, cover [0, M) exactly once and
    differ in size by at most one row."""
    from paper_2608_02560_gb300.distributed import shard_rows
    blocks = [shard_rows(M, world, r) for r in range(world)]
    pos = 0
    for off, rows in blocks:
        assert off == pos and rows >= 0
        pos += rows
    assert pos == M
    sizes = [rows for _, rows in blocks]
    assert max(sizes) - min(sizes) <= 1


def _gather_main(rank, world, port, queue):
    import torch
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        from paper_2608_02560_gb300.distributed import gather_owned_states, shard_rows
        M, L, E = 11, 2, 6
        bank = torch.arange(M * L * E, dtype=torch.float32).view(M, L, E) - 20.0
        bank[4, 1, 2] = float("nan")
        off, rows = shard_rows(M, world, rank)
        idx = torch.tensor([0, 10, 5, -1, 4, 5, 6], dtype=torch.int64)
        out = torch.full((idx.numel(), L, E), 7.0)
        gather_owned_states(bank[off:off + rows].clone(), off, idx, out)
        queue.put((rank, out.numpy().tolist()))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_gather_owned_states():
    """Sharded injection: every rank ends with the global bank rows its queries won (rows
    owned by either rank, a repeated row, a NaN entry), and row -1 gives the zero state."""
    import numpy as np
    import torch
    mp = pytest.importorskip("torch.multiprocessing")
    ctx = mp.get_context("spawn")
    queue = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_gather_main, args=(r, 2, port, queue)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=180)
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    res = sorted(queue.get(timeout=10) for _ in range(2))
    bank = torch.arange(11 * 2 * 6, dtype=torch.float32).view(11, 2, 6) - 20.0
    bank[4, 1, 2] = float("nan")
    want = torch.stack([bank[i] if i >= 0 else torch.zeros(2, 6) for i in (0, 10, 5, -1, 4, 5, 6)]).numpy()
    for _, got in res:
        np.testing.assert_array_equal(np.array(got), want)
