"""Row-sharded retrieval on one GPU: the shards' keys (combined by an elementwise maximum,
the all-reduce MAX that ranks would run) decode to exactly the rows and scores that
precog_retrieve returns on the whole index, including ties across shard boundaries, NaN
rows and empty shards."""
import numpy as np
import pytest

import synth

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dtype_name,Q", [("float16", 1), ("float16", 200), ("bfloat16", 7), ("float32", 5)])
def test_shard_keys_combine_to_whole_index_top1(cuda_device, dtype_name, Q):
    import torch
    import paper_2608_02560_gb300 as pg
    from paper_2608_02560_gb300.distributed import sharded_retrieve, shard_rows
    d = cuda_device
    dtype = getattr(torch, dtype_name)
    M, dim = 10000, 128
    index = synth.device_unit_index(M, dim, 11, d, dtype=dtype)
    q, _ = synth.device_planted_queries(index, Q, synth.QUERY_NOISE, 12)
    # ties across shard boundaries: the planted rows' duplicates sit in later shards
    index[5000] = index[1234]
    index[9999] = index[2999]
    q[0] = index[1234]
    if Q > 1:
        q[1] = index[2999]
    index[4321] = float("nan")
    ref_idx = torch.empty(Q, dtype=torch.int64, device=d)
    ref_score = torch.empty(Q, dtype=torch.float32, device=d)
    pg.precog_retrieve(index, q, ref_idx, ref_score)
    bounds = [0, 3000, 3001, 3001, 7000, M]          # a one-row and an empty shard
    keys = []
    for a, b in zip(bounds[:-1], bounds[1:]):
        k = torch.empty(Q, dtype=torch.int64, device=d)
        pg.precog_retrieve_keys(index[a:b], q, a, k)
        keys.append(k)
    combined = torch.stack(keys).max(dim=0).values
    idx = torch.empty(Q, dtype=torch.int64, device=d)
    score = torch.empty(Q, dtype=torch.float32, device=d)
    pg.precog_decode_keys(combined, idx, score)
    assert pg.precog_device_status()[0] == 0
    assert torch.equal(idx, ref_idx)
    assert torch.equal(score, ref_score)
    assert int(idx[0]) == 1234 and (Q == 1 or int(idx[1]) == 2999)
    # the helper without a process group is the single-shard case
    one = torch.empty(Q, dtype=torch.int64, device=d)
    sharded_retrieve(index, q, 0, one)
    assert torch.equal(one, ref_idx)
    assert shard_rows(M, 3, 0) == (0, 3334) and shard_rows(M, 3, 2) == (6667, 3333)


def test_empty_shard_and_no_row_keys(cuda_device):
    """A shard with no rows gives the 'no row' key; decoding it gives -1 and NaN."""
    import torch
    import paper_2608_02560_gb300 as pg
    d = cuda_device
    q = synth.device_unit_index(3, 64, 1, d, dtype=torch.float16)
    k = torch.empty(3, dtype=torch.int64, device=d)
    pg.precog_retrieve_keys(q[:0], q, 17, k)
    assert torch.all(k == torch.iinfo(torch.int64).min)
    idx = torch.empty(3, dtype=torch.int64, device=d)
    sc = torch.empty(3, dtype=torch.float32, device=d)
    pg.precog_decode_keys(k, idx, sc)
    assert torch.all(idx == -1) and torch.all(torch.isnan(sc))
