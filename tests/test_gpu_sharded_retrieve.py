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


def test_sharded_query_path_equals_whole_bank_injection(cuda_device):
    """The sharded query path of several ranks, emulated on one GPU: every shard of the
    bank contributes its owned winning rows (gather_owned_states without a process group),
    the sum over shards is the all-reduce the ranks run, and prefilling from those gathered
    states (no index) gives exactly the y and states of injecting from the whole bank."""
    import torch
    import paper_2608_02560_gb300 as pg
    from paper_2608_02560_gb300.distributed import gather_owned_states, shard_rows
    d = cuda_device
    M, L, D, N, Tq, Q = 1000, 3, 64, 16, 20, 6
    bank = synth.device_normal_bank(M, L * D * N, 4, d).view(M, L, D, N)
    idx = torch.tensor([0, 999, 333, -1, 334, 333], dtype=torch.int64, device=d)
    ins = [synth.device_scan_inputs(Q * Tq, D, N, 9, l, d) for l in range(L)]
    st = lambda k: torch.stack([i[k] for i in ins]).contiguous()
    si = pg.scan_inputs(st("x"), st("dt"), st("B"), st("A"), st("C"), a_kind=pg.PRECOG_A_POWER)
    y_ref = torch.empty((L, Q * Tq, D), dtype=torch.bfloat16, device=d)
    h_ref = torch.empty((Q, L, D, N), dtype=torch.bfloat16, device=d)
    pg.precog_prefill_from_state(si, Q, Tq, bank, idx=idx, y_out=y_ref, state_out=h_ref)
    world = 3
    total = torch.zeros((Q, L, D, N), dtype=torch.float32, device=d)
    for r in range(world):
        off, rows = shard_rows(M, world, r)
        part = torch.empty((Q, L, D, N), dtype=torch.bfloat16, device=d)
        gather_owned_states(bank[off:off + rows], off, idx, part)
        total += part.float()
    inj = total.to(torch.bfloat16)
    assert torch.equal(inj[3], torch.zeros_like(inj[3])) and torch.equal(inj[0], bank[0])
    y = torch.empty_like(y_ref)
    h = torch.empty_like(h_ref)
    pg.precog_prefill_from_state(si, Q, Tq, inj, idx=None, y_out=y, state_out=h)
    assert pg.precog_device_status()[0] == 0
    assert torch.equal(y, y_ref) and torch.equal(h, h_ref)
