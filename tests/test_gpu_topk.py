"""GPU parity of top-k retrieval and of the softmax-weighted top-k state composition
(Sec. 4.4 multi-chunk extension, Eq. smc-fusion) against the oracle."""
import numpy as np
import pytest

import oracle
import synth
from tests._util import TOL_BF16, TOL_F32, rel_err, rel_err_stored, to_np

pytestmark = pytest.mark.gpu


def _pg():
    import paper_2608_02560_gb300 as pg
    return pg


def _topk(index, queries, k):
    import torch
    pg = _pg()
    Q = queries.shape[0]
    idx = torch.full((Q, k), -7, dtype=torch.int64, device=index.device)
    score = torch.empty((Q, k), dtype=torch.float32, device=index.device)
    pg.precog_retrieve_topk(index, queries, k, idx, score)
    assert pg.precog_device_status()[0] == 0
    return idx.cpu().numpy(), score.cpu().numpy()


@pytest.mark.parametrize("dtype_name", ["float16", "bfloat16", "float32"])
@pytest.mark.parametrize("M,Q,k,dim", [(1, 1, 3, 64), (5, 2, 8, 64), (1000, 3, 3, 96),
                                       (4099, 9, 8, 64), (20000, 200, 5, 136), (300, 300, 2, 64),
                                       (39161, 257, 3, 96), (77824, 129, 8, 64)])
def test_topk_exact_integer_scores(cuda_device, dtype_name, M, Q, k, dim):
    """Small-integer keys: exact scores, many ties. Rows and scores must equal the
    oracle's stable ranking bit for bit, on the CUDA-core path (fp32 keys) and the
    tensor-core path (fp16/bf16 keys, any batch)."""
    import torch
    dtype = getattr(torch, dtype_name)
    if dtype == torch.float32 and Q > 50:
        pytest.skip("fp32 keys use the CUDA-core path one query per pass; covered at small Q")
    rng = np.random.default_rng(M + 13 * Q + k)
    index = rng.integers(-3, 4, size=(M, dim)).astype(np.float32)
    queries = rng.integers(-3, 4, size=(Q, dim)).astype(np.float32)
    idx, score = _topk(torch.from_numpy(index).to(cuda_device, dtype),
                       torch.from_numpy(queries).to(cuda_device, dtype), k)
    ref_i, ref_s = oracle.retrieve_topk(index, queries, k)
    np.testing.assert_array_equal(idx, ref_i)
    np.testing.assert_array_equal(score.astype(np.float64), ref_s)


def test_topk_k1_equals_top1_and_planted(cuda_device):
    """k = 1 agrees with precog_retrieve; on the 1M-key query workload every planted key
    is first in its query's top-3."""
    import torch
    pg = _pg()
    index = synth.device_unit_index(200_000, synth.QUERY_DIM, 3, cuda_device)
    for Q in (1, 64):
        queries, rows = synth.device_planted_queries(index, Q, synth.QUERY_NOISE, 40 + Q)
        i1 = torch.empty(Q, dtype=torch.int64, device=cuda_device)
        s1 = torch.empty(Q, dtype=torch.float32, device=cuda_device)
        pg.precog_retrieve(index, queries, i1, s1)
        ik, sk = _topk(index, queries, 1)
        np.testing.assert_array_equal(ik[:, 0], i1.cpu().numpy())
        np.testing.assert_array_equal(sk[:, 0], s1.cpu().numpy())
        i3, s3 = _topk(index, queries, 3)
        np.testing.assert_array_equal(i3[:, 0], rows.cpu().numpy())
        assert np.all(np.diff(s3, axis=1) <= 0)


@pytest.mark.parametrize("k,temperature", [(3, 1.0), (8, 0.05), (2, 10.0)])
def test_prefill_composed(cuda_device, k, temperature):
    """h_init = sum_j softmax(s/tau)_j bank[row_j] then prefill, vs the oracle's
    composition and rollout (fp32 bank and state); rows of -1 carry no weight."""
    import torch
    pg = _pg()
    d = cuda_device
    D, N, Tq, Q, entries = 64, 16, 40, 5, 50
    x, dt, A, B, C = synth.host_scan_inputs(Q * Tq, D, N, seed=k)
    rng = np.random.default_rng(k)
    bank = rng.standard_normal((entries, 2, D, N)).astype(np.float32)
    rows = rng.integers(0, entries, size=(Q, k)).astype(np.int64)
    rows[1, -1] = -1                                 # a missing entry
    scores = rng.uniform(0.2, 0.9, size=(Q, k)).astype(np.float32)
    t = lambda a, dtp=torch.float32: torch.from_numpy(np.ascontiguousarray(a)).to(d, dtp)
    y = torch.empty((1, Q * Tq, D), dtype=torch.float32, device=d)
    h = torch.empty((Q, 2, D, N), dtype=torch.float32, device=d)
    pg.precog_prefill_composed(pg.scan_inputs(t(x), t(dt), t(B), t(A), t(C), a_kind=pg.PRECOG_A_POWER),
                               Q, Tq, t(bank), t(rows, torch.int64), t(scores), k,
                               temperature=temperature, layer0=1, y_out=y, state_out=h)
    assert pg.precog_device_status()[0] == 0
    for q in range(Q):
        valid = rows[q] >= 0
        sc = np.where(valid, scores[q].astype(np.float64), np.nan)
        h0 = oracle.compose(bank[np.where(valid, rows[q], 0), 1], sc, temperature)
        sl = slice(q * Tq, (q + 1) * Tq)
        ref_h, ref_y = oracle.rollout(x[sl], dt[sl], A, B[sl], C[sl], h0=h0, want_y=True)
        assert rel_err(to_np(h[q, 1]), ref_h) < TOL_F32
        assert rel_err(to_np(y[0, sl]), ref_y) < TOL_F32


def test_retrieve_topk_then_compose_query_workload(cuda_device):
    """The paper's default k = 3 end to end at the query workload's per-query size:
    top-3 over 200K fp16 keys, composition of 24-layer bf16 states, 64-token prefill."""
    import torch
    pg = _pg()
    d = cuda_device
    L, D, N, Tq, Q, k = 24, 256, 16, synth.QUERY_TOKENS, 8, 3
    entries = 200_000
    index = synth.device_unit_index(entries, synth.QUERY_DIM, 5, d)
    queries, _ = synth.device_planted_queries(index, Q, synth.QUERY_NOISE, 77)
    idx = torch.empty((Q, k), dtype=torch.int64, device=d)
    sc = torch.empty((Q, k), dtype=torch.float32, device=d)
    pg.precog_retrieve_topk(index, queries, k, idx, sc)
    bank = synth.device_normal_bank(entries, L * D * N, 9, d).view(entries, L, D, N)
    ins = [synth.device_scan_inputs(Q * Tq, D, N, 3, l, d) for l in range(L)]
    st = lambda key: torch.stack([i[key] for i in ins]).contiguous()
    x, dt, B, C, A = st("x"), st("dt"), st("B"), st("C"), st("A")
    y = torch.empty((L, Q * Tq, D), dtype=torch.bfloat16, device=d)
    h = torch.empty((Q, L, D, N), dtype=torch.bfloat16, device=d)
    pg.precog_prefill_composed(pg.scan_inputs(x, dt, B, A, C, a_kind=pg.PRECOG_A_POWER), Q, Tq, bank,
                               idx, sc, k, y_out=y, state_out=h)
    assert pg.precog_device_status()[0] == 0
    picks = [0, Q - 1]
    ref_i, ref_s = oracle.retrieve_topk(index.cpu().numpy(), queries.float().cpu().numpy()[picks], k)
    np.testing.assert_array_equal(idx[picks].cpu().numpy(), ref_i)
    An = A[0].cpu().numpy()
    for qi, q in enumerate(picks):
        rows_q = torch.from_numpy(ref_i[qi]).to(d)
        for l in (0, 23):
            h0 = oracle.compose(to_np(bank[rows_q, l]), ref_s[qi])
            sl = slice(q * Tq, (q + 1) * Tq)
            ref_h, ref_y = oracle.rollout(to_np(x[l, sl]), to_np(dt[l, sl]), An, to_np(B[l, sl]),
                                          to_np(C[l, sl]), h0=h0, want_y=True)
            assert rel_err_stored(to_np(h[q, l]), ref_h) < TOL_BF16
            assert rel_err_stored(to_np(y[l, sl]), ref_y) < TOL_BF16


@pytest.mark.parametrize("dtype_name", ["float16", "float32"])
def test_topk_empty_index(cuda_device, dtype_name):
    """No rows: every entry of every query's list is row -1 with a NaN score."""
    import torch
    dtype = getattr(torch, dtype_name)
    idx, score = _topk(torch.empty((0, 64), dtype=dtype, device=cuda_device),
                       torch.ones((2, 64), dtype=dtype, device=cuda_device), 3)
    assert (idx == -1).all() and np.isnan(score).all()
