"""GPU parity of the SMC primitives (Sec. 5): two-level routing, semantic-state EMA and
O(1) session initialisation by injecting a consolidated state."""
import numpy as np
import pytest

import oracle
import synth
from tests._util import TOL_F32, rel_err, to_np

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dtype_name", ["float32", "float16", "bfloat16"])
def test_route_exact_integer_scores(cuda_device, dtype_name):
    """Small-integer embeddings and prototypes (exact scores, frequent ties): domain and
    sub-cluster must equal the oracle's; J[m] limits the sub-clusters searched."""
    import torch
    import paper_2608_02560_gb300 as pg
    dtype = getattr(torch, dtype_name)
    rng = np.random.default_rng(7)
    n, dim, M, J_max = 3000, 384, 5, 4
    emb = rng.integers(-2, 3, size=(n, dim)).astype(np.float32)
    P = rng.integers(-2, 3, size=(M, dim)).astype(np.float32)
    S = rng.integers(-2, 3, size=(M, J_max, dim)).astype(np.float32)
    J = np.array([4, 1, 3, 0, 2], dtype=np.int32)
    t = lambda a, dt=dtype: torch.from_numpy(np.ascontiguousarray(a)).to(cuda_device, dt)
    dm = torch.empty(n, dtype=torch.int32, device=cuda_device)
    dj = torch.empty(n, dtype=torch.int32, device=cuda_device)
    slot = torch.empty(n, dtype=torch.int64, device=cuda_device)
    pg.precog_smc_route(t(emb), t(P), t(S), t(J, torch.int32), dm, dj, slot)
    assert pg.precog_device_status()[0] == 0
    rm, rj = oracle.smc_route(emb, P, S, J)
    np.testing.assert_array_equal(dm.cpu().numpy(), rm)
    np.testing.assert_array_equal(dj.cpu().numpy(), rj)
    exp_slot = np.where(rj >= 0, rm * J_max + rj, -1)
    np.testing.assert_array_equal(slot.cpu().numpy(), exp_slot)


@pytest.mark.parametrize("dtype_name,dim", [("float16", 100), ("float32", 61), ("bfloat16", 96)])
def test_route_nan_prototypes_and_unaligned_rows(cuda_device, dtype_name, dim):
    """Rows that are not whole 16-byte vectors (element loads) and rows that are, more
    prototypes than one pass of eight at both levels, and NaN prototypes (a NaN score never
    wins; an embedding whose domain scores are all NaN routes nowhere)."""
    import torch
    import paper_2608_02560_gb300 as pg
    dtype = getattr(torch, dtype_name)
    rng = np.random.default_rng(dim)
    n, M, J_max = 700, 11, 13
    emb = rng.integers(-2, 3, size=(n, dim)).astype(np.float32)
    P = rng.integers(-2, 3, size=(M, dim)).astype(np.float32)
    S = rng.integers(-2, 3, size=(M, J_max, dim)).astype(np.float32)
    P[4, 7] = np.nan                      # domain 4 never wins
    S[:, 9, 3] = np.nan                   # sub-cluster 9 of every domain never wins
    emb[5, :] = np.nan                    # all scores NaN: routes nowhere
    J = rng.integers(0, J_max + 1, size=M).astype(np.int32)
    J[0] = J_max
    t = lambda a, dt=dtype: torch.from_numpy(np.ascontiguousarray(a)).to(cuda_device, dt)
    dm = torch.empty(n, dtype=torch.int32, device=cuda_device)
    dj = torch.empty(n, dtype=torch.int32, device=cuda_device)
    slot = torch.empty(n, dtype=torch.int64, device=cuda_device)
    pg.precog_smc_route(t(emb), t(P), t(S), t(J, torch.int32), dm, dj, slot)
    assert pg.precog_device_status()[0] == 0
    rm, rj = oracle.smc_route(emb, P, S, J)
    assert rm[5] == -1 and 4 not in set(rm.tolist()) and 9 not in set(rj.tolist())
    np.testing.assert_array_equal(dm.cpu().numpy(), rm)
    np.testing.assert_array_equal(dj.cpu().numpy(), rj)
    np.testing.assert_array_equal(slot.cpu().numpy(), np.where(rj >= 0, rm * J_max + rj, -1))


def test_consolidate_then_session_init(cuda_device):
    """Deposit 300 chunk states (bf16, 24 layers of D=256, N=16) into 20 semantic slots
    in order (some forgetting candidates, slot -1), compare the fp32 table with the
    oracle's EMA, then initialise sessions from two slots and prefill 64 tokens."""
    import torch
    import paper_2608_02560_gb300 as pg
    d = cuda_device
    L, D, N, n, slots, alpha = 24, 256, 16, 300, 20, 0.2
    rng = np.random.default_rng(3)
    states = synth.device_normal_bank(n, L * D * N, 4, d)            # [n, elems] bf16
    slot_np = rng.integers(-1, slots, size=n).astype(np.int64)
    sem0 = rng.standard_normal((slots, L * D * N)).astype(np.float32) * 0.1
    sem = torch.from_numpy(sem0).to(d)
    pg.precog_smc_consolidate(sem, states, torch.from_numpy(slot_np).to(d), alpha)
    assert pg.precog_device_status()[0] == 0
    ref = oracle.smc_consolidate(sem0, to_np(states), slot_np, alpha)
    got = to_np(sem)
    for s in range(slots):
        assert rel_err(got[s], ref[s]) < TOL_F32, s
    # O(1) session initialisation: inject s_{m*, j*} and prefill (Sec. 5.3)
    Tq, Q = 64, 2
    ins = [synth.device_scan_inputs(Q * Tq, D, N, 5, l, d) for l in range(L)]
    st = lambda k: torch.stack([i[k] for i in ins]).contiguous()
    x, dt, B, C, A = st("x"), st("dt"), st("B"), st("C"), st("A")
    idx = torch.tensor([3, 17], dtype=torch.int64, device=d)
    h = torch.empty((Q, L, D, N), dtype=torch.float32, device=d)
    pg.precog_prefill_from_state(pg.scan_inputs(x, dt, B, A, C, a_kind=pg.PRECOG_A_POWER), Q, Tq,
                                 sem.view(slots, L, D, N), idx=idx, state_out=h)
    assert pg.precog_device_status()[0] == 0
    An = A[0].cpu().numpy()
    for q, srow in enumerate((3, 17)):
        for l in (0, 23):
            sl = slice(q * Tq, (q + 1) * Tq)
            ref_h, _ = oracle.rollout(to_np(x[l, sl]), to_np(dt[l, sl]), An, to_np(B[l, sl]),
                                      h0=ref[srow].reshape(L, D, N)[l])
            assert rel_err(to_np(h[q, l]), ref_h) < TOL_F32


@pytest.mark.parametrize("n,n_slots,pattern", [(200, 64, "cyclic"), (77, 3, "runs"), (1, 5, "cyclic"),
                                               (96, 40, "random"), (2500, 7, "random"),
                                               (500, 300, "random"), (700, 1000, "runs")])
def test_consolidate_deposit_patterns(cuda_device, n, n_slots, pattern):
    """Deposit orders that exercise both folds (per-slot CTAs for tables of at most 256
    slots, deposit batches beyond): no slot repeated within a batch (cyclic), long runs of
    one slot, a single deposit, random slots with -1 mixed in, more deposits than one
    gathering pass; fp32 states of an odd element count."""
    import torch
    import paper_2608_02560_gb300 as pg
    rng = np.random.default_rng(n + n_slots)
    elems = 333
    states = rng.standard_normal((n, elems)).astype(np.float32)
    if pattern == "cyclic":
        slot_np = np.arange(n, dtype=np.int64) % n_slots
    elif pattern == "runs":
        slot_np = (np.arange(n, dtype=np.int64) // 10) % n_slots
    else:
        slot_np = rng.integers(-1, n_slots, size=n).astype(np.int64)
    sem0 = rng.standard_normal((n_slots, elems)).astype(np.float32)
    sem = torch.from_numpy(sem0).to(cuda_device)
    pg.precog_smc_consolidate(sem, torch.from_numpy(states).to(cuda_device),
                              torch.from_numpy(slot_np).to(cuda_device), 0.3)
    assert pg.precog_device_status()[0] == 0
    ref = oracle.smc_consolidate(sem0, states, slot_np, 0.3)
    got = to_np(sem)
    for s in range(n_slots):
        assert rel_err(got[s], ref[s]) < TOL_F32, s


@pytest.mark.parametrize("elems,n_slots", [(64, 3), (63, 3), (64, 300)])
def test_consolidate_flags_slot_outside_table(cuda_device, elems, n_slots):
    """A slot >= n_slots or below -1 deposits nothing and raises PRECOG_DEV_BAD_INDEX;
    the other deposits still apply (the staged per-slot fold, the register per-slot fold
    for a row of odd length, the batch fold for a table of more than 256 slots)."""
    import torch
    import paper_2608_02560_gb300 as pg
    rng = np.random.default_rng(5)
    states = rng.standard_normal((7, elems)).astype(np.float32)
    slot_np = np.array([0, 1, n_slots + 6, 1, 0, -2, 2], dtype=np.int64)
    sem0 = np.zeros((n_slots, elems), dtype=np.float32)
    sem = torch.from_numpy(sem0).to(cuda_device)
    pg.precog_smc_consolidate(sem, torch.from_numpy(states).to(cuda_device),
                              torch.from_numpy(slot_np).to(cuda_device), 0.5)
    st, bits = pg.precog_device_status()
    assert st != 0 and bits & pg.PRECOG_DEV_BAD_INDEX
    keep = slot_np.copy()
    keep[2] = keep[5] = -1
    ref = oracle.smc_consolidate(sem0, states, keep, 0.5)
    assert rel_err(to_np(sem), ref) < TOL_F32


@pytest.mark.parametrize("dtype,elems,n,n_slots,pattern", [
    ("f32", 4132, 200, 64, "cyclic"), ("bf16", 4200, 77, 3, "runs"), ("bf16", 8, 1, 5, "cyclic"),
    ("f32", 4, 96, 40, "random"), ("bf16", 4200, 2500, 7, "random"), ("bf16", 12296, 600, 256, "random"),
    ("f32", 2048, 300, 1, "runs"), ("f32", 6148, 1030, 100, "random")])
def test_consolidate_staged_patterns(cuda_device, dtype, elems, n, n_slots, pattern):
    """The fold that streams states through the shared-memory ring (rows of whole
    16-byte chunks, at most 256 slots): element ranges of 2048 (fp32) or 4096 (bf16)
    with a ragged last range, several tiles per CTA (256 slots x 4 ranges), more slot
    ids than one prefetch window (512), one slot, a single deposit, -1 mixed in."""
    import torch
    import paper_2608_02560_gb300 as pg
    rng = np.random.default_rng(elems + n + n_slots)
    states = rng.standard_normal((n, elems)).astype(np.float32)
    if dtype == "bf16":
        states_dev = torch.from_numpy(states).to(cuda_device).to(torch.bfloat16)
        states = states_dev.float().cpu().numpy()
    else:
        states_dev = torch.from_numpy(states).to(cuda_device)
    if pattern == "cyclic":
        slot_np = np.arange(n, dtype=np.int64) % n_slots
    elif pattern == "runs":
        slot_np = (np.arange(n, dtype=np.int64) // 10) % n_slots
    else:
        slot_np = rng.integers(-1, n_slots, size=n).astype(np.int64)
    sem0 = rng.standard_normal((n_slots, elems)).astype(np.float32)
    sem = torch.from_numpy(sem0).to(cuda_device)
    pg.precog_smc_consolidate(sem, states_dev, torch.from_numpy(slot_np).to(cuda_device), 0.3)
    assert pg.precog_device_status()[0] == 0
    ref = oracle.smc_consolidate(sem0, states, slot_np, 0.3)
    got = to_np(sem)
    for s in range(n_slots):
        assert rel_err(got[s], ref[s]) < TOL_F32, s


def test_smc_benchmark_sizes_sampled(cuda_device):
    """The launches the benchmark times: 4096 chunk embeddings (fp16, dim 768) routed over
    16 domains x 64 sub-clusters, and 4096 bf16 24-layer states folded into 64 slots.
    Routing is compared where the oracle's best score leads the runner-up by more than
    fp32 error can move (both levels); consolidation on sampled state elements."""
    import torch
    import paper_2608_02560_gb300 as pg
    d = cuda_device
    n, Md, J, dim = 4096, 16, 64, synth.QUERY_DIM
    index = synth.device_unit_index(n + Md + Md * J, dim, 21, d)
    emb, dom = index[:n], index[n:n + Md].contiguous()
    sub = index[n + Md:].contiguous().view(Md, J, dim)
    Jt = torch.full((Md,), J, dtype=torch.int32, device=d)
    om = torch.empty(n, dtype=torch.int32, device=d)
    oj = torch.empty(n, dtype=torch.int32, device=d)
    osl = torch.empty(n, dtype=torch.int64, device=d)
    pg.precog_smc_route(emb, dom, sub, Jt, om, oj, osl)
    assert pg.precog_device_status()[0] == 0
    E, P, S = (to_np(t) for t in (emb, dom, sub))
    rm, rj = oracle.smc_route(E, P, S, Jt.cpu().numpy())
    sd = E @ P.T
    top2 = np.sort(sd, axis=1)[:, -2:]
    ok_m = (top2[:, 1] - top2[:, 0]) > 1e-4
    ss = np.einsum("nd,njd->nj", E, S[rm])
    top2j = np.sort(ss, axis=1)[:, -2:]
    ok_j = ok_m & ((top2j[:, 1] - top2j[:, 0]) > 1e-4)
    assert ok_j.sum() > n // 2
    np.testing.assert_array_equal(om.cpu().numpy()[ok_m], rm[ok_m])
    np.testing.assert_array_equal(oj.cpu().numpy()[ok_j], rj[ok_j])
    # consolidation of 4096 24-layer states into 64 slots, in deposit order
    L, D, N = 24, 256, 16
    states = synth.device_normal_bank(n, L * D * N, 22, d)
    slots = torch.arange(n, dtype=torch.int64, device=d) * 7 % 64
    sem0 = torch.zeros((64, L * D * N), dtype=torch.float32, device=d)
    sem = sem0.clone()
    pg.precog_smc_consolidate(sem, states, slots, 0.1)
    assert pg.precog_device_status()[0] == 0
    cols = torch.from_numpy(np.random.default_rng(3).choice(L * D * N, size=257, replace=False)).to(d)
    ref = oracle.smc_consolidate(to_np(sem0[:, cols]), to_np(states[:, cols]), slots.cpu().numpy(), 0.1)
    got = to_np(sem[:, cols])
    for s in range(64):
        assert rel_err(got[s], ref[s]) < TOL_F32, s
