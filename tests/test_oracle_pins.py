"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: the
PRECOG-RAG equivalence (Theorem 1), the sufficient-statistic proposition
(Appendix A), the closed-form unroll (Appendix B.1, Eq. unroll), geometric and
cumulative-sum special cases, hand-expanded tiny rollouts with exact dyadic
values, numpy's argmax as the textbook top-1, and the state sizes printed in
Appendix C.1. The inputs are chosen so that a dropped term, a flipped sign, a
transposed (d, n) index or a readout taken before the update fails at least
one of them.
"""
import json
import math
import os

import numpy as np
import pytest

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rand_inputs(T, D, N, seed):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((T, D))
    dt = np.logaddexp(0.0, rng.standard_normal((T, D)) - 1.0)
    A = -rng.uniform(0.1, 2.0, size=(D, N))          # generic, unstructured
    B = rng.standard_normal((T, N))
    C = rng.standard_normal((T, N))
    return x, dt, A, B, C


# ---------------------------------------------------------------- Theorem 1 and the Proposition


@pytest.mark.parametrize("Lc,Tq", [(0, 5), (1, 1), (37, 11), (200, 64)])
def test_theorem1_precog_equals_in_context(Lc, Tq):
    """Theorem 1: S(h0, c (+) q) == S(S(h0, c), q), and every readout y_t of the query
    positions agrees (Proposition, Appendix A). Sequential fp64 => bit-identical."""
    D, N = 5, 3
    x, dt, A, B, C = _rand_inputs(Lc + Tq, D, N, seed=Lc * 31 + Tq)
    h0 = np.random.default_rng(7).standard_normal((D, N))
    h_full, y_full = oracle.rollout(x, dt, A, B, C, h0=h0, want_y=True)
    h_ctx, _ = oracle.rollout(x[:Lc], dt[:Lc], A, B[:Lc], C[:Lc], h0=h0, want_y=True)
    h_inj, y_inj = oracle.rollout(x[Lc:], dt[Lc:], A, B[Lc:], C[Lc:], h0=h_ctx, want_y=True)
    np.testing.assert_array_equal(h_full, h_inj)
    np.testing.assert_array_equal(y_full[Lc:], y_inj)


def test_proposition_outputs_depend_on_context_only_through_state():
    """Two different contexts that reach the same state give identical query outputs.

    A 'reset' token with dt*A = -1000 makes alpha = exp(-1000) == 0 exactly in double and,
    with x = 0, beta = 0; whatever preceded it, the state after it is exactly zero."""
    D, N = 3, 2
    xa, dta, A, Ba, Ca = _rand_inputs(9, D, N, seed=1)
    xb, dtb, _, Bb, Cb = _rand_inputs(4, D, N, seed=2)
    xq, dtq, _, Bq, Cq = _rand_inputs(6, D, N, seed=3)
    A = -np.ones((D, N))
    reset_x, reset_dt = np.zeros((1, D)), np.full((1, D), 1000.0)
    reset_B, reset_C = np.ones((1, N)), np.ones((1, N))
    ca = [np.vstack(v) for v in ((xa, reset_x), (dta, reset_dt), (Ba, reset_B), (Ca, reset_C))]
    cb = [np.vstack(v) for v in ((xb, reset_x), (dtb, reset_dt), (Bb, reset_B), (Cb, reset_C))]
    ha, _ = oracle.rollout(ca[0], ca[1], A, ca[2], ca[3], want_y=True)
    hb, _ = oracle.rollout(cb[0], cb[1], A, cb[2], cb[3], want_y=True)
    np.testing.assert_array_equal(ha, np.zeros((D, N)))
    np.testing.assert_array_equal(hb, np.zeros((D, N)))
    _, ya = oracle.rollout(xq, dtq, A, Bq, Cq, h0=ha, want_y=True)
    _, yb = oracle.rollout(xq, dtq, A, Bq, Cq, h0=hb, want_y=True)
    np.testing.assert_array_equal(ya, yb)


# ---------------------------------------------------------------- closed forms and special cases


def test_constant_gates_geometric_series():
    """dt = delta, x = xi, B = b constant: h_T = a^T h0 + delta*xi*b*(1 - a^T)/(1 - a),
    a = exp(delta*A) (Eq. unroll with a constant gate is a geometric series)."""
    D, N, T = 2, 3, 50
    delta = np.array([0.3, 0.05])
    xi = np.array([1.5, -0.7])
    b = np.array([0.2, -1.0, 0.6])
    A = np.array([[-1.0, -2.0, -0.5], [-0.25, -3.0, -1.5]])
    h0 = np.array([[1.0, -2.0, 0.5], [0.0, 3.0, -1.0]])
    x = np.tile(xi, (T, 1))
    dt = np.tile(delta, (T, 1))
    B = np.tile(b, (T, 1))
    h, _ = oracle.rollout(x, dt, A, B, h0=h0)
    a = np.exp(delta[:, None] * A)
    expect = a ** T * h0 + (delta * xi)[:, None] * b[None, :] * (1 - a ** T) / (1 - a)
    np.testing.assert_allclose(h, expect, rtol=1e-12, atol=1e-14)
    assert np.all(np.abs(h) < 1e3)  # decays to a finite fixed point (|a| < 1)


def test_A_zero_is_cumulative_sum_exact():
    """A = 0 => alpha = 1, h_T = h0 + sum_t dt_t x_t B_t, y_t = C_t . h_t with the
    updated state. Dyadic inputs make every product and sum exact in double."""
    rng = np.random.default_rng(5)
    T, D, N = 40, 4, 6
    x = rng.integers(-16, 17, size=(T, D)) / 16.0
    dt = rng.integers(1, 9, size=(T, D)) / 8.0
    B = rng.integers(-8, 9, size=(T, N)) / 8.0
    C = rng.integers(-8, 9, size=(T, N)) / 4.0
    h0 = rng.integers(-4, 5, size=(D, N)) / 2.0
    A = np.zeros((D, N))
    h, y = oracle.rollout(x, dt, A, B, C, h0=h0, want_y=True)
    traj = h0[None] + np.cumsum((dt * x)[:, :, None] * B[:, None, :], axis=0)  # [T, D, N]
    np.testing.assert_array_equal(h, traj[-1])
    np.testing.assert_array_equal(y, np.einsum("tn,tdn->td", C, traj))


def test_dyadic_gates_hand_expanded():
    """alpha chosen exactly through A = log(p)/dt: alpha[d, n] = p[d, n] (distinct per
    (d, n), D != N) and beta = dt*x*B. Two steps expanded by hand:
    h2 = p*(p*h0 + b1) + b2. Catches a flipped exponent sign, a transposed A or B index,
    and a beta missing dt."""
    D, N = 2, 3
    p = np.array([[0.5, 0.25, 0.75], [0.125, 0.875, 0.375]])
    dt = np.array([[2.0, 0.5], [2.0, 0.5]])            # per token, per channel
    A = np.log(p) / dt[0][:, None]
    x = np.array([[1.0, -2.0], [0.5, 4.0]])
    B = np.array([[1.0, 2.0, -1.0], [0.25, -0.5, 3.0]])
    C = np.array([[1.0, 0.0, 0.0], [0.0, 1.0, -1.0]])
    h0 = np.array([[8.0, -4.0, 2.0], [1.0, 0.0, -16.0]])
    h, y = oracle.rollout(x, dt, A, B, C, h0=h0, want_y=True)
    b1 = (dt[0] * x[0])[:, None] * B[0][None, :]
    b2 = (dt[1] * x[1])[:, None] * B[1][None, :]
    h1 = p * h0 + b1
    h2 = p * h1 + b2
    np.testing.assert_allclose(h, h2, rtol=1e-14, atol=1e-14)
    np.testing.assert_allclose(y[0], h1 @ C[0], rtol=1e-14, atol=1e-14)
    np.testing.assert_allclose(y[1], h2 @ C[1], rtol=1e-14, atol=1e-14)


def test_readout_uses_updated_state():
    """One token from the zero state: y_1 = sum_n C_n * B_n * x * dt (nonzero), which a
    readout taken before the update would report as 0 (Eq. 1: y_t = C(h_t))."""
    x = np.array([[2.0]])
    dt = np.array([[0.5]])
    A = np.array([[-1.0, -2.0]])
    B = np.array([[3.0, -1.0]])
    C = np.array([[0.5, 2.0]])
    h, y = oracle.rollout(x, dt, A, B, C, want_y=True)
    np.testing.assert_array_equal(h, np.array([[3.0, -1.0]]))
    assert y[0, 0] == 0.5 * 3.0 + 2.0 * -1.0


@pytest.mark.parametrize("L", [1, 2, 5, 8])
def test_unroll_closed_form_and_linearity(L):
    """Eq. unroll (Appendix B.1): S(0, c) = sum_t beta(c_t) prod_{s>t} alpha(c_s), and
    S(h0, c) = S(0, c) + (prod_t alpha(c_t)) * h0, evaluated by brute force.

    A = log(p) with dyadic p (distinct per (d, n)) and integer dt make every gate an
    exact power alpha_t[d, n] = p[d, n] ** dt_t[d]; x and B are dyadic too."""
    D, N = 2, 3
    rng = np.random.default_rng(100 + L)
    p = np.array([[0.5, 0.25, 0.75], [0.625, 0.375, 0.875]])
    A = np.log(p)
    dt = rng.integers(1, 4, size=(L, D)).astype(float)
    x = rng.integers(-8, 9, size=(L, D)) / 4.0
    B = rng.integers(-8, 9, size=(L, N)) / 8.0
    h0 = rng.integers(-8, 9, size=(D, N)) / 2.0
    alpha = p[None] ** dt[:, :, None]                     # [L, D, N]
    beta = (dt * x)[:, :, None] * B[:, None, :]
    zero_state = np.zeros((D, N))
    for t in range(L):
        prod = np.ones((D, N))
        for s in range(t + 1, L):
            prod = prod * alpha[s]
        zero_state = zero_state + beta[t] * prod
    total_decay = np.prod(alpha, axis=0)
    h_zero, _ = oracle.rollout(x, dt, A, B)
    h_init, _ = oracle.rollout(x, dt, A, B, h0=h0)
    np.testing.assert_allclose(h_zero, zero_state, rtol=1e-13, atol=1e-13)
    np.testing.assert_allclose(h_init, zero_state + total_decay * h0, rtol=1e-13, atol=1e-13)


def test_channel_isolation_and_state_index():
    """A[0, :] = 0 (channel 0 integrates: cumulative sum) while A[1, :] = -1000 (channel 1
    forgets instantly: its state is the last token's beta). A transposed A or a B
    indexed by channel instead of state index mixes the two."""
    rng = np.random.default_rng(9)
    T, D, N = 7, 2, 4
    x = rng.integers(-4, 5, size=(T, D)) / 4.0
    dt = np.full((T, D), 0.5)
    B = rng.integers(-4, 5, size=(T, N)) / 4.0
    A = np.vstack([np.zeros(N), np.full(N, -2000.0)])
    h, _ = oracle.rollout(x, dt, A, B)
    np.testing.assert_array_equal(h[0], np.sum((dt[:, 0] * x[:, 0])[:, None] * B, axis=0))
    np.testing.assert_array_equal(h[1], dt[-1, 1] * x[-1, 1] * B[-1])


def test_chunk_boundaries_and_empty_chunks():
    """Chunks are independent scans from the zero state (Sec. 4.2); a zero-length chunk
    captures h0 (here zero); rows between chunks are never mixed."""
    D, N = 3, 2
    lens = [5, 0, 1, 7, 0]
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    x, dt, A, B, C = _rand_inputs(int(off[-1]), D, N, seed=11)
    states, y = oracle.scan(x, dt, A, B, off, C=C, want_y=True)
    for c in range(len(lens)):
        s, e = off[c], off[c + 1]
        h, yc = oracle.rollout(x[s:e], dt[s:e], A, B[s:e], C[s:e], want_y=True)
        np.testing.assert_array_equal(states[c], h)
        np.testing.assert_array_equal(y[s:e], yc)
    np.testing.assert_array_equal(states[1], 0)
    np.testing.assert_array_equal(states[4], 0)
    h0 = np.random.default_rng(3).standard_normal((len(lens), D, N))
    states_h0, _ = oracle.scan(x, dt, A, B, off, h0=h0)
    np.testing.assert_array_equal(states_h0[1], h0[1])


def test_stability_bound():
    """|alpha| < 1 (Appendix B.1): |h_T| <= |h0| * prod alpha + max|beta| / (1 - max alpha)."""
    x, dt, A, B, _ = _rand_inputs(3000, 4, 5, seed=21)
    h, _ = oracle.rollout(x, dt, A, B)
    alpha = np.exp(dt[:, :, None] * A[None])
    beta = (dt * x)[:, :, None] * B[:, None, :]
    amax = alpha.max()
    assert amax < 1
    assert np.all(np.abs(h) <= np.abs(beta).max() / (1 - amax) + 1e-12)


def test_memory_horizon_contribution_decay():
    """Appendix B.1: a perturbation of token t changes h_T by beta-difference times
    prod_{s>t} alpha_s -- the token's contribution decays with its distance to the end."""
    D, N, T = 2, 2, 60
    x, dt, A, B, _ = _rand_inputs(T, D, N, seed=4)
    h, _ = oracle.rollout(x, dt, A, B)
    t = 10
    x2 = x.copy()
    x2[t] += 1.0
    h2, _ = oracle.rollout(x2, dt, A, B)
    alpha = np.exp(dt[:, :, None] * A[None])
    prod = np.prod(alpha[t + 1:], axis=0)
    dbeta = (dt[t] * 1.0)[:, None] * B[t][None, :]
    np.testing.assert_allclose(h2 - h, dbeta * prod, rtol=1e-9, atol=1e-15)


# ---------------------------------------------------------------- retrieval


def test_retrieve_matches_numpy_argmax_first_occurrence():
    rng = np.random.default_rng(13)
    M, dim, Q = 300, 17, 9
    index = rng.integers(-3, 4, size=(M, dim)).astype(float)   # many exact ties
    queries = rng.integers(-2, 3, size=(Q, dim)).astype(float)
    idx, score = oracle.retrieve(index, queries)
    S = queries @ index.T                                        # exact small integers
    np.testing.assert_array_equal(idx, np.argmax(S, axis=1))    # argmax = first occurrence
    np.testing.assert_array_equal(score, S.max(axis=1))


def test_retrieve_ties_nan_and_empty():
    index = np.array([[1.0, 0.0], [np.nan, 0.0], [1.0, 0.0], [0.5, 0.5]])
    idx, score = oracle.retrieve(index, np.array([[1.0, 0.0], [0.0, 1.0], [np.nan, 1.0]]))
    assert idx[0] == 0 and score[0] == 1.0                     # duplicate rows 0 and 2 -> 0
    assert idx[1] == 3 and score[1] == 0.5                     # NaN row 1 never wins
    assert idx[2] == -1 and math.isnan(score[2])                # every score NaN -> -1
    idx, score = oracle.retrieve(np.zeros((0, 2)), np.ones((1, 2)))
    assert idx[0] == -1 and math.isnan(score[0])


def test_retrieve_planted_tiny_workload():
    """The tiny workload's query is key 3 plus small noise: top-1 must be 3."""
    w = synth.tiny_workload(0)
    idx, score = oracle.retrieve(w.index, w.query)
    assert idx[0] == w.planted
    assert 0.8 < score[0] <= 1.0 + 1e-6


# ---------------------------------------------------------------- sizes printed by the paper


def test_paper_state_size():
    g = json.load(open(os.path.join(GOLDEN, "paper_sizes.json")))
    assert g["repeat"] * g["num_coeffs"] == g["state_per_layer"]
    total = g["layers"] * g["state_per_layer"] * g["bytes_per_value_fp16"]
    assert total == g["total_state_bytes"] == g["total_state_kib"] * 1024
    # 10K chunks x 196,608 B = 1.97e9 B, printed as "1.9 GB"
    assert abs(g["corpus_chunks_example"] * total / 1e9 - g["corpus_state_gb_example"]) < 0.1
    # the paper-shaped workload stores the same 192 KB: 24 layers x D=256 x N=16 x 2 B
    s = synth.PAPER
    assert s.n_layers * s.D * s.N * 2 == g["total_state_bytes"]


def test_bf16_storage_tolerance_helper():
    """The comparison used for bf16-stored outputs allows exactly the one rounding:
    torch's round-to-nearest-even bf16 cast of the exact value scores 0."""
    import torch
    from tests._util import rel_err_stored
    ref = np.random.default_rng(0).standard_normal(10000) * 3.0
    stored = torch.from_numpy(ref).to(torch.bfloat16).double().numpy()
    assert rel_err_stored(stored, ref) == 0.0
    bumped = stored.copy()
    bumped[np.argmax(np.abs(ref))] *= 1 + 2.0 ** -6         # two ulps off at the maximum
    assert rel_err_stored(bumped, ref) > 2e-3


# ---------------------------------------------------------------- top-k and composition


def test_topk_matches_numpy_stable_argsort():
    """Top-k = the first k of a stable sort by descending exact score (lower row first
    among equals), checked with numpy's stable argsort on exact small-integer scores."""
    rng = np.random.default_rng(3)
    M, dim, Q, k = 200, 9, 6, 5
    index = rng.integers(-2, 3, size=(M, dim)).astype(float)
    queries = rng.integers(-2, 3, size=(Q, dim)).astype(float)
    rows, vals = oracle.retrieve_topk(index, queries, k)
    S = queries @ index.T
    for q in range(Q):
        order = np.argsort(-S[q], kind="stable")[:k]
        np.testing.assert_array_equal(rows[q], order)
        np.testing.assert_array_equal(vals[q], S[q, order])
    r1, s1 = oracle.retrieve(index, queries)
    np.testing.assert_array_equal(rows[:, 0], r1)          # k = 1 is top-1 retrieval


def test_topk_nan_and_short_index():
    index = np.array([[1.0, 0.0], [np.nan, 1.0], [0.5, 0.0]])
    rows, vals = oracle.retrieve_topk(index, np.array([[1.0, 1.0]]), 4)
    assert list(rows[0]) == [0, 2, -1, -1]
    assert vals[0, 0] == 1.0 and vals[0, 1] == 0.5 and np.isnan(vals[0, 2:]).all()


def test_compose_softmax_weights():
    """Weights are the textbook softmax (scipy) of score / temperature; equal scores give
    the plain average; one entry gives that entry; missing entries get no weight."""
    scipy_special = pytest.importorskip("scipy.special")
    rng = np.random.default_rng(8)
    rows = rng.standard_normal((3, 4, 5))
    sc = np.array([0.9, 0.2, -0.3])
    for tau in (1.0, 0.1):
        w = scipy_special.softmax(sc / tau)
        np.testing.assert_allclose(oracle.compose(rows, sc, tau),
                                   np.tensordot(w, rows, axes=1), rtol=1e-13, atol=1e-13)
    np.testing.assert_allclose(oracle.compose(rows, np.full(3, 0.4)), rows.mean(axis=0), rtol=1e-13)
    np.testing.assert_array_equal(oracle.compose(rows[:1], [0.7]), rows[0])
    np.testing.assert_allclose(oracle.compose(rows, [0.5, np.nan, 0.5]), (rows[0] + rows[2]) / 2,
                               rtol=1e-13)


def test_composition_commutes_with_the_scan():
    """The scan is affine in its initial state (Eq. unroll): with weights summing to one,
    S(sum_j w_j h_j, q) = sum_j w_j S(h_j, q) -- injecting the composed state equals
    composing the individually injected rollouts."""
    D, N, T = 3, 4, 20
    x, dt, A, B, C = _rand_inputs(T, D, N, seed=17)
    rng = np.random.default_rng(4)
    hs = rng.standard_normal((3, D, N))
    sc = np.array([0.3, 0.8, 0.1])
    h_comp, y_comp = oracle.rollout(x, dt, A, B, C, h0=oracle.compose(hs, sc), want_y=True)
    e = np.exp(sc - sc.max())
    w = e / e.sum()
    parts = [oracle.rollout(x, dt, A, B, C, h0=hs[j], want_y=True) for j in range(3)]
    np.testing.assert_allclose(h_comp, sum(w[j] * parts[j][0] for j in range(3)), rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(y_comp, sum(w[j] * parts[j][1] for j in range(3)), rtol=1e-11, atol=1e-12)


# ---------------------------------------------------------------- K-dial trajectory


@pytest.mark.parametrize("stride", [1, 3, 7, 50])
def test_trajectory_is_prefix_rollouts(stride):
    """Entry j of chunk c is S(0, c_{1:t}) with t = min((j+1) * stride, len_c): brute
    force by rolling every prefix separately; the last entry is the chunk's final state
    (K = 1 is the PRECOG state, Sec. 5.2); empty chunks keep nothing."""
    D, N = 3, 4
    lens = [10, 0, 1, 21, 7]
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    x, dt, A, B, _ = _rand_inputs(int(off[-1]), D, N, seed=stride)
    traj, eo = oracle.trajectory(x, dt, A, B, off, stride)
    finals, _ = oracle.scan(x, dt, A, B, off)
    for c, L in enumerate(lens):
        K = -(-L // stride)
        assert eo[c + 1] - eo[c] == K
        for j in range(K):
            t = min((j + 1) * stride, L)
            s = off[c]
            ref, _ = oracle.rollout(x[s:s + t], dt[s:s + t], A, B[s:s + t])
            np.testing.assert_allclose(traj[eo[c] + j], ref, rtol=1e-12, atol=1e-14)
        if K:
            np.testing.assert_array_equal(traj[eo[c + 1] - 1], finals[c])


# ---------------------------------------------------------------- SMC routing and consolidation


def test_smc_route_two_levels():
    """Hand-built prototypes: the domain is the best prototype, the sub-cluster the best
    among that domain's J[m] sub-prototypes only (not the global best sub-prototype)."""
    P = np.array([[1.0, 0.0, 0.0], [0.0, 1.0, 0.0], [0.0, 0.0, 1.0]])
    Qs = np.zeros((3, 2, 3))
    Qs[0] = [[1.0, 1.0, 0.0], [1.0, -1.0, 0.0]]
    Qs[1] = [[0.0, 1.0, 5.0], [0.0, 9.0, 9.0]]          # second entry unused (J[1] = 1), though it scores higher
    Qs[2] = [[0.0, 0.0, 1.0], [9.0, 9.0, 9.0]]
    J = [2, 1, 2]
    e = np.array([[0.9, -0.2, 0.1], [0.1, 0.8, 0.7], [0.2, 0.1, 0.95], [1.0, 1.0, 0.0]])
    m, j = oracle.smc_route(e, P, Qs, J)
    assert list(m) == [0, 1, 2, 0]                      # ties (row 3) go to the lower domain
    assert list(j) == [1, 0, 1, 0]


def test_smc_consolidate_closed_form():
    """Constant deposits h into one slot n times from s0: s_n = (1-a)^n s0 + (1-(1-a)^n) h;
    a = 1 keeps the last deposit; slot -1 deposits nothing; other slots are untouched."""
    rng = np.random.default_rng(2)
    s0 = rng.standard_normal((3, 5))
    h = rng.standard_normal(5)
    a, n = 0.3, 7
    out = oracle.smc_consolidate(s0, np.tile(h, (n + 1, 1)), [1] * n + [-1], a)
    np.testing.assert_allclose(out[1], (1 - a) ** n * s0[1] + (1 - (1 - a) ** n) * h, rtol=1e-12)
    np.testing.assert_array_equal(out[[0, 2]], s0[[0, 2]])
    hs = rng.standard_normal((4, 5))
    out = oracle.smc_consolidate(s0, hs, [2, 0, 2, 0], 1.0)
    np.testing.assert_array_equal(out[2], hs[2])
    np.testing.assert_array_equal(out[0], hs[3])


# ---------------------------------------------------------------- complex diagonal A


def test_complex_scan_real_special_case():
    """A_im = 0: the complex scan is the real scan (imaginary part stays exactly 0)."""
    D, N = 3, 4
    off = np.array([0, 9, 9, 30], dtype=np.int64)
    x, dt, A, B, C = _rand_inputs(30, D, N, seed=5)
    st, y = oracle.scan_complex(x, dt, A, np.zeros_like(A), B, off, C=C, want_y=True)
    rs, ry = oracle.scan(x, dt, A, B, off, C=C, want_y=True)
    np.testing.assert_allclose(st.real, rs, rtol=1e-13, atol=1e-14)
    np.testing.assert_array_equal(st.imag, 0.0)
    np.testing.assert_allclose(y, ry, rtol=1e-13, atol=1e-14)


def test_complex_scan_theorem1_and_geometric_series():
    """Theorem 1 holds for the complex recurrence (bit-identical sequential double), and
    constant gates give the complex geometric series h_T = a^T h0 + b (1 - a^T)/(1 - a)."""
    D, N = 2, 3
    rng = np.random.default_rng(9)
    A_re = -np.logaddexp(0.0, rng.standard_normal((D, N)))
    A_im = np.pi * np.arange(N)[None, :].repeat(D, 0)          # i*pi*k of Eq. 1
    x, dt, _, B, C = _rand_inputs(40, D, N, seed=10)
    h0 = rng.standard_normal((1, D, N)) + 1j * rng.standard_normal((1, D, N))
    full, yf = oracle.scan_complex(x, dt, A_re, A_im, B, [0, 40], C=C, h0=h0, want_y=True)
    ctx, _ = oracle.scan_complex(x[:25], dt[:25], A_re, A_im, B[:25], [0, 25], h0=h0)
    inj, yi = oracle.scan_complex(x[25:], dt[25:], A_re, A_im, B[25:], [0, 15], C=C[25:], h0=ctx,
                                  want_y=True)
    np.testing.assert_array_equal(full, inj)
    np.testing.assert_array_equal(yf[25:], yi)
    T, delta, xi = 30, 0.4, np.array([1.5, -0.5])
    b = np.array([0.3, -1.0, 0.7])
    hs, _ = oracle.scan_complex(np.tile(xi, (T, 1)), np.full((T, D), delta), A_re, A_im,
                                np.tile(b, (T, 1)), [0, T], h0=h0)
    a = np.exp(delta * (A_re + 1j * A_im))
    beta = (delta * xi)[:, None] * b[None, :]
    np.testing.assert_allclose(hs[0], a ** T * h0[0] + beta * (1 - a ** T) / (1 - a), rtol=1e-12)


def test_scan_threads_matches_scan_bit_for_bit():
    """The threaded driver only splits chunks over host threads: ragged and empty chunks
    give exactly scan's states, for any thread count."""
    x, dt, A, B, _ = synth.host_scan_inputs(1300, 32, 16, seed=5)
    off = np.array([0, 300, 300, 650, 651, 1200, 1300], dtype=np.int64)
    ref, _ = oracle.scan(x, dt, A, B, off)
    for threads in (1, 2, 4, 9):
        assert np.array_equal(oracle.scan_threads(x, dt, A, B, off, threads), ref)
