"""GPU parity of the scan kernel (encode with state capture, readout y) against the oracle.

Called through the C ABI. Small cases are compared element by element; the full-size
workloads (single-layer wide encode, paper-shaped encode, ragged large-scale encode) run
in the launch configuration the benchmark times, and sampled chunks are compared with
the oracle one by one on inputs copied back from the device generator.
"""
import os

import numpy as np
import pytest

import oracle
import synth
from tests._util import TOL_BF16, TOL_F32, rel_err, rel_err_stored, to_np

pytestmark = pytest.mark.gpu


def _pg():
    import paper_2608_02560_gb300 as pg
    return pg


def _t(a, dev, dtype=None):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev, dtype or torch.float32)


def _encode(dev, x, dt, B, A, offsets, C=None, state_dtype=None, y_dtype=None, power=False):
    import torch
    pg = _pg()
    kind = pg.PRECOG_A_POWER if power else pg.PRECOG_A_GENERAL
    n_chunks = offsets.numel() - 1
    L = 1 if x.dim() == 2 else x.shape[0]
    D, N = A.shape[-2], A.shape[-1]
    states = torch.full((n_chunks, L, D, N), float("nan"), dtype=state_dtype or torch.float32,
                        device=dev)
    y = None
    if y_dtype is not None:
        T = x.shape[-2]
        y = torch.zeros((L, T, D), dtype=y_dtype, device=dev)
    pg.precog_encode_chunks(pg.scan_inputs(x, dt, B, A, C, a_kind=kind), offsets, x.shape[-2],
                            states_out=states, y_out=y)
    st, bits = pg.precog_device_status()
    assert st == 0, f"device status {st} bits {bits:#x}"
    return states, y


@pytest.mark.parametrize("power", [False, True])
def test_tiny_workload_fp32(cuda_device, power):
    """1 layer, D=64, N=16, fp32, 8 chunks x 256 tokens: states and every y_t (direct
    update), and states alone (rescaled accumulation when A is stated structured)."""
    import torch
    w = synth.tiny_workload(0)
    d = cuda_device
    args = (d, _t(w.x, d), _t(w.dt, d), _t(w.B, d), _t(w.A, d), _t(w.offsets, d, torch.int64))
    states, y = _encode(*args, C=_t(w.C, d), y_dtype=torch.float32, power=power)
    capt, _ = _encode(*args, power=power)
    ref_s, ref_y = oracle.scan(w.x, w.dt, w.A, w.B, w.offsets, C=w.C, want_y=True)
    for c in range(ref_s.shape[0]):
        assert rel_err(to_np(states[c, 0]), ref_s[c]) < TOL_F32
        assert rel_err(to_np(capt[c, 0]), ref_s[c]) < TOL_F32
        s, e = w.offsets[c], w.offsets[c + 1]
        assert rel_err(to_np(y[0, s:e]), ref_y[s:e]) < TOL_F32


@pytest.mark.parametrize("D,lens", [(64, [1, 15, 16, 17, 0, 300]), (96, [40, 33]),
                                    (8, [5, 100]), (512, [70, 0, 2])])
def test_ragged_lengths_and_widths_generic_A(cuda_device, D, lens):
    """Unstructured A (one exponential per (d, n)), ragged tails, empty chunks, widths
    that need several channel slices or fewer than a warp of threads."""
    import torch
    d = cuda_device
    N = 16
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    T = int(off[-1])
    x, dt, _, B, C = synth.host_scan_inputs(T, D, N, seed=D + len(lens))
    A = -np.random.default_rng(D).uniform(0.05, 3.0, size=(D, N)).astype(np.float32)
    states, y = _encode(d, _t(x, d), _t(dt, d), _t(B, d), _t(A, d), _t(off, d, torch.int64),
                        C=_t(C, d), y_dtype=torch.float32)
    ref_s, ref_y = oracle.scan(x, dt, A, B, off, C=C, want_y=True)
    for c in range(len(lens)):
        if lens[c] == 0:
            assert np.all(to_np(states[c, 0]) == 0)
            continue
        assert rel_err(to_np(states[c, 0]), ref_s[c]) < TOL_F32
        assert rel_err(to_np(y[0, off[c]:off[c + 1]]), ref_y[off[c]:off[c + 1]]) < TOL_F32


def test_A_zero_cumulative_sum_bit_exact(cuda_device):
    """A = 0: alpha = 1 exactly and h is a running sum. Dyadic inputs keep every fp32
    product and sum exact, so the GPU must match the exact cumulative sum bit for bit."""
    import torch
    d = cuda_device
    rng = np.random.default_rng(3)
    T, D, N = 200, 64, 16
    x = (rng.integers(-8, 9, size=(T, D)) / 8.0).astype(np.float32)
    dt = (rng.integers(1, 5, size=(T, D)) / 4.0).astype(np.float32)
    B = (rng.integers(-4, 5, size=(T, N)) / 4.0).astype(np.float32)
    C = (rng.integers(-4, 5, size=(T, N)) / 4.0).astype(np.float32)
    A = np.zeros((D, N), dtype=np.float32)
    off = np.array([0, 77, T], dtype=np.int64)
    args = (d, _t(x, d), _t(dt, d), _t(B, d), _t(A, d), _t(off, d, torch.int64))
    for power in (False, True):
        states, y = _encode(*args, C=_t(C, d), y_dtype=torch.float32, power=power)
        capt, _ = _encode(*args, power=power)
        for c in range(2):
            s, e = off[c], off[c + 1]
            traj = np.cumsum((dt[s:e] * x[s:e]).astype(np.float64)[:, :, None] * B[s:e, None, :],
                             axis=0)
            np.testing.assert_array_equal(to_np(states[c, 0]), traj[-1])
            np.testing.assert_array_equal(to_np(capt[c, 0]), traj[-1])
            np.testing.assert_array_equal(to_np(y[0, s:e]), np.einsum("tn,tdn->td", C[s:e], traj))


def test_multi_layer_call_and_layer_offset(cuda_device):
    """Three layers in one call with independent inputs, written at layer0=2 of a
    5-layer bank entry; the other layers stay untouched."""
    import torch
    pg = _pg()
    d = cuda_device
    L, T, D, N = 3, 96, 64, 16
    lens = [30, 66]
    off = np.array([0, 30, 96], dtype=np.int64)
    ins = [synth.host_scan_inputs(T, D, N, seed=50 + l) for l in range(L)]
    x = _t(np.stack([i[0] for i in ins]), d)
    dt = _t(np.stack([i[1] for i in ins]), d)
    B = _t(np.stack([i[3] for i in ins]), d)
    A = _t(np.stack([synth.structured_A(D, N) * (1 + 0.5 * l) for l in range(L)]), d)
    bank = torch.full((2, 5, D, N), 7.0, dtype=torch.float32, device=d)
    pg.precog_encode_chunks(pg.scan_inputs(x, dt, B, A, a_kind=pg.PRECOG_A_POWER),
                            _t(off, d, torch.int64), T, states_out=bank, layer0=2, L_total=5)
    assert pg.precog_device_status()[0] == 0
    got = to_np(bank)
    assert np.all(got[:, :2] == 7.0)
    for l in range(L):
        ref, _ = oracle.scan(ins[l][0], ins[l][1], synth.structured_A(D, N) * (1 + 0.5 * l),
                             ins[l][3], off)
        for c in range(2):
            assert rel_err(got[c, 2 + l], ref[c]) < TOL_F32


def test_concurrent_calls_on_two_streams_write_disjoint_layers(cuda_device):
    """Encode calls that write disjoint layers of one bank may run at the same time on two
    streams (the benchmark's step alternates its calls that way): the bank equals the one
    written by the same calls one after the other, bit for bit, and every entry is written."""
    import torch
    pg = _pg()
    d = cuda_device
    n_chunks, clen, D, N = 304, 1000, 256, 16
    T = n_chunks * clen
    sets = [synth.device_scan_inputs(T, D, N, 70, l, d, with_C=False) for l in range(4)]
    off = torch.from_numpy(synth.fixed_offsets(n_chunks, clen)).to(d)

    def call_inputs(first):
        st = lambda k: torch.stack([sets[first + i][k] for i in range(2)]).contiguous()
        return pg.scan_inputs(st("x"), st("dt"), st("B"), st("A"), a_kind=pg.PRECOG_A_POWER)

    calls = [call_inputs(0), call_inputs(2)]
    seq = torch.full((n_chunks, 4, D, N), float("nan"), dtype=torch.bfloat16, device=d)
    for c in range(2):
        pg.precog_encode_chunks(calls[c], off, T, states_out=seq, layer0=2 * c, L_total=4)
    torch.cuda.synchronize()
    conc = torch.full_like(seq, float("nan"))
    streams = [torch.cuda.Stream(device=d), torch.cuda.Stream(device=d)]
    start = torch.cuda.Event()
    start.record()
    for c in range(2):
        streams[c].wait_event(start)
        pg.precog_encode_chunks(calls[c], off, T, states_out=conc, layer0=2 * c, L_total=4,
                                stream=streams[c])
    for s_ in streams:
        torch.cuda.current_stream(d).wait_stream(s_)
    torch.cuda.synchronize()
    assert pg.precog_device_status()[0] == 0
    assert bool(torch.isfinite(seq.float()).all())
    assert torch.equal(conc, seq)


@pytest.mark.parametrize("D,y_mode,dtype_name", [(512, False, "float32"), (1024, False, "float32"),
                                                 (768, False, "float32"), (4096, False, "float32"),
                                                 (1024, True, "float32"), (768, True, "float32"),
                                                 (1024, False, "bfloat16"), (2048, True, "bfloat16"),
                                                 (768, False, "bfloat16")])
def test_multi_layer_sliced_channels(cuda_device, D, y_mode, dtype_name):
    """Rows wider than one CTA's channel slice (512 channels with the power-form A, 256
    where 512 does not divide D: 2, 3, 4 and 8 slices here), three layers in one call: each
    CTA stages its slice of TILE rows of x and dt with one tensor-map copy per tensor (a box
    that reaches past the last row arrives zero-filled); D = 512 stays one slice. Chunks
    (one of them empty) end inside and at the end of 16-row tiles. fp32 and bf16 inputs
    (the bf16 values widened exactly for the oracle). Every layer's states (and y) vs the
    oracle."""
    import torch
    pg = _pg()
    d = cuda_device
    dtype = getattr(torch, dtype_name)
    L, N = 3, 16
    off = np.array([0, 1, 17, 17, 53, 200], dtype=np.int64)
    T = int(off[-1])
    ins = [synth.host_scan_inputs(T, D, N, seed=90 + l) for l in range(L)]
    if dtype == torch.bfloat16:
        # the values the kernel sees: rounded to bf16 once, exactly representable in fp64
        ins = [tuple(a if i == 2 else torch.from_numpy(np.ascontiguousarray(a)).to(torch.bfloat16).double().numpy()
                     for i, a in enumerate(t)) for t in ins]
    st = lambda k: _t(np.stack([i[k] for i in ins]), d, dtype)
    x, dt, B, C = st(0), st(1), st(3), st(4)
    A = _t(np.stack([synth.structured_A(D, N) * (1 + 0.25 * l) for l in range(L)]), d)
    n = len(off) - 1
    bank = torch.full((n, L, D, N), float("nan"), dtype=torch.float32, device=d)
    y = torch.full((L, T, D), float("nan"), dtype=torch.float32, device=d) if y_mode else None
    pg.precog_encode_chunks(pg.scan_inputs(x, dt, B, A, C if y_mode else None, a_kind=pg.PRECOG_A_POWER),
                            _t(off, d, torch.int64), T, states_out=bank, y_out=y)
    assert pg.precog_device_status()[0] == 0
    got = to_np(bank)
    for l in range(L):
        ref, ref_y = oracle.scan(ins[l][0], ins[l][1], synth.structured_A(D, N) * (1 + 0.25 * l),
                                 ins[l][3], off, C=ins[l][4] if y_mode else None, want_y=y_mode)
        tol = TOL_F32 if dtype == torch.float32 else TOL_BF16
        for c in range(n):
            if off[c] == off[c + 1]:
                assert np.all(got[c, l] == 0)
            else:
                assert rel_err(got[c, l], ref[c]) < tol
        if y_mode:
            assert rel_err(to_np(y[l]), ref_y) < tol


def test_bf16_capture_and_readout(cuda_device):
    """bf16 inputs, fp32 accumulation: bf16 and fp32 state capture, bf16 readout."""
    import torch
    d = cuda_device
    T, D, N = 700, 256, 16
    off = np.array([0, 300, 301, 700], dtype=np.int64)
    x, dt, A, B, C = synth.host_scan_inputs(T, D, N, seed=77)
    tb = lambda a: _t(a, d, torch.bfloat16)
    xb, dtb, Bb, Cb = tb(x), tb(dt), tb(B), tb(C)
    s16, y16 = _encode(d, xb, dtb, Bb, _t(A, d), _t(off, d, torch.int64), C=Cb,
                       state_dtype=torch.bfloat16, y_dtype=torch.bfloat16, power=True)
    s32, _ = _encode(d, xb, dtb, Bb, _t(A, d), _t(off, d, torch.int64), power=True)
    ref_s, ref_y = oracle.scan(to_np(xb), to_np(dtb), A, to_np(Bb), off, C=to_np(Cb), want_y=True)
    for c in range(3):
        assert rel_err(to_np(s32[c, 0]), ref_s[c]) < 1e-5
        assert rel_err_stored(to_np(s16[c, 0]), ref_s[c]) < TOL_BF16
        sl = slice(off[c], off[c + 1])
        assert rel_err_stored(to_np(y16[0, sl]), ref_y[sl]) < TOL_BF16


def test_bad_offsets_flag_device_status(cuda_device):
    """Non-monotone or out-of-range offsets are skipped and reported, never faulted."""
    import torch
    pg = _pg()
    d = cuda_device
    T, D, N = 64, 64, 16
    x, dt, A, B, _ = synth.host_scan_inputs(T, D, N, seed=1)
    off = _t(np.array([0, 40, 20, 64, 1000], dtype=np.int64), d, torch.int64)
    states = torch.zeros((4, 1, D, N), dtype=torch.float32, device=d)
    pg.precog_encode_chunks(pg.scan_inputs(_t(x, d), _t(dt, d), _t(B, d), _t(A, d)), off, T,
                            states_out=states)
    st, bits = pg.precog_device_status()
    assert st == 5 and bits & pg.PRECOG_DEV_BAD_OFFSETS
    assert pg.precog_device_status() == (0, 0)   # the word was cleared
    ref, _ = oracle.scan(x, dt, A, B, np.array([0, 40], dtype=np.int64))
    assert rel_err(to_np(states[0, 0]), ref[0]) < TOL_F32


def test_deterministic(cuda_device):
    import torch
    d = cuda_device
    x, dt, A, B, _ = synth.host_scan_inputs(512, 256, 16, seed=9)
    off = _t(np.array([0, 256, 512], dtype=np.int64), d, torch.int64)
    args = [_t(v, d, torch.bfloat16) for v in (x, dt, B)]
    for power in (False, True):
        a, _ = _encode(d, args[0], args[1], args[2], _t(A, d), off, power=power)
        b, _ = _encode(d, args[0], args[1], args[2], _t(A, d), off, power=power)
        assert torch.equal(a, b)


def test_power_statement_is_verified(cuda_device):
    """a_kind = PRECOG_A_POWER with an A that is not (n+1)*A[d,0]: nothing is written for
    the affected channel blocks and PRECOG_DEV_BAD_A is flagged; A[d,0] > 0 as well. A
    1024-channel layer is encoded in two blocks of 512 channels."""
    import torch
    pg = _pg()
    d = cuda_device
    T, D, N = 50, 1024, 16
    x, dt, A, B, _ = synth.host_scan_inputs(T, D, N, seed=2)
    A_bad = A.copy()
    A_bad[600, 5] *= 1.5                    # channel 600 sits in the second 512-channel block
    off = _t(np.array([0, T], dtype=np.int64), d, torch.int64)
    for Ab in (A_bad, -A):
        states = torch.full((1, 1, D, N), 3.0, dtype=torch.float32, device=d)
        pg.precog_encode_chunks(pg.scan_inputs(_t(x, d), _t(dt, d), _t(B, d), _t(Ab, d),
                                               a_kind=pg.PRECOG_A_POWER), off, T, states_out=states)
        st, bits = pg.precog_device_status()
        assert st == 5 and bits == pg.PRECOG_DEV_BAD_A
        assert torch.all(states[0, 0, 512:] == 3.0)
    ref, _ = oracle.rollout(x, dt, A, B)
    states = torch.full((1, 1, D, N), 3.0, dtype=torch.float32, device=d)
    pg.precog_encode_chunks(pg.scan_inputs(_t(x, d), _t(dt, d), _t(B, d), _t(A_bad, d),
                                           a_kind=pg.PRECOG_A_POWER), off, T, states_out=states)
    pg.precog_device_status()
    assert rel_err(to_np(states[0, 0, :512]), ref[:512]) < TOL_F32   # the valid block is done


@pytest.mark.parametrize("scale,dt_shift", [(1.0, -2.0), (40.0, -2.0), (1.0, 2.5), (0.02, -4.0)])
def test_rescaled_renormalisation_regimes(cuda_device, scale, dt_shift):
    """The rescaled accumulation against the oracle where renormalisation is frequent
    (large |A| or large dt: single tokens that decay past the window go through the
    direct update), rare (tiny |A|, long memory) or mixed, fp32 inputs, 1e-5."""
    import torch
    d = cuda_device
    T, D, N = 1500, 64, 16
    rng = np.random.default_rng(int(scale * 100) + 7)
    x = rng.standard_normal((T, D)).astype(np.float32)
    dt = np.logaddexp(0.0, rng.standard_normal((T, D)) + dt_shift).astype(np.float32)
    B = (rng.standard_normal((T, N)) * 0.25).astype(np.float32)
    A = (synth.structured_A(D, N) * scale).astype(np.float32)
    off = np.array([0, 700, 701, T], dtype=np.int64)
    capt, _ = _encode(d, _t(x, d), _t(dt, d), _t(B, d), _t(A, d), _t(off, d, torch.int64),
                      power=True)
    ref, _ = oracle.scan(x, dt, A, B, off)
    for c in range(3):
        assert rel_err(to_np(capt[c, 0]), ref[c]) < TOL_F32, c


# ------------------------------------------------------------- full-size workloads, sampled


def _sample(n_chunks, fixed, count=32, seed=0, last=64):
    """The listed chunks, ``count`` seeded random ones, and four of the last ``last``
    chunks (the launch's last wave)."""
    rng = np.random.default_rng(1000 + seed)
    pick = set(int(c) for c in fixed) | set(int(c) for c in rng.choice(n_chunks, count, replace=False))
    pick |= set(int(c) for c in rng.choice(np.arange(n_chunks - last, n_chunks), 4, replace=False))
    return sorted(pick)


def _oracle_states(x, dt, B, A, off_np, chunks):
    """Oracle final states of the listed chunks of one layer (inputs copied back from the
    device exactly), the chunks split over host threads."""
    import torch
    rows = np.concatenate([np.arange(off_np[c], off_np[c + 1]) for c in chunks])
    it = torch.from_numpy(rows).to(x.device)
    lens = np.array([off_np[c + 1] - off_np[c] for c in chunks], dtype=np.int64)
    sub_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    return oracle.scan_threads(to_np(x[it]), to_np(dt[it]), A, to_np(B[it]), sub_off, os.cpu_count() or 1)


def _sampled_check(dev, shape, layer, sample_chunks, y_mode=False, seed=0, state_dtype=None):
    """Generate one layer of a workload on the device at full size, run the encode as the
    benchmark does into a bank filled with NaN, check that exactly the layer's entries were
    written (all finite) and compare the sampled chunks with the oracle. A bf16 bank is
    held to the tolerance before its one rounding (half a bf16 ulp allowed), an fp32 one to
    the plain tolerance."""
    import torch
    pg = _pg()
    sdt = torch.bfloat16 if state_dtype is None else state_dtype
    off_np = synth.shape_offsets(shape, seed)
    T = int(off_np[-1])
    inp = synth.device_scan_inputs(T, shape.D, shape.N, seed, layer, dev, with_C=y_mode)
    off = torch.from_numpy(off_np).to(dev)
    L_bank, slot = shape.n_layers, layer
    states = torch.full((shape.n_chunks, L_bank, shape.D, shape.N), float("nan"), dtype=sdt, device=dev)
    y = torch.empty((1, T, shape.D), dtype=torch.bfloat16, device=dev) if y_mode else None
    pg.precog_encode_chunks(pg.scan_inputs(inp["x"], inp["dt"], inp["B"], inp["A"],
                                           inp.get("C") if y_mode else None,
                                           a_kind=pg.PRECOG_A_POWER),
                            off, T, states_out=states, layer0=slot, L_total=L_bank,
                            y_out=y)
    assert pg.precog_device_status()[0] == 0
    assert bool(torch.isfinite(states[:, slot]).all()), "an entry of the written layer was not written"
    assert bool(torch.isnan(states[:, :slot]).all()) and bool(torch.isnan(states[:, slot + 1:]).all()), \
        "another layer was written"
    A = inp["A"].cpu().numpy()
    ref = _oracle_states(inp["x"], inp["dt"], inp["B"], A, off_np, sample_chunks)
    check = rel_err_stored if sdt == torch.bfloat16 else rel_err
    worst = 0.0
    for i, c in enumerate(sample_chunks):
        err = check(to_np(states[c, slot]), ref[i])
        worst = max(worst, err)
        assert err < TOL_BF16, (c, err)
    if y_mode:
        for c in sample_chunks[:3]:
            s, e = int(off_np[c]), int(off_np[c + 1])
            _, ref_y = oracle.rollout(to_np(inp["x"][s:e]), to_np(inp["dt"][s:e]), A, to_np(inp["B"][s:e]),
                                      to_np(inp["C"][s:e]), want_y=True)
            assert rel_err_stored(to_np(y[0, s:e]), ref_y) < TOL_BF16, c
    del inp, states, y
    torch.cuda.empty_cache()
    return worst


def test_paper_shaped_multi_layer_call_sampled(cuda_device):
    """The launch the benchmark times: one call encodes 4 paper-shaped layers (4096 chunks x
    3000 tokens each, contiguous inputs of 4 independent draws) into layers 8..11 of the
    24-layer bf16 bank filled with NaN: every entry of those layers written and finite, the
    other layers untouched, and per layer 36 seeded chunks (last wave included) vs the
    oracle."""
    import torch
    pg = _pg()
    d = cuda_device
    shape, S, layer0 = synth.PAPER, 4, 8
    off_np = synth.shape_offsets(shape, 0)
    T = int(off_np[-1])
    x = torch.empty((S, T, shape.D), dtype=torch.bfloat16, device=d)
    dt = torch.empty_like(x)
    B = torch.empty((S, T, shape.N), dtype=torch.bfloat16, device=d)
    sets = [synth.device_scan_inputs(T, shape.D, shape.N, 0, l, d, with_C=False,
                                     out={"x": x[l], "dt": dt[l], "B": B[l]}) for l in range(S)]
    A = torch.stack([st["A"] for st in sets]).contiguous()
    states = torch.full((shape.n_chunks, shape.n_layers, shape.D, shape.N), float("nan"),
                        dtype=torch.bfloat16, device=d)
    pg.precog_encode_chunks(pg.scan_inputs(x, dt, B, A, a_kind=pg.PRECOG_A_POWER),
                            torch.from_numpy(off_np).to(d), T, states_out=states, layer0=layer0,
                            L_total=shape.n_layers)
    assert pg.precog_device_status()[0] == 0
    assert bool(torch.isnan(states[:, :layer0]).all()) and bool(torch.isnan(states[:, layer0 + S:]).all())
    assert bool(torch.isfinite(states[:, layer0:layer0 + S]).all())
    An = sets[0]["A"].cpu().numpy()
    for l in range(S):
        pick = _sample(shape.n_chunks, (0, 2047, shape.n_chunks - 1), seed=l)
        ref = _oracle_states(x[l], dt[l], B[l], An, off_np, pick)
        for i, c in enumerate(pick):
            assert rel_err_stored(to_np(states[c, layer0 + l]), ref[i]) < TOL_BF16, (l, c)


def test_wide_single_layer_full_size(cuda_device):
    """1 layer, D=2048, N=16, 1024 chunks x 512 tokens, bf16: fp32 state capture (plain
    tolerance) and the readout mode into a bf16 bank."""
    _sampled_check(cuda_device, synth.WIDE, 0, _sample(1024, [0, 511, 1023]), state_dtype=_f32())
    _sampled_check(cuda_device, synth.WIDE, 0, _sample(1024, [3, 1000], count=8, seed=1), y_mode=True)


def _f32():
    import torch
    return torch.float32


def test_paper_shaped_encode_full_size(cuda_device):
    """24 x (D=256, N=16) layers, 4096 chunks x 3000 tokens, bf16: layers 0 and 23 at
    full size into the 192 KB-per-chunk bf16 bank layout, and layer 5 captured in fp32
    (plain tolerance, no rounding allowance)."""
    _sampled_check(cuda_device, synth.PAPER, 0, _sample(4096, [0, 2047, 4095]))
    _sampled_check(cuda_device, synth.PAPER, 23, _sample(4096, [1, 4094], seed=23))
    _sampled_check(cuda_device, synth.PAPER, 5, _sample(4096, [7], seed=5), state_dtype=_f32())


def test_ragged_large_scale_encode_full_size(cuda_device):
    """8192 ragged chunks (lengths 256..4096), D=512, N=16, bf16: the longest, the
    shortest, the first and last and 36 seeded chunks of one layer."""
    off = synth.shape_offsets(synth.RAGGED, 0)
    lens = np.diff(off)
    fixed = [int(np.argmax(lens)), int(np.argmin(lens)), 0, 4097, 8191]
    _sampled_check(cuda_device, synth.RAGGED, 5, _sample(8192, fixed, seed=5))


@pytest.mark.parametrize("case", ["capture_bf16", "readout_f32", "few_chunks_readout", "complex"])
def test_ordered_encode_matches_unordered(cuda_device, case):
    """precog_encode_chunks_ordered: any processing order (random, longest first) gives
    bit for bit the states (and y) of the plain call; an order entry outside the chunks
    is skipped with PRECOG_DEV_BAD_INDEX and leaves that work item's chunk unwritten."""
    import math
    import torch
    pg = _pg()
    d = cuda_device
    rng = np.random.default_rng(77)
    few = case == "few_chunks_readout"
    n = 5 if few else (200 if case == "readout_f32" else 40)
    lens = rng.integers(0, 300, size=n)
    lens[3] = 0
    off_np = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    T = int(off_np[-1])
    D, N = (256, 16) if case != "readout_f32" else (64, 16)
    dtype = torch.bfloat16 if case in ("capture_bf16", "complex") else torch.float32
    inp = synth.device_scan_inputs(T, D, N, 5, 0, d, dtype=dtype)
    y_mode = case in ("readout_f32", "few_chunks_readout")
    if case == "complex":
        A = torch.complex(inp["A"], (math.pi * torch.arange(N, device=d, dtype=torch.float32)).expand(D, N))
        si = pg.scan_inputs(inp["x"], inp["dt"], inp["B"], A.contiguous(), a_kind=pg.PRECOG_A_COMPLEX)
        shape = (n, 1, D, N, 2)
    else:
        si = pg.scan_inputs(inp["x"], inp["dt"], inp["B"], inp["A"], inp["C"] if y_mode else None,
                            a_kind=pg.PRECOG_A_POWER)
        shape = (n, 1, D, N)
    off = torch.from_numpy(off_np).to(d)

    def run(order):
        st = torch.full(shape, 7.0, dtype=torch.float32, device=d)
        y = torch.full((1, T, D), 7.0, dtype=torch.float32, device=d) if y_mode else None
        if order is None:
            pg.precog_encode_chunks(si, off, T, states_out=st, y_out=y)
        else:
            pg.precog_encode_chunks_ordered(si, off, T, torch.from_numpy(order).to(d), states_out=st, y_out=y)
        return st, y

    ref_st, ref_y = run(None)
    assert pg.precog_device_status()[0] == 0
    for order in (rng.permutation(n).astype(np.int64), np.argsort(-lens, kind="stable").astype(np.int64)):
        st, y = run(order)
        assert pg.precog_device_status()[0] == 0
        assert torch.equal(st, ref_st)
        if y_mode:
            assert torch.equal(y, ref_y)
    bad = np.arange(n, dtype=np.int64)
    bad[1] = n + 5                                   # chunk 1 is never taken up
    st, _ = run(bad)
    status, bits = pg.precog_device_status()
    assert bits & pg.PRECOG_DEV_BAD_INDEX
    assert bool((st[1] == 7.0).all())
    keep = [c for c in range(n) if c != 1]
    assert torch.equal(st[keep], ref_st[keep])
