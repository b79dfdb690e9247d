"""GPU parity of the K-dial trajectory capture (Sec. 5.2) against the oracle."""
import numpy as np
import pytest

import oracle
import synth
from tests._util import TOL_BF16, TOL_F32, rel_err, rel_err_stored, to_np

pytestmark = pytest.mark.gpu


def _run(dev, x, dt, B, A, off, stride, dtype, power, layer0=0, L_total=1):
    import torch
    import paper_2608_02560_gb300 as pg
    eo = oracle.trajectory_offsets(off, stride)
    traj = torch.full((int(eo[-1]), L_total, A.shape[-2], A.shape[-1]), 9.0, dtype=dtype, device=dev)
    pg.precog_encode_trajectory(
        pg.scan_inputs(x, dt, B, A, a_kind=pg.PRECOG_A_POWER if power else pg.PRECOG_A_GENERAL),
        torch.from_numpy(off).to(dev), x.shape[-2], stride, torch.from_numpy(eo).to(dev), traj,
        layer0=layer0, L_total=L_total)
    st, bits = pg.precog_device_status()
    assert st == 0, bits
    return traj


@pytest.mark.parametrize("stride", [1, 5, 16, 17, 64, 1000])
@pytest.mark.parametrize("power", [False, True])
def test_trajectory_fp32(cuda_device, stride, power):
    """Ragged chunks (incl. empty and single-token), fp32: every kept state vs the oracle."""
    import torch
    D, N = 64, 16
    lens = [100, 0, 1, 37, 64, 250]
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    x, dt, A, B, _ = synth.host_scan_inputs(int(off[-1]), D, N, seed=stride)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(cuda_device)
    traj = _run(cuda_device, t(x), t(dt), t(B), t(A), off, stride, torch.float32, power,
                layer0=1, L_total=2)
    ref, eo = oracle.trajectory(x, dt, A, B, off, stride)
    got = to_np(traj)
    assert np.all(got[:, 0] == 9.0)                  # other layers untouched
    for e in range(ref.shape[0]):
        assert rel_err(got[e, 1], ref[e]) < TOL_F32, e


def test_trajectory_paper_shaped_bf16(cuda_device):
    """Paper-shaped rows (D=256, N=16, bf16 in, bf16 states), 64 chunks x 3000 tokens,
    stride 512 (the paper's 512-token granularity): sampled entries vs the oracle."""
    import torch
    shape = synth.PAPER
    n, clen, stride = 64, shape.chunk_len, 512
    off = synth.fixed_offsets(n, clen)
    inp = synth.device_scan_inputs(n * clen, shape.D, shape.N, 4, 2, cuda_device, with_C=False)
    traj = _run(cuda_device, inp["x"], inp["dt"], inp["B"], inp["A"], off, stride, torch.bfloat16, True)
    eo = oracle.trajectory_offsets(off, stride)
    A = inp["A"].cpu().numpy()
    for c in (0, 63):
        s = int(off[c])
        ref, reo = oracle.trajectory(to_np(inp["x"][s:s + clen]), to_np(inp["dt"][s:s + clen]), A,
                                     to_np(inp["B"][s:s + clen]), np.array([0, clen]), stride)
        for j in range(int(eo[c + 1] - eo[c])):
            assert rel_err_stored(to_np(traj[eo[c] + j, 0]), ref[j]) < TOL_BF16
