"""Failure detection without a GPU fault: a device-side wait that runs out of iterations
turns into a status the host reads, and the context stays usable afterwards."""
import numpy as np
import pytest

import oracle
import synth
from tests._util import TOL_F32, rel_err, to_np

pytestmark = pytest.mark.gpu


def test_bounded_wait_reports_timeout_and_context_survives(cuda_device):
    import torch
    import paper_2608_02560_gb300 as pg
    assert pg.precog_device_status()[0] == 0
    pg.precog_selftest_wait_timeout(4096)
    st, bits = pg.precog_device_status()
    assert st == 4 and bits & pg.PRECOG_DEV_TIMEOUT          # PRECOG_ERR_TIMEOUT
    assert pg.precog_device_status() == (0, 0)               # read and cleared
    # the same context still computes: a small encode against the oracle
    T, D, N = 200, 64, 16
    x, dt, A, B, _ = synth.host_scan_inputs(T, D, N, seed=3)
    off = np.array([0, 120, 200], dtype=np.int64)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(cuda_device)
    states = torch.empty((2, 1, D, N), dtype=torch.float32, device=cuda_device)
    pg.precog_encode_chunks(pg.scan_inputs(t(x), t(dt), t(B), t(A)), t(off), T, states_out=states)
    assert pg.precog_device_status()[0] == 0
    ref, _ = oracle.scan(x, dt, A, B, off)
    for c in range(2):
        assert rel_err(to_np(states[c, 0]), ref[c]) < TOL_F32
