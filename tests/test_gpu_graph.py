"""The public calls are CUDA-graph capturable: encode, retrieve (with a caller workspace)
and prefill from the retrieved state, captured once and replayed on refilled inputs, give
results bit-identical to the same calls made eagerly (no host synchronisation, allocation or
host-side branching on device values inside any of them)."""
import numpy as np
import pytest

import synth

pytestmark = pytest.mark.gpu


def test_capture_encode_retrieve_prefill_and_replay(cuda_device):
    import torch
    import paper_2608_02560_gb300 as pg
    d = cuda_device
    L, D, N, n, T_c, Tq, M, dim = 2, 256, 16, 16, 200, 32, 4096, 128
    off = torch.arange(0, n * T_c + 1, T_c, dtype=torch.int64, device=d)
    index = synth.device_unit_index(M, dim, 3, d, dtype=torch.float16)

    def fill(seed, buf):
        ins = [synth.device_scan_inputs(n * T_c, D, N, seed, l, d) for l in range(L)]
        qin = [synth.device_scan_inputs(Tq, D, N, seed + 100, l, d) for l in range(L)]
        for k in ("x", "dt", "B"):
            buf[k].copy_(torch.stack([i[k] for i in ins]))
        for k in ("x", "dt", "B", "C"):
            buf["q" + k].copy_(torch.stack([i[k] for i in qin]))
        q, _ = synth.device_planted_queries(index, 1, synth.QUERY_NOISE, seed)
        buf["q"].copy_(q)

    bf = torch.bfloat16
    buf = {"x": torch.empty((L, n * T_c, D), dtype=bf, device=d),
           "dt": torch.empty((L, n * T_c, D), dtype=bf, device=d),
           "B": torch.empty((L, n * T_c, N), dtype=bf, device=d),
           "qx": torch.empty((L, Tq, D), dtype=bf, device=d),
           "qdt": torch.empty((L, Tq, D), dtype=bf, device=d),
           "qB": torch.empty((L, Tq, N), dtype=bf, device=d),
           "qC": torch.empty((L, Tq, N), dtype=bf, device=d),
           "q": torch.empty((1, dim), dtype=torch.float16, device=d)}
    A = torch.from_numpy(np.stack([synth.structured_A(D, N)] * L)).to(d)
    ws = torch.empty(pg.precog_retrieve_workspace_size(M, dim, 1) + 16, dtype=torch.uint8, device=d)
    ins = pg.scan_inputs(buf["x"], buf["dt"], buf["B"], A, a_kind=pg.PRECOG_A_POWER)
    qins = pg.scan_inputs(buf["qx"], buf["qdt"], buf["qB"], A, buf["qC"], a_kind=pg.PRECOG_A_POWER)

    def path(out):
        pg.precog_encode_chunks(ins, off, n * T_c, states_out=out["bank"])
        pg.precog_retrieve(index[:n], buf["q"], out["idx"], out["score"], workspace=ws)
        pg.precog_prefill_from_state(qins, 1, Tq, out["bank"], idx=out["idx"], y_out=out["y"],
                                     state_out=out["h"])

    def outputs():
        return {"bank": torch.empty((n, L, D, N), dtype=bf, device=d),
                "idx": torch.empty(1, dtype=torch.int64, device=d),
                "score": torch.empty(1, dtype=torch.float32, device=d),
                "y": torch.empty((L, Tq, D), dtype=bf, device=d),
                "h": torch.empty((1, L, D, N), dtype=torch.float32, device=d)}

    g_out = outputs()
    fill(1, buf)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        path(g_out)                       # warm-up outside the capture
    torch.cuda.current_stream().wait_stream(side)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        path(g_out)
    for seed in (2, 3):
        fill(seed, buf)
        graph.replay()
        e_out = outputs()
        path(e_out)
        torch.cuda.synchronize()
        assert pg.precog_device_status()[0] == 0
        for k in g_out:
            assert torch.equal(g_out[k], e_out[k]), (seed, k)
