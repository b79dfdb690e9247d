"""precog_retrieve_noalloc: retrieval for callers that cannot allocate device memory
when they retrieve (for example a serving loop that must never call cudaMalloc).

Called through the C ABI and compared with precog_retrieve (which uses a caller
workspace) on the same inputs, twice in a row: over an fp16 index for a single query and
for a batch (both on the tensor-core kernel), and over an fp32 index for a batch near the
scratch limit (the CUDA-core kernel, whose partitions take the most scratch). The file
sorts last so that a failure here never hides another test, and it passes both alone in a
fresh process and after the others."""
import ctypes

import numpy as np
import pytest

import synth

pytestmark = pytest.mark.gpu


def _noalloc(lib):
    f = lib.precog_retrieve_noalloc
    f.restype = ctypes.c_int32
    f.argtypes = [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p,
                  ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]
    return f


@pytest.mark.parametrize("dtype_name,Q", [("float16", 1), ("float16", 256), ("float32", 400)])
def test_noalloc_matches_workspace_retrieval_twice(cuda_device, dtype_name, Q):
    import torch
    import paper_2608_02560_gb300 as pg
    lib = pg.load_library()
    noalloc = _noalloc(lib)
    dtype = getattr(torch, dtype_name)
    M, dim = 262_144, synth.QUERY_DIM
    index = synth.device_unit_index(M, dim, 7, cuda_device, dtype=dtype)
    queries, rows = synth.device_planted_queries(index, Q, synth.QUERY_NOISE, 11 + Q)
    ref_idx = torch.empty(Q, dtype=torch.int64, device=cuda_device)
    ref_score = torch.empty(Q, dtype=torch.float32, device=cuda_device)
    pg.precog_retrieve(index, queries, ref_idx, ref_score)
    code = pg.PRECOG_F16 if dtype == torch.float16 else pg.PRECOG_F32
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    for call in range(2):
        idx = torch.full((Q,), -5, dtype=torch.int64, device=cuda_device)
        score = torch.full((Q,), float("nan"), dtype=torch.float32, device=cuda_device)
        st = noalloc(index.data_ptr(), code, M, dim, queries.data_ptr(), Q,
                     idx.data_ptr(), score.data_ptr(), stream)
        assert st == 0, lib.precog_last_error().decode()
        assert pg.precog_device_status()[0] == 0
        assert torch.equal(idx, ref_idx), f"call {call}"
        np.testing.assert_allclose(score.cpu().numpy(), ref_score.cpu().numpy(), rtol=0, atol=1e-6)
        assert torch.equal(idx, rows)


def test_noalloc_rejects_batches_beyond_its_scratch(cuda_device):
    import torch
    import paper_2608_02560_gb300 as pg
    lib = pg.load_library()
    noalloc = _noalloc(lib)
    M, dim, Q = 1_000_000, 64, 4096
    # buffers of the stated sizes: even if the size check ever ran after a launch, no
    # access could leave them
    index = torch.zeros((M, dim), dtype=torch.float16, device=cuda_device)
    queries = torch.zeros((Q, dim), dtype=torch.float16, device=cuda_device)
    out = torch.full((Q,), -5, dtype=torch.int64, device=cuda_device)
    st = noalloc(index.data_ptr(), pg.PRECOG_F16, M, dim, queries.data_ptr(), Q, out.data_ptr(),
                 None, ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == 2                                          # PRECOG_ERR_UNSUPPORTED
    assert b"scratch" in lib.precog_last_error()
    torch.cuda.synchronize()
    assert bool((out == -5).all())                          # nothing was launched
