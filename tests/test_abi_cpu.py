"""The C-ABI library loads and exports every symbol include/precog.h declares, and its
host-side argument checks return the documented status codes without touching a GPU
(no pointer passed here is ever dereferenced on the host)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "precog.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2608_02560_gb300 import build
    build.build()
    import paper_2608_02560_gb300 as pg
    return pg.load_library()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(precog_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_three_calls():
    names = declared_functions()
    for n in ("precog_encode_chunks", "precog_retrieve", "precog_prefill_from_state"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 8
    for n in names:
        assert hasattr(lib, n), f"{n} declared in include/precog.h but not exported"


def test_abi_version_and_status_strings(lib):
    assert lib.precog_abi_version() == 1
    for code, name in [(0, b"PRECOG_OK"), (1, b"PRECOG_ERR_INVALID_ARG"),
                       (2, b"PRECOG_ERR_UNSUPPORTED"), (3, b"PRECOG_ERR_CUDA"),
                       (4, b"PRECOG_ERR_TIMEOUT"), (5, b"PRECOG_ERR_DEVICE")]:
        assert lib.precog_status_string(code) == name


FAKE = 0x10000  # a 16-byte aligned address that the host never dereferences


def _inputs(pg, **kw):
    s = pg.ScanInputs()
    s.n_layers, s.D, s.N, s.in_dtype = 1, 64, 16, pg.PRECOG_BF16
    s.x = s.dt = s.B = s.C = s.A = FAKE
    s.layer_stride_xd = s.layer_stride_bc = 0
    for k, v in kw.items():
        setattr(s, k, v)
    return s


def _encode(lib, s, offsets=FAKE, n_chunks=4, T_tot=64, states=FAKE, sdt=0, layer0=0, L=1,
            y=None, ydt=0):
    return lib.precog_encode_chunks(ctypes.byref(s) if s is not None else None, offsets, n_chunks,
                                    T_tot, states, sdt, layer0, L, y, ydt, None)


@pytest.mark.parametrize("change,expect", [
    ({"N": 8}, 2), ({"D": 0}, 1), ({"D": 12}, 2), ({"in_dtype": 2}, 2), ({"x": 0}, 1),
    ({"A": FAKE + 4}, 1), ({"n_layers": 0}, 1), ({"n_layers": 2, "layer_stride_xd": 10}, 1),
    ({"a_kind": 3}, 1), ({"a_kind": -1}, 1),
])
def test_encode_rejects_bad_inputs(lib, change, expect):
    import paper_2608_02560_gb300 as pg
    assert _encode(lib, _inputs(pg, **change)) == expect
    assert lib.precog_last_error() != b""


def test_complex_A_forms_without_a_kernel_are_rejected(lib):
    """Trajectories and k > 1 composition of complex states are refused as unsupported
    before any launch."""
    import paper_2608_02560_gb300 as pg
    s = _inputs(pg, a_kind=pg.PRECOG_A_COMPLEX)
    st = lib.precog_encode_trajectory(ctypes.byref(s), FAKE, 4, 64, 8, FAKE, FAKE, 0, 0, 1, None)
    assert st == 2 and b"complex" in lib.precog_last_error()
    st = lib.precog_prefill_composed(ctypes.byref(s), 2, 32, FAKE, 0, 10, 1, 0, 3, FAKE, FAKE,
                                     1.0, None, 0, FAKE, 0, None)
    assert st == 2 and b"complex" in lib.precog_last_error()


def test_encode_rejects_bad_call_arguments(lib):
    import paper_2608_02560_gb300 as pg
    s = _inputs(pg)
    assert _encode(lib, None) == 1
    assert _encode(lib, s, offsets=None) == 1
    assert _encode(lib, s, n_chunks=-1) == 1
    assert _encode(lib, s, T_tot=-5) == 1
    assert _encode(lib, s, states=None, y=None) == 1
    assert _encode(lib, s, sdt=2) == 2                      # fp16 states unsupported
    assert _encode(lib, s, layer0=1, L=1) == 1              # layer outside the bank entry
    assert _encode(lib, s, states=FAKE + 8) == 1            # misaligned output
    assert _encode(lib, _inputs(pg, C=None), y=FAKE) == 1   # readout needs C
    assert _encode(lib, s, n_chunks=0) == 0                 # nothing to do: OK, no launch


def test_ordered_encode_checks_its_arguments(lib):
    """The ordered encode needs an order array and otherwise checks what the plain one
    checks, before any launch."""
    import paper_2608_02560_gb300 as pg
    s = _inputs(pg)
    f = lib.precog_encode_chunks_ordered
    f.restype = ctypes.c_int32
    f.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p,
                  ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_void_p,
                  ctypes.c_int32, ctypes.c_void_p]
    call = lambda order=FAKE, **kw: f(ctypes.byref(s), kw.get("offsets", FAKE), kw.get("n_chunks", 3), 64, order,
                                      kw.get("states", FAKE), 0, 0, 1, None, 0, None)
    assert call(order=None) == 1
    assert call(offsets=None) == 1
    assert call(states=FAKE + 8) == 1
    assert call(n_chunks=0) == 0


def test_prefill_rejects_bad_arguments(lib):
    import paper_2608_02560_gb300 as pg
    s = _inputs(pg)
    f = lib.precog_prefill_from_state
    assert f(ctypes.byref(s), 1, 4, None, 1, 10, 24, 0, FAKE, FAKE, 0, FAKE, 0, None) == 1
    assert f(ctypes.byref(s), 1, 4, FAKE, 1, 10, 24, 24, FAKE, FAKE, 0, FAKE, 0, None) == 1
    assert f(ctypes.byref(s), 3, 4, FAKE, 1, 2, 24, 0, None, FAKE, 0, FAKE, 0, None) == 1
    assert f(ctypes.byref(s), 1, 4, FAKE, 1, 10, 24, 0, FAKE, None, 0, None, 0, None) == 1
    assert f(ctypes.byref(s), -1, 4, FAKE, 1, 10, 24, 0, FAKE, FAKE, 0, FAKE, 0, None) == 1
    assert f(ctypes.byref(s), 0, 4, FAKE, 1, 10, 24, 0, FAKE, FAKE, 0, FAKE, 0, None) == 0


def test_retrieve_rejects_bad_arguments(lib):
    f = lib.precog_retrieve
    assert f(FAKE, 2, 100, 768, FAKE, 1, FAKE, FAKE, FAKE, 0, None) == 1       # no workspace
    assert f(FAKE, 2, 100, 12, FAKE, 1, FAKE, FAKE, FAKE, 1 << 20, None) == 2   # 24 B rows
    assert f(FAKE, 7, 100, 768, FAKE, 1, FAKE, FAKE, FAKE, 1 << 20, None) == 2  # dtype
    assert f(FAKE, 2, -1, 768, FAKE, 1, FAKE, FAKE, FAKE, 1 << 20, None) == 1
    assert f(FAKE, 2, 1 << 31, 768, FAKE, 1, FAKE, FAKE, FAKE, 1 << 40, None) == 2
    assert f(FAKE, 2, 100, 768, None, 1, FAKE, FAKE, FAKE, 1 << 20, None) == 1
    assert f(FAKE, 2, 100, 768, FAKE, 0, FAKE, FAKE, FAKE, 0, None) == 0       # no queries
    assert lib.precog_retrieve_workspace_size(100, 768, 4) >= 4 * 8


def test_missing_library_fails_loudly(tmp_path):
    """No CPU fallback: loading the binding against a path with no libprecog.so raises
    instead of computing anything another way."""
    import paper_2608_02560_gb300 as pg
    saved = pg._lib
    try:
        pg._lib = None
        with pytest.raises(ImportError):
            pg.load_library(str(tmp_path / "libprecog.so"))
    finally:
        pg._lib = saved


def test_product_package_does_not_import_the_oracle():
    """The product path never reaches the test oracle: no module of the package names it."""
    pkg = os.path.join(ROOT, "paper_2608_02560_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h", ".cpp")):
                text = open(os.path.join(dirpath, f)).read()
                assert not re.search(r"^\s*(import|from)\s+oracle\b", text, flags=re.M), f
                assert "precog_oracle" not in text, f


def test_selftest_rejects_bad_iteration_counts(lib):
    lib.precog_selftest_wait_timeout.argtypes = [ctypes.c_uint32, ctypes.c_void_p]
    lib.precog_selftest_wait_timeout.restype = ctypes.c_int32
    assert lib.precog_selftest_wait_timeout(0, None) == 1
    assert lib.precog_selftest_wait_timeout((1 << 20) + 1, None) == 1


def test_shard_key_calls_reject_bad_arguments(lib):
    """Row-sharded retrieval: a negative row offset, an offset that pushes global rows past
    2^32 - 1, missing key output and negative counts are argument errors returned before
    any launch; zero queries is a no-op."""
    f = lib.precog_retrieve_keys
    ws = 1 << 20
    assert f(FAKE, 2, 100, 768, FAKE, 1, -1, FAKE, FAKE, ws, None) == 1
    assert f(FAKE, 2, 100, 768, FAKE, 1, (1 << 32) - 100, FAKE, FAKE, ws, None) == 1
    assert f(FAKE, 2, 100, 768, FAKE, 1, 0, None, FAKE, ws, None) == 1
    assert f(FAKE, 2, 100, 768, FAKE, 1, 0, FAKE, FAKE, 0, None) == 1          # no workspace
    assert f(FAKE, 7, 100, 768, FAKE, 1, 0, FAKE, FAKE, ws, None) == 2          # dtype
    assert f(FAKE, 2, 100, 768, FAKE, 0, 0, FAKE, FAKE, 0, None) == 0           # no queries
    g = lib.precog_decode_keys
    assert g(FAKE, -1, FAKE, FAKE, None) == 1
    assert g(None, 3, FAKE, FAKE, None) == 1
    assert g(FAKE, 0, FAKE, FAKE, None) == 0


def test_binding_has_every_declared_call():
    """The Python binding carries every C-ABI entry point under the same name, and the
    host-only ones answer without a GPU."""
    import paper_2608_02560_gb300 as pg
    for n in declared_functions():
        assert callable(getattr(pg, n, None)), f"{n} has no same-named Python binding"
    assert pg.precog_abi_version() == 1
    assert pg.precog_status_string(1) == "PRECOG_ERR_INVALID_ARG"
    assert pg.precog_launch_count() >= 0


def test_extension_calls_reject_bad_arguments(lib):
    """Top-k, trajectory, composition, SMC and no-workspace retrieval: invalid sizes,
    counts and pointers return their status before any launch."""
    import paper_2608_02560_gb300 as pg
    ws = 1 << 20
    t = lib.precog_retrieve_topk
    assert t(FAKE, 2, 100, 768, FAKE, 1, 0, FAKE, FAKE, FAKE, ws, None) == 2     # k < 1
    assert t(FAKE, 2, 100, 768, FAKE, 1, 9, FAKE, FAKE, FAKE, ws, None) == 2     # k > 8
    assert t(FAKE, 2, 100, 768, FAKE, 1, 3, None, FAKE, FAKE, ws, None) == 1     # no d_idx
    assert t(FAKE, 2, 100, 768, FAKE, 1, 3, FAKE, FAKE, FAKE, 0, None) == 1      # no workspace
    assert t(FAKE, 2, 100, 768, FAKE, 0, 3, FAKE, FAKE, FAKE, 0, None) == 0      # no queries
    s = _inputs(pg, a_kind=pg.PRECOG_A_POWER)
    tr = lib.precog_encode_trajectory
    assert tr(ctypes.byref(s), FAKE, 4, 64, 0, FAKE, FAKE, 0, 0, 1, None) == 1   # stride 0
    assert tr(ctypes.byref(s), FAKE, 4, 64, 8, None, FAKE, 0, 0, 1, None) == 1   # no entry offsets
    assert tr(ctypes.byref(s), FAKE, 4, 64, 8, FAKE, FAKE + 8, 0, 0, 1, None) == 1  # misaligned
    assert tr(ctypes.byref(s), FAKE, 0, 64, 8, FAKE, FAKE, 0, 0, 1, None) == 0   # no chunks
    c = lib.precog_prefill_composed
    assert c(ctypes.byref(s), 2, 32, FAKE, 0, 10, 1, 0, 9, FAKE, FAKE, 1.0, FAKE, 0, None, 0, None) == 2
    assert c(ctypes.byref(s), 2, 32, FAKE, 0, 10, 1, 0, 3, FAKE, None, 1.0, FAKE, 0, None, 0, None) == 1
    assert c(ctypes.byref(s), 2, 32, FAKE, 0, 10, 1, 0, 3, FAKE, FAKE, 0.0, FAKE, 0, None, 0, None) == 1
    assert c(ctypes.byref(s), 2, 32, FAKE, 0, 10, 1, 0, 3, FAKE, FAKE, 1.0, None, 0, None, 0, None) == 1
    r = lib.precog_smc_route
    assert r(FAKE, 7, 10, 64, FAKE, 4, FAKE, 8, FAKE, FAKE, FAKE, None, None) == 2   # dtype
    assert r(FAKE, 2, 10, 0, FAKE, 4, FAKE, 8, FAKE, FAKE, FAKE, None, None) == 1    # dim 0
    assert r(FAKE, 2, 10, 64, None, 4, FAKE, 8, FAKE, FAKE, FAKE, None, None) == 1   # no prototypes
    assert r(FAKE, 2, 0, 64, FAKE, 4, FAKE, 8, FAKE, FAKE, FAKE, None, None) == 0    # nothing to route
    k = lib.precog_smc_consolidate
    assert k(FAKE, 4, 64, FAKE, 2, FAKE, 8, 0.5, None) == 2                          # fp16 states
    assert k(FAKE, 4, 64, FAKE, 0, FAKE, 8, 0.0, None) == 1                          # alpha 0
    assert k(FAKE, 4, 64, FAKE, 0, FAKE, 8, 1.5, None) == 1                          # alpha > 1
    assert k(FAKE + 4, 4, 64, FAKE, 0, FAKE, 8, 0.5, None) == 1                      # misaligned
    assert k(FAKE, 4, 64, FAKE, 0, FAKE, 0, 0.5, None) == 0                          # no deposits
    n = lib.precog_retrieve_noalloc
    assert n(FAKE, 2, 100, 768, FAKE, -1, FAKE, FAKE, None) == 1
    assert n(FAKE, 2, -1, 768, FAKE, 1, FAKE, FAKE, None) == 1
