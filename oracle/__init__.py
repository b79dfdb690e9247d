"""PRECOG oracle: slow, sequential fp64 CPU reference of the hot path.

TEST INFRASTRUCTURE ONLY. Only the test suite, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import this package. The product
library never loads it and shares no code with it.

The arithmetic lives in ``precog_oracle.c`` (plain C, double precision); this
module compiles it with gcc and marshals numpy arrays into it.

* :func:`scan` -- the selective-SSM rollout of Eq. 1 / Appendix A over every
  chunk of one layer, with final-state capture (Sec. 4.2) and optional
  readout ``y_t = C(h_t)``.
* :func:`retrieve` -- exact top-1 dot-product retrieval (Sec. 4.2), lowest row
  on ties, NaN never wins.
* :func:`rollout` -- one chunk convenience wrapper of :func:`scan`.
* :func:`scan_threads` -- :func:`scan` with the chunks split over host threads
  (chunks are independent, Sec. 4.2); the per-chunk arithmetic is :func:`scan`'s.
* :func:`retrieve_topk` -- the k best rows per query by exact score (ties to the
  lower row), the top-k of Sec. 4.2 / Sec. 5.4.
* :func:`compose` -- the softmax-weighted state composition of Sec. 4.4
  (multi-chunk extension) and Eq. smc-fusion.
* :func:`trajectory` -- the K-dial trajectory of Sec. 5.2 (every k-th state).
* :func:`smc_route` -- two-level cluster routing of Sec. 5.1 (Eqs. smc-domain,
  smc-sub).
* :func:`smc_consolidate` -- the semantic-state EMA of Sec. 5.3 (Eq. smc-ema).
* :func:`scan_complex` -- the scan with the complex diagonal A of Eq. 1.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "precog_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "liboracle.so")

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the C oracle into ``oracle/_build/liboracle.so`` (gcc, -O2,
    no floating-point contraction, no fast-math) and return its path."""
    with _lock:
        if (not force and os.path.exists(_LIB_PATH)
                and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
            return _LIB_PATH
        os.makedirs(_BUILD_DIR, exist_ok=True)
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math",
               "-shared", "-fPIC", _SRC, "-o", tmp, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
        return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB_PATH)
        p_i64 = ctypes.POINTER(ctypes.c_int64)
        p_f64 = ctypes.POINTER(ctypes.c_double)
        lib.oracle_scan.restype = ctypes.c_int
        lib.oracle_scan.argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_int64, p_i64,
                                    p_f64, p_f64, p_f64, p_f64, p_f64, p_f64, p_f64, p_f64]
        lib.oracle_trajectory.restype = ctypes.c_int
        lib.oracle_trajectory.argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_int64, p_i64,
                                          p_f64, p_f64, p_f64, p_f64, ctypes.c_int64, p_i64, p_f64]
        lib.oracle_scan_complex.restype = ctypes.c_int
        lib.oracle_scan_complex.argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_int64, p_i64,
                                            p_f64, p_f64, p_f64, p_f64, p_f64, p_f64, p_f64, p_f64,
                                            p_f64]
        lib.oracle_scores.restype = ctypes.c_int
        lib.oracle_scores.argtypes = [ctypes.c_int64, ctypes.c_int64, p_f64, ctypes.c_int64, p_f64,
                                      p_f64]
        lib.oracle_retrieve.restype = ctypes.c_int
        lib.oracle_retrieve.argtypes = [ctypes.c_int64, ctypes.c_int64, p_f64, ctypes.c_int64,
                                        p_f64, p_i64, p_f64]
        _lib = lib
    return _lib


def _f64(a):
    if a is None:
        return None
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def _ptr(a, ctype):
    if a is None:
        return ctypes.POINTER(ctype)()
    return a.ctypes.data_as(ctypes.POINTER(ctype))


def scan(x, dt, A, B, offsets, C=None, h0=None, want_y=False):
    """Scan one layer of chunks from ``h0`` (zero state when None).

    Shapes: x, dt ``[T_tot, D]``; A ``[D, N]``; B, C ``[T_tot, N]``;
    offsets ``[n_chunks + 1]`` int64 prefix sums; h0 ``[n_chunks, D, N]``.
    Returns ``(states [n_chunks, D, N], y [T_tot, D] or None)`` in float64.
    """
    lib = _load()
    x, dt, A, B = _f64(x), _f64(dt), _f64(A), _f64(B)
    C = _f64(C) if want_y else None
    h0 = _f64(h0)
    offsets = np.ascontiguousarray(np.asarray(offsets, dtype=np.int64))
    D, N = A.shape
    n_chunks = offsets.shape[0] - 1
    T_tot = x.shape[0]
    if x.shape != (T_tot, D) or dt.shape != (T_tot, D) or B.shape != (T_tot, N):
        raise ValueError("oracle.scan: inconsistent input shapes")
    if want_y and (C is None or C.shape != (T_tot, N)):
        raise ValueError("oracle.scan: y requested but C has the wrong shape")
    if h0 is not None and h0.shape != (n_chunks, D, N):
        raise ValueError("oracle.scan: h0 must be [n_chunks, D, N]")
    if n_chunks > 0 and (offsets[0] < 0 or offsets[-1] > T_tot):
        raise ValueError("oracle.scan: offsets out of range")
    states = np.zeros((n_chunks, D, N), dtype=np.float64)
    y = np.zeros((T_tot, D), dtype=np.float64) if want_y else None
    p64, pi = ctypes.c_double, ctypes.c_int64
    rc = lib.oracle_scan(D, N, n_chunks, _ptr(offsets, pi), _ptr(x, p64), _ptr(dt, p64),
                         _ptr(A, p64), _ptr(B, p64), _ptr(C, p64), _ptr(h0, p64),
                         _ptr(states, p64), _ptr(y, p64))
    if rc != 0:
        raise ValueError(f"oracle_scan rejected its arguments (rc={rc})")
    return states, y


def scan_threads(x, dt, A, B, offsets, threads: int):
    """:func:`scan` (capture only, zero initial state) with the chunks split into
    ``threads`` contiguous groups, each scanned by its own host thread. The C rollout
    releases the interpreter lock while it runs, so the groups run on separate cores.
    The arithmetic is :func:`scan`'s: every chunk's result is bit-identical to it.
    Returns the ``[n_chunks, D, N]`` states."""
    import concurrent.futures as cf
    offsets = np.asarray(offsets, dtype=np.int64)
    n_chunks = offsets.shape[0] - 1
    x, dt, A, B = _f64(x), _f64(dt), _f64(A), _f64(B)
    D, N = A.shape
    states = np.zeros((n_chunks, D, N), dtype=np.float64)
    bounds = np.linspace(0, n_chunks, max(1, min(threads, n_chunks)) + 1).astype(np.int64)

    def part(i):
        c0, c1 = int(bounds[i]), int(bounds[i + 1])
        if c1 == c0:
            return
        r0, r1 = int(offsets[c0]), int(offsets[c1])
        st, _ = scan(x[r0:r1], dt[r0:r1], A, B[r0:r1], offsets[c0:c1 + 1] - r0)
        states[c0:c1] = st

    with cf.ThreadPoolExecutor(max_workers=len(bounds) - 1) as ex:
        list(ex.map(part, range(len(bounds) - 1)))
    return states


def rollout(x, dt, A, B, C=None, h0=None, want_y=False):
    """S(h0, x_{1:T}) of Appendix A for one chunk: returns ``(h_T [D, N], y [T, D])``."""
    x = _f64(x)
    T = x.shape[0]
    D, N = np.asarray(A).shape
    h0b = None if h0 is None else _f64(h0).reshape(1, D, N)
    states, y = scan(x, dt, A, B, np.array([0, T], dtype=np.int64), C=C, h0=h0b, want_y=want_y)
    return states[0], y


def retrieve(index, queries):
    """Exact top-1 by dot product; returns ``(best_idx int64 [Q], best_score float64 [Q])``."""
    lib = _load()
    index = _f64(index)
    queries = _f64(queries)
    if queries.ndim == 1:
        queries = queries.reshape(1, -1)
    M, dim = index.shape
    Q = queries.shape[0]
    if queries.shape[1] != dim:
        raise ValueError("oracle.retrieve: query dim mismatch")
    best_idx = np.empty(Q, dtype=np.int64)
    best_score = np.empty(Q, dtype=np.float64)
    rc = lib.oracle_retrieve(M, dim, _ptr(index, ctypes.c_double), Q,
                             _ptr(queries, ctypes.c_double),
                             _ptr(best_idx, ctypes.c_int64), _ptr(best_score, ctypes.c_double))
    if rc != 0:
        raise ValueError(f"oracle_retrieve rejected its arguments (rc={rc})")
    return best_idx, best_score


def scores(index, queries):
    """All dot products ``[Q, M]`` in double."""
    lib = _load()
    index = _f64(index)
    queries = _f64(queries)
    if queries.ndim == 1:
        queries = queries.reshape(1, -1)
    M, dim = index.shape
    Q = queries.shape[0]
    out = np.empty((Q, M), dtype=np.float64)
    rc = lib.oracle_scores(M, dim, _ptr(index, ctypes.c_double), Q, _ptr(queries, ctypes.c_double),
                           _ptr(out, ctypes.c_double))
    if rc != 0:
        raise ValueError(f"oracle_scores rejected its arguments (rc={rc})")
    return out


def retrieve_topk(index, queries, k):
    """The k rows with the highest exact score per query, best first; among equal scores
    the lower row comes first; NaN scores are never selected; missing entries are row -1
    with score NaN. Returns ``(rows int64 [Q, k], scores float64 [Q, k])``."""
    S = scores(index, queries)
    Q, M = S.shape
    rows = np.full((Q, k), -1, dtype=np.int64)
    vals = np.full((Q, k), np.nan)
    for q in range(Q):
        cand = [(-S[q, i], i) for i in range(M) if not np.isnan(S[q, i])]
        cand.sort()
        for j, (neg, i) in enumerate(cand[:k]):
            rows[q, j] = i
            vals[q, j] = -neg
    return rows, vals


def compose(bank_rows, row_scores, temperature=1.0):
    """h_init = sum_j w_j h^(j), w = softmax(score / temperature) over the valid entries
    (Sec. 4.4, Eq. smc-fusion). ``bank_rows [k, ...]`` are the states of the k retrieved
    chunks, ``row_scores [k]`` their scores (NaN marks a missing entry, weight 0)."""
    s = np.asarray(row_scores, dtype=np.float64)
    valid = ~np.isnan(s)
    out = np.zeros(np.asarray(bank_rows).shape[1:], dtype=np.float64)
    if not valid.any():
        return out
    z = s[valid] / temperature
    e = np.exp(z - z.max())
    w = e / e.sum()
    rows = np.asarray(bank_rows, dtype=np.float64)[valid]
    for j in range(len(w)):
        out = out + w[j] * rows[j]
    return out


def trajectory_offsets(offsets, stride):
    """Prefix sums of K_c = ceil(len_c / stride) (entries kept per chunk)."""
    offsets = np.asarray(offsets, dtype=np.int64)
    lens = np.diff(offsets)
    k = (lens + stride - 1) // stride
    out = np.zeros(len(offsets), dtype=np.int64)
    np.cumsum(k, out=out[1:])
    return out


def trajectory(x, dt, A, B, offsets, stride):
    """States after every stride-th token of each chunk and after its last token
    (Sec. 5.2). Returns ``(traj [entries, D, N], entry_offsets [n_chunks + 1])``."""
    lib = _load()
    x, dt, A, B = _f64(x), _f64(dt), _f64(A), _f64(B)
    offsets = np.ascontiguousarray(np.asarray(offsets, dtype=np.int64))
    D, N = A.shape
    eo = trajectory_offsets(offsets, stride)
    traj = np.zeros((int(eo[-1]), D, N), dtype=np.float64)
    p64, pi = ctypes.c_double, ctypes.c_int64
    rc = lib.oracle_trajectory(D, N, len(offsets) - 1, _ptr(offsets, pi), _ptr(x, p64), _ptr(dt, p64),
                               _ptr(A, p64), _ptr(B, p64), stride, _ptr(eo, pi), _ptr(traj, p64))
    if rc != 0:
        raise ValueError(f"oracle_trajectory rejected its arguments (rc={rc})")
    return traj, eo


def smc_route(embeddings, domain_protos, sub_protos, J):
    """m* = argmax_m <e, p_m>, then j* = argmax_{j < J[m*]} <e, q_{m*, j}> (Sec. 5.1);
    both argmaxes keep the lowest index on ties and never pick a NaN score.
    ``sub_protos [M, J_max, dim]``. Returns ``(m* int64 [n], j* int64 [n])``; -1 when no
    comparable score exists."""
    emb = _f64(embeddings)
    if emb.ndim == 1:
        emb = emb.reshape(1, -1)
    sub = _f64(sub_protos)
    m_idx, _ = retrieve(domain_protos, emb)
    j_idx = np.full(emb.shape[0], -1, dtype=np.int64)
    for c in range(emb.shape[0]):
        m = int(m_idx[c])
        if m < 0 or int(J[m]) <= 0:
            continue
        jj, _ = retrieve(sub[m, : int(J[m])], emb[c:c + 1])
        j_idx[c] = jj[0]
    return m_idx, j_idx


def smc_consolidate(semantic, states, slots, alpha):
    """For c = 0, 1, ... in order: s[slot_c] <- (1 - alpha) s[slot_c] + alpha h^(c)
    (Eq. smc-ema); a slot of -1 (a forgetting candidate) deposits nothing. Returns the
    updated table in double."""
    out = _f64(semantic).copy()
    h = _f64(states)
    for c, slot in enumerate(np.asarray(slots, dtype=np.int64)):
        if slot < 0:
            continue
        out[slot] = (1.0 - alpha) * out[slot] + alpha * h[c]
    return out


def scan_complex(x, dt, A_re, A_im, B, offsets, C=None, h0=None, want_y=False):
    """Complex-A scan of one layer (Eq. 1 with A = A_re + i A_im). h0 ``[n_chunks, D, N]``
    complex. Returns ``(states complex128 [n_chunks, D, N], y float64 [T_tot, D] or None)``."""
    lib = _load()
    x, dt, A_re, A_im, B = _f64(x), _f64(dt), _f64(A_re), _f64(A_im), _f64(B)
    C = _f64(C) if want_y else None
    offsets = np.ascontiguousarray(np.asarray(offsets, dtype=np.int64))
    D, N = A_re.shape
    n_chunks = offsets.shape[0] - 1
    T_tot = x.shape[0]
    h0c = None if h0 is None else np.ascontiguousarray(np.asarray(h0, dtype=np.complex128))
    states = np.zeros((n_chunks, D, N), dtype=np.complex128)
    y = np.zeros((T_tot, D), dtype=np.float64) if want_y else None
    p64, pi = ctypes.c_double, ctypes.c_int64
    h0p = ctypes.POINTER(p64)() if h0c is None else h0c.ctypes.data_as(ctypes.POINTER(p64))
    rc = lib.oracle_scan_complex(D, N, n_chunks, _ptr(offsets, pi), _ptr(x, p64), _ptr(dt, p64),
                                 _ptr(A_re, p64), _ptr(A_im, p64), _ptr(B, p64), _ptr(C, p64), h0p,
                                 states.ctypes.data_as(ctypes.POINTER(p64)), _ptr(y, p64))
    if rc != 0:
        raise ValueError(f"oracle_scan_complex rejected its arguments (rc={rc})")
    return states, y

