"""Seeded synthetic inputs shaped like PRECOG's workloads.

This module is shared by the CUDA path and the oracle and holds none of the
method's arithmetic: it only draws random numbers and lays them out. Host
inputs come from numpy's PCG64 generator; large inputs are drawn on the
device with a ``torch.Generator`` keyed by ``(seed, layer, stream)``, so every
layer can be regenerated independently and sampled rows can be copied back to
the host for the oracle.

Input recipe (shared by every configuration):
  x ~ N(0, 1); dt = softplus(z - 2) with z ~ N(0, 1); A[d, n] = -(n + 1);
  B, C ~ N(0, 1/N) (variance 1/N); key embeddings unit-norm Gaussian;
  query embedding = a key + Gaussian noise (std given per workload),
  renormalised.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

# ----------------------------------------------------------------------------------------------
# Workload shapes (the sizes of the paper's workloads: 512- and 3000-token chunks, a 24-layer
# 192 KB state, a 1M-entry key index).
# ----------------------------------------------------------------------------------------------


@dataclass(frozen=True)
class EncodeShape:
    name: str
    n_layers: int
    D: int
    N: int
    n_chunks: int
    chunk_len: int          # fixed length, or 0 for ragged
    min_len: int = 0        # ragged lengths are uniform in [min_len, max_len]
    max_len: int = 0
    dtype: str = "bf16"     # dtype of x, dt, B, C


TINY = EncodeShape("tiny-exact-check", 1, 64, 16, 8, 256, dtype="f32")
WIDE = EncodeShape("single-layer-wide-encode", 1, 2048, 16, 1024, 512)
PAPER = EncodeShape("paper-shaped-corpus-encode", 24, 256, 16, 4096, 3000)
RAGGED = EncodeShape("ragged-large-scale-encode", 24, 512, 16, 8192, 0, 256, 4096)

QUERY_INDEX_M = 1_000_000
QUERY_DIM = 768
QUERY_TOKENS = 64
QUERY_NOISE = 0.02
TINY_QUERY_TOKENS = 32
TINY_INDEX_M = 8
TINY_DIM = 64
TINY_PLANTED = 3
TINY_NOISE = 0.05


def structured_A(D: int, N: int) -> np.ndarray:
    """A[d, n] = -(n + 1) for every channel d (the configurations' A)."""
    return -np.tile(np.arange(1, N + 1, dtype=np.float32), (D, 1))


def softplus_np(z: np.ndarray) -> np.ndarray:
    return np.logaddexp(0.0, z)


def ragged_offsets(n_chunks: int, min_len: int, max_len: int, seed: int) -> np.ndarray:
    """int64 prefix sums of chunk lengths drawn uniformly in [min_len, max_len]."""
    rng = np.random.default_rng([seed, 0x0FF5E7])
    lens = rng.integers(min_len, max_len + 1, size=n_chunks, dtype=np.int64)
    off = np.zeros(n_chunks + 1, dtype=np.int64)
    np.cumsum(lens, out=off[1:])
    return off


def fixed_offsets(n_chunks: int, length: int) -> np.ndarray:
    return np.arange(n_chunks + 1, dtype=np.int64) * length


def shape_offsets(shape: EncodeShape, seed: int = 0) -> np.ndarray:
    if shape.chunk_len > 0:
        return fixed_offsets(shape.n_chunks, shape.chunk_len)
    return ragged_offsets(shape.n_chunks, shape.min_len, shape.max_len, seed)


# ----------------------------------------------------------------------------------------------
# Host (numpy) generators: small cases, the tiny exact-check workload
# ----------------------------------------------------------------------------------------------


def host_scan_inputs(T: int, D: int, N: int, seed: int, dtype=np.float32):
    """x, dt, B, C ``[T, D] / [T, N]`` and A ``[D, N]`` with the shared recipe."""
    rng = np.random.default_rng([seed, 0x5CA9])
    x = rng.standard_normal((T, D)).astype(dtype)
    dt = softplus_np(rng.standard_normal((T, D)) - 2.0).astype(dtype)
    s = 1.0 / math.sqrt(N)
    B = (rng.standard_normal((T, N)) * s).astype(dtype)
    C = (rng.standard_normal((T, N)) * s).astype(dtype)
    A = structured_A(D, N)
    return x, dt, A, B, C


def unit_rows(rng, M: int, dim: int) -> np.ndarray:
    e = rng.standard_normal((M, dim))
    return e / np.linalg.norm(e, axis=1, keepdims=True)


def planted_queries(rng, index: np.ndarray, rows, noise: float) -> np.ndarray:
    q = index[np.asarray(rows)] + noise * rng.standard_normal((len(rows), index.shape[1]))
    return q / np.linalg.norm(q, axis=1, keepdims=True)


@dataclass
class TinyWorkload:
    x: np.ndarray
    dt: np.ndarray
    A: np.ndarray
    B: np.ndarray
    C: np.ndarray
    offsets: np.ndarray
    qx: np.ndarray
    qdt: np.ndarray
    qB: np.ndarray
    qC: np.ndarray
    index: np.ndarray
    query: np.ndarray
    planted: int


def tiny_workload(seed: int = 0) -> TinyWorkload:
    """1 layer, D=64, N=16, fp32: 8 chunks x 256 tokens, a 32-token query, an 8-entry index
    of unit-norm dim-64 keys and a query embedding = key 3 + N(0, 0.05^2) noise, renormalised."""
    s = TINY
    x, dt, A, B, C = host_scan_inputs(s.n_chunks * s.chunk_len, s.D, s.N, seed)
    qx, qdt, _, qB, qC = host_scan_inputs(TINY_QUERY_TOKENS, s.D, s.N, seed + 1)
    rng = np.random.default_rng([seed, 0x1D3])
    index = unit_rows(rng, TINY_INDEX_M, TINY_DIM).astype(np.float32)
    query = planted_queries(rng, index.astype(np.float64), [TINY_PLANTED], TINY_NOISE).astype(np.float32)
    return TinyWorkload(x, dt, A, B, C, fixed_offsets(s.n_chunks, s.chunk_len),
                        qx, qdt, qB, qC, index, query, TINY_PLANTED)


# ----------------------------------------------------------------------------------------------
# Device generators (torch RNG on the GPU): large workloads, regenerated per (seed, layer)
# ----------------------------------------------------------------------------------------------

_SLICE = 1 << 27  # elements drawn per slice, bounds temporaries to ~0.5 GB of fp32


def _seed(seed: int, layer: int, stream: int) -> int:
    return (seed * 1_000_003 + layer * 7_919 + stream * 104_729 + 17) & 0x7FFF_FFFF_FFFF


def _fill_normal(out, gen, std=1.0, shift=0.0, softplus=False):
    import torch
    flat = out.view(-1)
    n = flat.numel()
    for s in range(0, n, _SLICE):
        e = min(n, s + _SLICE)
        z = torch.randn(e - s, generator=gen, device=out.device, dtype=torch.float32)
        if shift:
            z.add_(shift)
        if softplus:
            z = torch.nn.functional.softplus(z)
        if std != 1.0:
            z.mul_(std)
        flat[s:e].copy_(z)
    return out


def device_scan_inputs(T: int, D: int, N: int, seed: int, layer: int, device, dtype=None,
                       with_C: bool = True, out=None):
    """Per-layer inputs on the device: dict of x, dt ``[T, D]``, B, C ``[T, N]``, A ``[D, N]``.

    ``out`` may hold preallocated tensors (same keys) that are refilled in place."""
    import torch
    dtype = torch.bfloat16 if dtype is None else dtype
    res = {} if out is None else out
    for key, shape in (("x", (T, D)), ("dt", (T, D)), ("B", (T, N)), ("C", (T, N))):
        if key == "C" and not with_C:
            continue
        if key not in res:
            res[key] = torch.empty(shape, dtype=dtype, device=device)
    g = torch.Generator(device=device)
    g.manual_seed(_seed(seed, layer, 1))
    _fill_normal(res["x"], g)
    g.manual_seed(_seed(seed, layer, 2))
    _fill_normal(res["dt"], g, shift=-2.0, softplus=True)
    g.manual_seed(_seed(seed, layer, 3))
    _fill_normal(res["B"], g, std=1.0 / math.sqrt(N))
    if with_C:
        g.manual_seed(_seed(seed, layer, 4))
        _fill_normal(res["C"], g, std=1.0 / math.sqrt(N))
    if "A" not in res:
        res["A"] = torch.from_numpy(structured_A(D, N)).to(device)
    return res


def device_unit_index(M: int, dim: int, seed: int, device, dtype=None, out=None):
    """[M, dim] unit-norm Gaussian keys (normalised in fp32, stored in ``dtype``)."""
    import torch
    dtype = torch.float16 if dtype is None else dtype
    idx = torch.empty((M, dim), dtype=dtype, device=device) if out is None else out
    g = torch.Generator(device=device)
    g.manual_seed(_seed(seed, 0, 11))
    rows = max(1, _SLICE // dim)
    for s in range(0, M, rows):
        e = min(M, s + rows)
        z = torch.randn((e - s, dim), generator=g, device=device, dtype=torch.float32)
        z.div_(torch.linalg.vector_norm(z, dim=1, keepdim=True))
        idx[s:e].copy_(z)
    return idx


def device_planted_queries(index, n_queries: int, noise: float, seed: int):
    """Queries = randomly chosen keys + N(0, noise^2) noise, renormalised; returns (q, rows)."""
    import torch
    g = torch.Generator(device=index.device)
    g.manual_seed(_seed(seed, 0, 12))
    rows = torch.randint(0, index.shape[0], (n_queries,), generator=g, device=index.device)
    z = torch.randn((n_queries, index.shape[1]), generator=g, device=index.device,
                    dtype=torch.float32)
    q = index[rows].float() + noise * z
    q = q / torch.linalg.vector_norm(q, dim=1, keepdim=True)
    return q.to(index.dtype), rows


def device_normal_bank(entries: int, per_entry: int, seed: int, device, dtype=None, out=None):
    """[entries, per_entry] standard-normal state bank (random-normal stand-in states)."""
    import torch
    dtype = torch.bfloat16 if dtype is None else dtype
    bank = torch.empty((entries, per_entry), dtype=dtype, device=device) if out is None else out
    g = torch.Generator(device=device)
    g.manual_seed(_seed(seed, 0, 13))
    _fill_normal(bank, g)
    return bank
