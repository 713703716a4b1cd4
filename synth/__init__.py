"""Seeded synthetic inputs shared by the tests, the bench and the oracle.

This module holds no attention arithmetic: it only draws numbers and lays out
pages.  Both sides of a parity test obtain their inputs from here; the CUDA
library never imports it and the oracle never reads an input back from the
device.

Element generator (counter based, identical on host and device):

    value(stream, i) = TABLE[splitmix64(base(stream) + i) >> (64 - TABLE_BITS)]

``splitmix64`` is the published SplitMix64 output function (Steele, Lea and
Flood, "Fast splittable pseudorandom number generators", OOPSLA 2014; the
constants of Vigna's reference implementation).  ``TABLE`` holds 2**20
standard-normal samples from numpy's PCG64 rounded to bf16 (round to nearest
even), so every element is an exact N(0, 1) draw rounded to bf16.  The device
fill kernel (``synth/fill.cu``) evaluates the same integer formula against the
same uploaded table, so any element the oracle needs can be recomputed on the
host bit for bit without reading device memory.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

TABLE_BITS = 20
TABLE_SEED = 0x5EED_0B16

_M64 = np.uint64(0xFFFFFFFFFFFFFFFF)
_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_C1 = np.uint64(0xBF58476D1CE4E5B9)
_C2 = np.uint64(0x94D049BB133111EB)

_table_cache = {}


def splitmix64(x):
    """SplitMix64 on a numpy uint64 array (wrapping arithmetic)."""
    x = np.asarray(x, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = x + _GOLDEN
        z = (z ^ (z >> np.uint64(30))) * _C1
        z = (z ^ (z >> np.uint64(27))) * _C2
        return z ^ (z >> np.uint64(31))


def f32_to_bf16_bits(x) -> np.ndarray:
    """Round float32 values to bf16 (nearest even) and return the bit patterns."""
    u = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    rnd = ((u >> np.uint64(16)) & np.uint64(1)) + np.uint64(0x7FFF)
    return ((u + rnd) >> np.uint64(16)).astype(np.uint16)


def bf16_bits_to_f32(b) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def normal_table(seed: int = TABLE_SEED) -> np.ndarray:
    """2**TABLE_BITS N(0,1) samples as bf16 bit patterns (uint16)."""
    if seed not in _table_cache:
        rng = np.random.default_rng(seed)
        vals = rng.standard_normal(1 << TABLE_BITS).astype(np.float32)
        _table_cache[seed] = f32_to_bf16_bits(vals)
    return _table_cache[seed]


def stream_base(seed: int, stream: int) -> int:
    """Per-stream counter offset: splitmix64(seed * 2**32 + stream)."""
    key = np.uint64(((int(seed) & 0xFFFFFFFF) << 32) | (int(stream) & 0xFFFFFFFF))
    return int(splitmix64(key))


def values(base: int, idx, table: np.ndarray | None = None) -> np.ndarray:
    """bf16 bit patterns of elements ``idx`` of the stream with offset ``base``."""
    t = normal_table() if table is None else table
    with np.errstate(over="ignore"):
        h = splitmix64(np.asarray(idx, dtype=np.uint64) + np.uint64(base))
    return t[(h >> np.uint64(64 - TABLE_BITS)).astype(np.int64)]


_HERE = os.path.dirname(os.path.abspath(__file__))
_HOSTLIB = os.path.join(_HERE, "libsynth_host.so")
_host = None


def _hostgen():
    """The C version of the same formula (OpenMP), built on first use."""
    global _host
    if _host is None:
        src = os.path.join(_HERE, "hostgen.c")
        if (not os.path.exists(_HOSTLIB)
                or os.path.getmtime(_HOSTLIB) < os.path.getmtime(src)):
            tmp = _HOSTLIB + f".tmp{os.getpid()}"
            subprocess.check_call(["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared",
                                   "-o", tmp, src])
            os.replace(tmp, _HOSTLIB)
        lib = ctypes.CDLL(_HOSTLIB)
        P, i64, u64 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_uint64
        lib.synth_range.argtypes = [P, i64, u64, u64, P]
        lib.synth_range.restype = None
        lib.synth_pages.argtypes = [P, P, i64, i64, u64, P]
        lib.synth_pages.restype = None
        _host = lib
    return _host


def values_range(base: int, start: int, n: int, table: np.ndarray | None = None) -> np.ndarray:
    """Elements [start, start + n) of a stream (C fast path)."""
    t = normal_table() if table is None else table
    out = np.empty(int(n), dtype=np.uint16)
    if n:
        _hostgen().synth_range(out.ctypes.data, int(n), ctypes.c_uint64(base),
                               ctypes.c_uint64(int(start)), t.ctypes.data)
    return out


def values_pages(base: int, pages, page_elems: int, table: np.ndarray | None = None) -> np.ndarray:
    """Elements of whole pages (page p covers [p*page_elems, (p+1)*page_elems))."""
    t = normal_table() if table is None else table
    pg = np.ascontiguousarray(np.asarray(pages, dtype=np.int64))
    out = np.empty(len(pg) * int(page_elems), dtype=np.uint16)
    if len(pg):
        _hostgen().synth_pages(out.ctypes.data, pg.ctypes.data, len(pg), int(page_elems),
                               ctypes.c_uint64(base), t.ctypes.data)
    return out


def fill(base: int, shape, table: np.ndarray | None = None) -> np.ndarray:
    """A whole tensor of the stream, element i at flat index i."""
    n = int(np.prod(shape))
    return values_range(base, 0, n, table).reshape(shape)


# Stream identifiers: one per (layer, tensor) so that layers are independent.
STREAM_Q, STREAM_K, STREAM_V, STREAM_KPOOL, STREAM_VPOOL = range(5)


def stream_id(layer: int, kind: int, salt: int = 0) -> int:
    return (int(salt) << 20) | (int(layer) << 4) | int(kind)
